// Page-backed cache buffers for the in-place path (Sec. 3.4: evicted states are
// physically removed). A buffer is one reserved device address range backed by
// separate physical pages of the allocation granularity; after the in-place
// compaction, the pages that hold no kept row, reserve row or guard row of any
// slab are unmapped and their memory returned to the device.
//
// The driver's virtual-memory calls (cuMemCreate, cuMemMap, ...) are reached
// through the runtime's driver entry point, so the library links no driver
// library.
#include "dkv.h"
#include "dkv_internal.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <cstdio>
#include <mutex>
#include <new>
#include <vector>

namespace dkv {
dkv_status set_error(dkv_status st, const char* msg);  // dkv_api.cu
}

struct dkv_vmm {
    CUdeviceptr base = 0;
    int64_t bytes = 0;   // reserved (a multiple of page)
    int64_t page = 0;    // allocation granularity
    int device = 0;
    std::vector<CUmemGenericAllocationHandle> handles;  // one per page; 0 once released
};

namespace {

struct Vmm {
    PFN_cuMemGetAllocationGranularity_v10020 granularity = nullptr;
    PFN_cuMemAddressReserve_v10020 reserve = nullptr;
    PFN_cuMemAddressFree_v10020 address_free = nullptr;
    PFN_cuMemCreate_v10020 create = nullptr;
    PFN_cuMemRelease_v10020 release = nullptr;
    PFN_cuMemMap_v10020 map = nullptr;
    PFN_cuMemUnmap_v10020 unmap = nullptr;
    PFN_cuMemSetAccess_v10020 set_access = nullptr;
    bool ok = false;
};

const Vmm& vmm()
{
    static std::once_flag once;
    static Vmm v;
    std::call_once(once, [] {
        auto get = [](const char* name, void** fn) {
            cudaDriverEntryPointQueryResult q;
            return cudaGetDriverEntryPointByVersion(name, fn, 12000, cudaEnableDefault, &q) == cudaSuccess &&
                   q == cudaDriverEntryPointSuccess && *fn != nullptr;
        };
        v.ok = get("cuMemGetAllocationGranularity", reinterpret_cast<void**>(&v.granularity)) &&
               get("cuMemAddressReserve", reinterpret_cast<void**>(&v.reserve)) &&
               get("cuMemAddressFree", reinterpret_cast<void**>(&v.address_free)) &&
               get("cuMemCreate", reinterpret_cast<void**>(&v.create)) &&
               get("cuMemRelease", reinterpret_cast<void**>(&v.release)) &&
               get("cuMemMap", reinterpret_cast<void**>(&v.map)) &&
               get("cuMemUnmap", reinterpret_cast<void**>(&v.unmap)) &&
               get("cuMemSetAccess", reinterpret_cast<void**>(&v.set_access));
    });
    return v;
}

dkv_status fail(dkv_status st, const char* fmt, long long a = 0, long long b = 0)
{
    char msg[256];
    snprintf(msg, sizeof msg, fmt, a, b);
    return dkv::set_error(st, msg);
}

CUmemAllocationProp page_prop(int device)
{
    CUmemAllocationProp prop = {};
    prop.type = CU_MEM_ALLOCATION_TYPE_PINNED;
    prop.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    prop.location.id = device;
    return prop;
}

void release_all(dkv_vmm* m)
{
    const Vmm& v = vmm();
    for (size_t i = 0; i < m->handles.size(); ++i)
        if (m->handles[i]) {
            v.unmap(m->base + i * m->page, m->page);
            v.release(m->handles[i]);
            m->handles[i] = 0;
        }
    if (m->base) v.address_free(m->base, m->bytes);
    m->base = 0;
}

}  // namespace

namespace dkv {

// Pages [0, npages) of a buffer whose slab h (rows [h * T_stride, (h + 1) *
// T_stride), row_bytes each) must keep its first min(T_stride, len[h] + reserve
// + guard) rows mapped: keep[i] = 1 when page i holds any such row.
void vmm_pages_to_keep(const int32_t* len, int64_t nslabs, int64_t T_stride, int64_t reserve, int64_t guard,
                       int64_t row_bytes, int64_t page, int64_t npages, uint8_t* keep)
{
    std::fill(keep, keep + npages, uint8_t(0));
    for (int64_t h = 0; h < nslabs; ++h) {
        const int64_t rows = std::min<int64_t>(T_stride, (int64_t)len[h] + reserve + guard);
        if (rows <= 0) continue;
        const int64_t b0 = h * T_stride * row_bytes, b1 = b0 + rows * row_bytes;  // [b0, b1)
        const int64_t p0 = b0 / page, p1 = std::min<int64_t>(npages, (b1 + page - 1) / page);
        for (int64_t i = p0; i < p1; ++i) keep[i] = 1;
    }
}

}  // namespace dkv

extern "C" {

dkv_status dkv_vmm_alloc(int64_t bytes, dkv_vmm** out, void** dptr)
{
    if (!out || !dptr) return fail(DKV_ERR_INVALID_ARG, "NULL out or dptr");
    *out = nullptr;
    *dptr = nullptr;
    if (bytes < 1) return fail(DKV_ERR_INVALID_ARG, "bytes=%lld < 1", bytes);
    const Vmm& v = vmm();
    if (!v.ok) return fail(DKV_ERR_CUDA, "virtual memory driver entry points unavailable");
    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess) return fail(DKV_ERR_CUDA, "cudaGetDevice failed");
    CUmemAllocationProp prop = page_prop(device);
    size_t gran = 0;
    if (v.granularity(&gran, &prop, CU_MEM_ALLOC_GRANULARITY_MINIMUM) != CUDA_SUCCESS || gran == 0)
        return fail(DKV_ERR_CUDA, "cuMemGetAllocationGranularity failed");
    dkv_vmm* m = new (std::nothrow) dkv_vmm();
    if (!m) return fail(DKV_ERR_OOM, "host allocation failed");
    m->page = (int64_t)gran;
    m->bytes = (bytes + m->page - 1) / m->page * m->page;
    m->device = device;
    const int64_t npages = m->bytes / m->page;
    if (v.reserve(&m->base, m->bytes, m->page, 0, 0) != CUDA_SUCCESS) {
        delete m;
        return fail(DKV_ERR_OOM, "cuMemAddressReserve of %lld bytes failed", bytes);
    }
    m->handles.assign((size_t)npages, 0);
    for (int64_t i = 0; i < npages; ++i) {
        CUmemGenericAllocationHandle h = 0;
        if (v.create(&h, m->page, &prop, 0) != CUDA_SUCCESS) {
            release_all(m);
            delete m;
            return fail(DKV_ERR_OOM, "cuMemCreate of page %lld failed", i);
        }
        if (v.map(m->base + i * m->page, m->page, 0, h, 0) != CUDA_SUCCESS) {
            v.release(h);
            release_all(m);
            delete m;
            return fail(DKV_ERR_CUDA, "cuMemMap of page %lld failed", i);
        }
        m->handles[(size_t)i] = h;
    }
    CUmemAccessDesc access = {};
    access.location.type = CU_MEM_LOCATION_TYPE_DEVICE;
    access.location.id = device;
    access.flags = CU_MEM_ACCESS_FLAGS_PROT_READWRITE;
    if (v.set_access(m->base, m->bytes, &access, 1) != CUDA_SUCCESS) {
        release_all(m);
        delete m;
        return fail(DKV_ERR_CUDA, "cuMemSetAccess failed");
    }
    *out = m;
    *dptr = reinterpret_cast<void*>(m->base);
    return dkv::set_error(DKV_OK, "");
}

int64_t dkv_vmm_page_bytes(const dkv_vmm* m) { return m ? m->page : 0; }

void dkv_vmm_pages_to_keep(const int32_t* len, int64_t nslabs, int64_t T_stride, int32_t reserve, int32_t guard,
                           int64_t row_bytes, int64_t page_bytes, int64_t npages, uint8_t* keep)
{
    if (!len || !keep || nslabs < 0 || T_stride < 1 || row_bytes < 1 || page_bytes < 1 || npages < 0) return;
    dkv::vmm_pages_to_keep(len, nslabs, T_stride, reserve, guard, row_bytes, page_bytes, npages, keep);
}

int64_t dkv_vmm_mapped_bytes(const dkv_vmm* m)
{
    if (!m) return 0;
    int64_t n = 0;
    for (CUmemGenericAllocationHandle h : m->handles) n += h ? m->page : 0;
    return n;
}

void dkv_vmm_free(dkv_vmm* m)
{
    if (!m) return;
    cudaDeviceSynchronize();
    release_all(m);
    delete m;
}

}  // extern "C"

namespace dkv {
// Used by dkv_api.cu, which owns the plan: unmap and release every mapped page
// of m that holds no row the plan still needs.
dkv_status vmm_release_pages(dkv_vmm* m, const uint8_t* keep, int64_t npages, int64_t* freed)
{
    const Vmm& v = vmm();
    if (cudaDeviceSynchronize() != cudaSuccess) return fail(DKV_ERR_CUDA, "cudaDeviceSynchronize failed");
    int64_t n = 0;
    for (int64_t i = 0; i < npages && i < (int64_t)m->handles.size(); ++i) {
        if (keep[i] || !m->handles[(size_t)i]) continue;
        if (v.unmap(m->base + i * m->page, m->page) != CUDA_SUCCESS)
            return fail(DKV_ERR_CUDA, "cuMemUnmap of page %lld failed", i);
        v.release(m->handles[(size_t)i]);
        m->handles[(size_t)i] = 0;
        n += m->page;
    }
    if (freed) *freed = n;
    return dkv::set_error(DKV_OK, "");
}

int64_t vmm_bytes(const dkv_vmm* m) { return m->bytes; }
int64_t vmm_page(const dkv_vmm* m) { return m->page; }
}  // namespace dkv
