// Host side of the C ABI declared in include/dkv.h: argument checks, the plan
// object, device allocations and kernel launches. No computation of the path
// happens here; every step runs in the kernels of dkv_map.cu, dkv_compact.cu,
// dkv_decode_mma.cu, dkv_decode.cu and dkv_topk.cu.
#include "dkv.h"
#include "dkv_internal.cuh"

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <new>
#include <vector>

struct dkv_plan {
    dkv_shape s{};
    int B = 0;
    int G = 0;
    int dense = 0;
    int reserve = 0;
    int64_t T_stride = 0;     // dense plans
    int64_t total_rows = 0;   // rows of the packed (or dense) cache
    int64_t kept_rows = 0;
    int device = 0;
    int32_t* d_len = nullptr;   // [NH]
    int64_t* d_off = nullptr;   // [NH+1]
    int64_t* d_ioff = nullptr;  // [NH+1]
    int32_t* d_idx = nullptr;   // [kept]
    int32_t* d_status = nullptr;
    float* d_work = nullptr;    // split-K partials
    int32_t* d_slab_count = nullptr;  // [B*H_kv][cols][2] arrival / written counters of the fused combine
    dkv::DecodeConfig cfg{};        // the decode step's kernel
    dkv::DecodeConfig cfg_multi1{};  // multi-query, one column tile (tensor-core plans)
    dkv::DecodeConfig cfg_multi{};   // multi-query, two column tiles (tensor-core plans)
    int64_t slots = 0;              // (CTA, slab) partial slots: CTAs + slabs of a layer
    dkv::WorkspaceLayout work{};    // carve-up of d_work
    int nctas_cap = 0, warps_cap = 0, cols_cap = 0;  // workspace sized for these
    int use_mma = 0;  // tensor-core decode kernel (needs the cache's row count for its tensor maps)
    int64_t inplace_stride = 0;  // > 0: slab h lives at rows h * stride of the dense buffer (in place)
    int32_t* d_order = nullptr;  // in place: [NH] slabs by length, longest first, then a claim counter
    std::vector<int64_t> layer_rows;  // kept rows of each layer (tensor-core plans: the grid of a launch)
};

namespace {

thread_local char g_err[512] = "";

dkv_status fail(dkv_status st, const char* fmt, ...)
{
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return st;
}

dkv_status ok()
{
    g_err[0] = '\0';
    return DKV_OK;
}

// Host-side fault injection for tests: DKV_FAULT=alloc makes the next device
// allocations fail, DKV_FAULT=launch makes kernel launches report failure, and
// DKV_FAULT=copy gives the tensor-core decode tensor maps whose boxes deliver
// half the bytes a stage expects, so every bounded copy wait runs out (the
// kernel then sets DKV_DEV_TMA_TIMEOUT and returns; nothing faults),
// DKV_FAULT=merge makes the last CTA of each fused merge wait for one partial
// more than the slab has (the wait runs out, sets DKV_DEV_MERGE_TIMEOUT and
// skips that merge), and DKV_FAULT=barrier makes the Top-K export's grid
// barriers wait for a CTA that does not exist (the first wait runs out and sets
// the workspace status word).
bool fault(const char* what)
{
    const char* f = std::getenv("DKV_FAULT");
    return f && std::strcmp(f, what) == 0;
}

dkv_status cuda_fail(cudaError_t e, const char* where)
{
    return fail(DKV_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

template <class T>
dkv_status dalloc(T** p, size_t count, const char* what)
{
    *p = nullptr;
    if (count == 0) count = 1;
    if (fault("alloc")) return fail(DKV_ERR_OOM, "%s: injected allocation failure", what);
    cudaError_t e = cudaMalloc(reinterpret_cast<void**>(p), count * sizeof(T));
    if (e != cudaSuccess) {
        cudaGetLastError();
        *p = nullptr;
        return fail(e == cudaErrorMemoryAllocation ? DKV_ERR_OOM : DKV_ERR_CUDA, "%s: cudaMalloc(%zu B): %s",
                    what, count * sizeof(T), cudaGetErrorString(e));
    }
    return DKV_OK;
}

dkv_status launched(cudaError_t e, const char* where)
{
    if (fault("launch")) return fail(DKV_ERR_CUDA, "%s: injected launch failure", where);
    if (e != cudaSuccess) return cuda_fail(e, where);
    return DKV_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

void release(dkv_plan* p)
{
    if (!p) return;
    cudaFree(p->d_len);
    cudaFree(p->d_off);
    cudaFree(p->d_ioff);
    cudaFree(p->d_idx);
    cudaFree(p->d_status);
    cudaFree(p->d_work);
    cudaFree(p->d_slab_count);
    cudaFree(p->d_order);
    delete p;
}

dkv_status check_shape(const dkv_shape* s, int32_t B)
{
    if (!s) return fail(DKV_ERR_INVALID_ARG, "shape is NULL");
    if (s->L < 1 || s->H < 1 || s->H_kv < 1 || s->D < 0)
        return fail(DKV_ERR_INVALID_ARG, "bad shape: L=%d H=%d H_kv=%d D=%d", s->L, s->H, s->H_kv, s->D);
    if (s->H % s->H_kv != 0)
        return fail(DKV_ERR_INVALID_ARG, "H=%d is not a multiple of H_kv=%d", s->H, s->H_kv);
    if (s->H / s->H_kv > 8)
        return fail(DKV_ERR_INVALID_ARG, "group size H/H_kv=%d > 8 is not supported", s->H / s->H_kv);
    if (s->head_dim != dkv::kHeadDim)
        return fail(DKV_ERR_INVALID_ARG, "head_dim=%d: only 128 is supported", s->head_dim);
    if (s->sink < 0 || s->recent < 0 || s->bin_width < 1)
        return fail(DKV_ERR_INVALID_ARG, "bad sink/recent/bin_width: %d/%d/%d", s->sink, s->recent,
                    s->bin_width);
    if (B < 1 || B > 512) return fail(DKV_ERR_INVALID_ARG, "B=%d out of [1, 512]", B);
    return DKV_OK;
}

// Split-K workspace and decode launch configuration of a finished plan.
dkv_status finish_plan(dkv_plan* p)
{
    cudaGetDevice(&p->device);
    p->use_mma = p->total_rows >= 1 && p->total_rows <= dkv::kMaxMmaRows;
    cudaError_t e;
    if (p->use_mma) {
        const int NHl = p->B * p->s.H_kv;
        std::vector<int32_t> len((size_t)p->s.L * NHl);
        if ((e = cudaMemcpy(len.data(), p->d_len, sizeof(int32_t) * len.size(), cudaMemcpyDeviceToHost)) != cudaSuccess)
            return cuda_fail(e, "read lengths");
        p->layer_rows.assign((size_t)p->s.L, 0);
        for (size_t h = 0; h < len.size(); ++h) p->layer_rows[h / NHl] += len[h];
        if ((e = dkv::decode_config_mma(p->G, p->B, 0, &p->cfg)) != cudaSuccess) return cuda_fail(e, "decode_config");
        if ((e = dkv::decode_config_mma(p->G, p->B, 1, &p->cfg_multi1)) != cudaSuccess ||
            (e = dkv::decode_config_mma(p->G, p->B, 2, &p->cfg_multi)) != cudaSuccess)
            return cuda_fail(e, "decode_config (multi-query)");
        p->nctas_cap = std::max({p->cfg.nctas, p->cfg_multi1.nctas, p->cfg_multi.nctas});
        p->warps_cap = std::max({p->cfg.nwarps, p->cfg_multi1.nwarps, p->cfg_multi.nwarps});
        p->cols_cap = dkv::kMaxCols;
    } else {
        if ((e = dkv::decode_config(p->G, p->B, &p->cfg)) != cudaSuccess) return cuda_fail(e, "decode_config");
        p->nctas_cap = p->cfg.nctas;
        p->warps_cap = p->cfg.nwarps;
        p->cols_cap = p->G;
    }
    p->slots = (int64_t)p->nctas_cap + p->B * p->s.H_kv;
    p->work = dkv::decode_workspace(p->nctas_cap, p->warps_cap, p->cols_cap, p->B * p->s.H_kv);
    dkv_status st = dalloc(&p->d_work, (size_t)p->work.total, "split-K workspace");
    if (st != DKV_OK) return st;
    st = dalloc(&p->d_status, 1, "status word");
    if (st != DKV_OK) return st;
    if ((e = cudaMemset(p->d_status, 0, sizeof(int32_t))) != cudaSuccess) return cuda_fail(e, "cudaMemset");
    st = dalloc(&p->d_slab_count, (size_t)2 * p->B * p->s.H_kv * p->cols_cap, "slab counters");
    if (st != DKV_OK) return st;
    if ((e = cudaMemset(p->d_slab_count, 0, sizeof(int32_t) * 2 * p->B * p->s.H_kv * p->cols_cap)) != cudaSuccess)
        return cuda_fail(e, "cudaMemset");
    return DKV_OK;
}

}  // namespace

namespace dkv {
// Page-backed buffers (dkv_vmm.cu).
dkv_status vmm_release_pages(dkv_vmm* m, const uint8_t* keep, int64_t npages, int64_t* freed);
int64_t vmm_bytes(const dkv_vmm* m);
int64_t vmm_page(const dkv_vmm* m);
}  // namespace dkv

namespace dkv {
// Lets other translation units of the library report through dkv_last_error().
dkv_status set_error(dkv_status st, const char* msg)
{
    snprintf(g_err, sizeof g_err, "%s", msg ? msg : "");
    return st;
}
}  // namespace dkv

extern "C" {

const char* dkv_last_error(void) { return g_err; }

// The map of dkv_map_pattern and dkv_map_pattern_inplace: slab offsets are the
// running sum of (len + reserve), or h * inplace_stride when that is > 0.
static dkv_status map_pattern_impl(const uint8_t* M_host, const int32_t* ctx_len_host, int32_t B,
                                   const dkv_shape* s, int32_t reserve_rows, int64_t inplace_stride,
                                   cudaStream_t stream, dkv_plan** out)
{
    if (!out) return fail(DKV_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!M_host || !ctx_len_host) return fail(DKV_ERR_INVALID_ARG, "M or ctx_len is NULL");
    dkv_status st = check_shape(s, B);
    if (st != DKV_OK) return st;
    if (reserve_rows < 0) return fail(DKV_ERR_INVALID_ARG, "reserve_rows=%d < 0", reserve_rows);
    const size_t nM = (size_t)s->L * s->H * s->D;
    for (size_t i = 0; i < nM; ++i)
        if (M_host[i] > 1) return fail(DKV_ERR_INVALID_ARG, "M[%zu]=%u is not 0/1", i, M_host[i]);
    int32_t Tmax = 0;
    for (int b = 0; b < B; ++b) {
        const int32_t T = ctx_len_host[b];
        if (T < 0) return fail(DKV_ERR_INVALID_ARG, "ctx_len[%d]=%d < 0", b, T);
        if ((int64_t)T > 65535LL * dkv::kMapChunk)
            return fail(DKV_ERR_INVALID_ARG, "ctx_len[%d]=%d too long", b, T);
        if ((int64_t)T - s->sink - s->recent > (int64_t)s->D * s->bin_width)
            return fail(DKV_ERR_RANGE, "ctx_len[%d]=%d needs more than D=%d bins of width %d", b, T,
                        s->D, s->bin_width);
        if (T > Tmax) Tmax = T;
    }
    if (inplace_stride > 0 && inplace_stride < (int64_t)Tmax + reserve_rows)
        return fail(DKV_ERR_INVALID_ARG, "T_stride=%lld < longest context %d + reserve %d", (long long)inplace_stride,
                    Tmax, reserve_rows);
    // Rows of one layer (with reserve) must fit the decode kernel's int32 row arithmetic.
    {
        int64_t layer_rows = 0;
        for (int b = 0; b < B; ++b) layer_rows += (int64_t)s->H_kv * ((int64_t)ctx_len_host[b] + reserve_rows);
        if (layer_rows > 0x7fffffffLL)
            return fail(DKV_ERR_INVALID_ARG, "a layer would hold %lld rows (> 2^31-1)", (long long)layer_rows);
    }

    dkv_plan* p = new (std::nothrow) dkv_plan();
    if (!p) return fail(DKV_ERR_OOM, "host allocation of the plan failed");
    p->s = *s;
    p->B = B;
    p->G = s->H / s->H_kv;
    p->reserve = reserve_rows;
    p->inplace_stride = inplace_stride;
    p->T_stride = inplace_stride;

    const int NH = s->L * B * s->H_kv;
    const int nchunks = Tmax > 0 ? (Tmax + dkv::kMapChunk - 1) / dkv::kMapChunk : 1;
    uint8_t *dM = nullptr, *dU = nullptr;
    int32_t *dTc = nullptr, *dcnt = nullptr;
    std::vector<int64_t> tail(2);
    auto cleanup = [&]() {
        cudaFree(dM);
        cudaFree(dU);
        cudaFree(dTc);
        cudaFree(dcnt);
    };
    if ((st = dalloc(&dM, nM, "pattern")) != DKV_OK ||
        (st = dalloc(&dU, (size_t)s->L * s->H_kv * s->D, "union pattern")) != DKV_OK ||
        (st = dalloc(&dTc, (size_t)B, "context lengths")) != DKV_OK ||
        (st = dalloc(&dcnt, (size_t)NH * nchunks, "chunk counts")) != DKV_OK ||
        (st = dalloc(&p->d_len, (size_t)NH, "lengths")) != DKV_OK ||
        (st = dalloc(&p->d_off, (size_t)NH + 1, "offsets")) != DKV_OK ||
        (st = dalloc(&p->d_ioff, (size_t)NH + 1, "index offsets")) != DKV_OK) {
        cleanup();
        release(p);
        return st;
    }
    cudaError_t e;
    if (nM && (e = cudaMemcpyAsync(dM, M_host, nM, cudaMemcpyHostToDevice, stream)) != cudaSuccess) {
        cleanup();
        release(p);
        return cuda_fail(e, "copy pattern");
    }
    if ((e = cudaMemcpyAsync(dTc, ctx_len_host, (size_t)B * 4, cudaMemcpyHostToDevice, stream)) != cudaSuccess) {
        cleanup();
        release(p);
        return cuda_fail(e, "copy ctx_len");
    }
    // Pass A: union, counts, scan (idx is allocated once its size is known).
    dkv::MapArgs ma{};
    ma.M = dM;
    ma.U = dU;
    ma.Tc = dTc;
    ma.chunk_cnt = dcnt;
    ma.len = p->d_len;
    ma.off = p->d_off;
    ma.ioff = p->d_ioff;
    ma.idx = nullptr;
    ma.L = s->L;
    ma.H = s->H;
    ma.Hkv = s->H_kv;
    ma.D = s->D;
    ma.B = B;
    ma.sink = s->sink;
    ma.recent = s->recent;
    ma.bin_width = s->bin_width;
    ma.reserve = reserve_rows;
    ma.nchunks = nchunks;
    ma.NH = NH;
    ma.stride = inplace_stride;
    if ((st = launched(dkv::launch_map(ma, stream), "map kernels")) != DKV_OK) {
        cleanup();
        release(p);
        return st;
    }
    // The one synchronisation: learn total and kept row counts.
    if ((e = cudaMemcpyAsync(&tail[0], p->d_off + NH, 8, cudaMemcpyDeviceToHost, stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(&tail[1], p->d_ioff + NH, 8, cudaMemcpyDeviceToHost, stream)) != cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess) {
        cleanup();
        release(p);
        return cuda_fail(e, "map: read totals");
    }
    p->total_rows = tail[0];
    p->kept_rows = tail[1];
    if ((st = dalloc(&p->d_idx, (size_t)p->kept_rows, "kept index list")) != DKV_OK) {
        cleanup();
        release(p);
        return st;
    }
    ma.idx = p->d_idx;
    if ((st = launched(dkv::launch_map_write(ma, stream), "map write kernel")) != DKV_OK) {
        cleanup();
        release(p);
        return st;
    }
    if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) {
        cleanup();
        release(p);
        return cuda_fail(e, "map: kernels");
    }
    cleanup();
    if (inplace_stride > 0) {
        // The in-place compaction streams whole slabs, longest first.
        std::vector<int32_t> len((size_t)NH), order((size_t)NH + 1, 0);
        if ((e = cudaMemcpy(len.data(), p->d_len, sizeof(int32_t) * NH, cudaMemcpyDeviceToHost)) != cudaSuccess) {
            release(p);
            return cuda_fail(e, "map: read lengths");
        }
        for (int h = 0; h < NH; ++h) order[(size_t)h] = h;
        std::stable_sort(order.begin(), order.begin() + NH, [&](int32_t x, int32_t y) { return len[x] > len[y]; });
        if ((st = dalloc(&p->d_order, (size_t)NH + 1, "slab order")) != DKV_OK) {
            release(p);
            return st;
        }
        if ((e = cudaMemcpy(p->d_order, order.data(), sizeof(int32_t) * (NH + 1), cudaMemcpyHostToDevice)) !=
            cudaSuccess) {
            release(p);
            return cuda_fail(e, "map: slab order");
        }
    }
    if ((st = finish_plan(p)) != DKV_OK) {
        release(p);
        return st;
    }
    *out = p;
    return ok();
}

dkv_status dkv_map_pattern(const uint8_t* M_host, const int32_t* ctx_len_host, int32_t B, const dkv_shape* s,
                           int32_t reserve_rows, cudaStream_t stream, dkv_plan** out)
{
    return map_pattern_impl(M_host, ctx_len_host, B, s, reserve_rows, 0, stream, out);
}

dkv_status dkv_map_pattern_inplace(const uint8_t* M_host, const int32_t* ctx_len_host, int32_t B,
                                   const dkv_shape* s, int32_t reserve_rows, int64_t T_stride, cudaStream_t stream,
                                   dkv_plan** out)
{
    if (out) *out = nullptr;
    if (T_stride < 1) return fail(DKV_ERR_INVALID_ARG, "T_stride=%lld < 1", (long long)T_stride);
    return map_pattern_impl(M_host, ctx_len_host, B, s, reserve_rows, T_stride, stream, out);
}

dkv_status dkv_plan_dense(const int32_t* ctx_len_host, int32_t B, const dkv_shape* s, int64_t T_stride,
                          cudaStream_t stream, dkv_plan** out)
{
    if (!out) return fail(DKV_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    if (!ctx_len_host) return fail(DKV_ERR_INVALID_ARG, "ctx_len is NULL");
    dkv_status st = check_shape(s, B);
    if (st != DKV_OK) return st;
    int32_t Tmax = 0;
    for (int b = 0; b < B; ++b) {
        if (ctx_len_host[b] < 0) return fail(DKV_ERR_INVALID_ARG, "ctx_len[%d] < 0", b);
        if (ctx_len_host[b] > Tmax) Tmax = ctx_len_host[b];
    }
    if (T_stride < Tmax || T_stride > 0x7fffffffLL)
        return fail(DKV_ERR_INVALID_ARG, "T_stride=%lld out of [max ctx_len=%d, 2^31)", (long long)T_stride, Tmax);
    if ((int64_t)B * s->H_kv * T_stride > 0x7fffffffLL)
        return fail(DKV_ERR_INVALID_ARG, "a layer would hold more than 2^31-1 rows");
    dkv_plan* p = new (std::nothrow) dkv_plan();
    if (!p) return fail(DKV_ERR_OOM, "host allocation of the plan failed");
    p->s = *s;
    p->B = B;
    p->G = s->H / s->H_kv;
    p->dense = 1;
    p->T_stride = T_stride;
    p->reserve = (int)(T_stride - Tmax);
    const int NH = s->L * B * s->H_kv;
    std::vector<int32_t> len(NH);
    std::vector<int64_t> off(NH + 1), ioff(NH + 1);
    int64_t run = 0;
    for (int h = 0; h < NH; ++h) {
        const int b = (h / s->H_kv) % B;
        len[h] = ctx_len_host[b];
        off[h] = (int64_t)h * T_stride;
        ioff[h] = run;
        run += len[h];
    }
    off[NH] = (int64_t)NH * T_stride;
    ioff[NH] = run;
    p->total_rows = off[NH];
    p->kept_rows = run;
    cudaError_t e;
    if ((st = dalloc(&p->d_len, (size_t)NH, "lengths")) != DKV_OK ||
        (st = dalloc(&p->d_off, (size_t)NH + 1, "offsets")) != DKV_OK ||
        (st = dalloc(&p->d_ioff, (size_t)NH + 1, "row prefix")) != DKV_OK) {
        release(p);
        return st;
    }
    if ((e = cudaMemcpyAsync(p->d_len, len.data(), (size_t)NH * 4, cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(p->d_off, off.data(), (size_t)(NH + 1) * 8, cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(p->d_ioff, ioff.data(), (size_t)(NH + 1) * 8, cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess) {
        release(p);
        return cuda_fail(e, "dense plan upload");
    }
    if ((st = finish_plan(p)) != DKV_OK) {
        release(p);
        return st;
    }
    *out = p;
    return ok();
}

dkv_status dkv_plan_query(const dkv_plan* p, int64_t* total_rows, int64_t* kept_rows, const int32_t** d_len,
                          const int64_t** d_off, const int64_t** d_ioff, const int32_t** d_idx)
{
    if (!p) return fail(DKV_ERR_INVALID_ARG, "plan is NULL");
    if (total_rows) *total_rows = p->total_rows;
    if (kept_rows) *kept_rows = p->kept_rows;
    if (d_len) *d_len = p->d_len;
    if (d_off) *d_off = p->d_off;
    if (d_ioff) *d_ioff = p->dense ? nullptr : p->d_ioff;
    if (d_idx) *d_idx = p->dense ? nullptr : p->d_idx;
    return ok();
}

dkv_status dkv_plan_read(const dkv_plan* p, int32_t* len_host, int64_t* off_host, int64_t* ioff_host,
                         int32_t* idx_host, cudaStream_t stream)
{
    if (!p) return fail(DKV_ERR_INVALID_ARG, "plan is NULL");
    const size_t NH = (size_t)p->s.L * p->B * p->s.H_kv;
    cudaError_t e = cudaSuccess;
    if (len_host && e == cudaSuccess)
        e = cudaMemcpyAsync(len_host, p->d_len, NH * 4, cudaMemcpyDeviceToHost, stream);
    if (off_host && e == cudaSuccess)
        e = cudaMemcpyAsync(off_host, p->d_off, (NH + 1) * 8, cudaMemcpyDeviceToHost, stream);
    if (!p->dense && ioff_host && e == cudaSuccess)
        e = cudaMemcpyAsync(ioff_host, p->d_ioff, (NH + 1) * 8, cudaMemcpyDeviceToHost, stream);
    if (!p->dense && idx_host && p->kept_rows > 0 && e == cudaSuccess)
        e = cudaMemcpyAsync(idx_host, p->d_idx, (size_t)p->kept_rows * 4, cudaMemcpyDeviceToHost, stream);
    if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e, "dkv_plan_read");
    return ok();
}

dkv_status dkv_compact_inplace(const dkv_plan* p, void* K, void* V, cudaStream_t stream)
{
    if (!p) return fail(DKV_ERR_INVALID_ARG, "plan is NULL");
    if (p->dense || p->inplace_stride <= 0)
        return fail(DKV_ERR_INVALID_ARG, "dkv_compact_inplace needs a plan from dkv_map_pattern_inplace");
    if (!K || !V) return fail(DKV_ERR_INVALID_ARG, "NULL K/V");
    if (!aligned16(K) || !aligned16(V)) return fail(DKV_ERR_INVALID_ARG, "K/V must be 16-byte aligned");
    if (K == V) return fail(DKV_ERR_INVALID_ARG, "K and V must be different buffers");
    dkv::CompactArgs a{};
    a.len = p->d_len;
    a.off = p->d_off;
    a.ioff = p->d_ioff;
    a.idx = p->d_idx;
    a.K = static_cast<const uint16_t*>(K);
    a.V = static_cast<const uint16_t*>(V);
    a.T_stride = p->inplace_stride;
    a.kept = p->kept_rows;
    a.NH = p->s.L * p->B * p->s.H_kv;
    dkv_status st =
        launched(dkv::launch_compact_inplace(a, p->d_order, p->d_order + a.NH, stream), "in-place compact kernel");
    return st == DKV_OK ? ok() : st;
}

dkv_status dkv_vmm_trim(dkv_vmm* m, const dkv_plan* p, int32_t guard_rows, int64_t* freed_bytes)
{
    if (freed_bytes) *freed_bytes = 0;
    if (!m || !p) return fail(DKV_ERR_INVALID_ARG, "NULL buffer or plan");
    if (p->inplace_stride <= 0) return fail(DKV_ERR_INVALID_ARG, "dkv_vmm_trim needs a plan from dkv_map_pattern_inplace");
    if (guard_rows < 16)
        return fail(DKV_ERR_INVALID_ARG, "guard_rows=%d < 16: decode reads whole 16-row tiles past a slab's last row",
                    guard_rows);
    const int64_t NH = (int64_t)p->s.L * p->B * p->s.H_kv;
    const int64_t need = NH * p->inplace_stride * dkv::kRowBytes;
    if (dkv::vmm_bytes(m) < need)
        return fail(DKV_ERR_INVALID_ARG, "buffer of %lld bytes is smaller than the plan's cache (%lld bytes)",
                    (long long)dkv::vmm_bytes(m), (long long)need);
    std::vector<int32_t> len((size_t)NH);
    cudaError_t e = cudaMemcpy(len.data(), p->d_len, sizeof(int32_t) * NH, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(e, "read lengths");
    const int64_t page = dkv::vmm_page(m), npages = dkv::vmm_bytes(m) / page;
    std::vector<uint8_t> keep((size_t)npages);
    dkv::vmm_pages_to_keep(len.data(), NH, p->inplace_stride, p->reserve, guard_rows, dkv::kRowBytes, page, npages,
                           keep.data());
    return dkv::vmm_release_pages(m, keep.data(), npages, freed_bytes);
}

dkv_status dkv_compact(const dkv_plan* p, const void* K, const void* V, int64_t T_stride, void* Kc, void* Vc,
                       cudaStream_t stream)
{
    if (!p) return fail(DKV_ERR_INVALID_ARG, "plan is NULL");
    if (p->dense) return fail(DKV_ERR_INVALID_ARG, "dkv_compact needs a plan from dkv_map_pattern");
    if (p->inplace_stride > 0)
        return fail(DKV_ERR_INVALID_ARG, "an in-place plan is compacted by dkv_compact_inplace");
    if (!K || !V || !Kc || !Vc) return fail(DKV_ERR_INVALID_ARG, "NULL K/V/Kc/Vc");
    if (!aligned16(K) || !aligned16(V) || !aligned16(Kc) || !aligned16(Vc))
        return fail(DKV_ERR_INVALID_ARG, "K/V/Kc/Vc must be 16-byte aligned");
    if (T_stride < 1) return fail(DKV_ERR_INVALID_ARG, "T_stride=%lld < 1", (long long)T_stride);
    dkv::CompactArgs a{};
    a.len = p->d_len;
    a.off = p->d_off;
    a.ioff = p->d_ioff;
    a.idx = p->d_idx;
    a.K = static_cast<const uint16_t*>(K);
    a.V = static_cast<const uint16_t*>(V);
    a.Kc = static_cast<uint16_t*>(Kc);
    a.Vc = static_cast<uint16_t*>(Vc);
    a.T_stride = T_stride;
    a.kept = p->kept_rows;
    a.NH = p->s.L * p->B * p->s.H_kv;
    dkv_status st = launched(dkv::launch_compact(a, stream), "compact kernel");
    return st == DKV_OK ? ok() : st;
}

namespace {

// Shared argument checks and marshalling of the three decode entry points.
// CTAs of a tensor-core launch over one layer: half the grid for a layer of
// fewer than kSmallLaunchRows kept rows. Half the SMs already draw the full HBM
// bandwidth, and a layer of 26 MB streams in a few microseconds, so fewer
// partials per slab (a shorter end-of-pass merge) count for more there:
// measured 3.5 % faster per step at a 16K context, equal at 128K, 1 % slower
// at 32K (50 MB layers), hence the bound.
constexpr int64_t kSmallLaunchRows = 65536;  // 32 MB of K and V rows
int launch_ctas(const dkv_plan* p, int layer, const dkv::DecodeConfig& cfg)
{
    if (!p->use_mma || layer < 0 || layer >= (int)p->layer_rows.size()) return cfg.nctas;
    return p->layer_rows[(size_t)layer] < kSmallLaunchRows ? std::max(1, cfg.nctas / 2) : cfg.nctas;
}

dkv_status decode_args(const dkv_plan* p, int32_t layer, const void* q, const void* k_new, const void* v_new,
                       int with_new, const int32_t* n_appended, void* Kc, void* Vc, float scale, float* out,
                       bool need_q, bool need_out, dkv::DecodeArgs* a)
{
    if (!p) return fail(DKV_ERR_INVALID_ARG, "plan is NULL");
    if (layer < 0 || layer >= p->s.L) return fail(DKV_ERR_INVALID_ARG, "layer=%d out of [0, %d)", layer, p->s.L);
    if (need_q && (!q || !Kc || !Vc)) return fail(DKV_ERR_INVALID_ARG, "NULL q/Kc/Vc");
    if (need_out && !out) return fail(DKV_ERR_INVALID_ARG, "NULL out");
    if ((k_new == nullptr) != (v_new == nullptr))
        return fail(DKV_ERR_INVALID_ARG, "k_new and v_new must both be given or both be NULL");
    if (!aligned16(q) || !aligned16(Kc) || !aligned16(Vc) || !aligned16(out) || !aligned16(k_new) ||
        !aligned16(v_new))
        return fail(DKV_ERR_INVALID_ARG, "q/k_new/v_new/Kc/Vc/out must be 16-byte aligned");
    if (!std::isfinite(scale)) return fail(DKV_ERR_INVALID_ARG, "scale is not finite");
    const int NHl = p->B * p->s.H_kv;
    *a = dkv::DecodeArgs{};
    a->q = static_cast<const uint16_t*>(q);
    a->k_new = static_cast<const uint16_t*>(k_new);
    a->v_new = static_cast<const uint16_t*>(v_new);
    a->n_app = n_appended;
    a->Kc = static_cast<uint16_t*>(Kc);
    a->Vc = static_cast<uint16_t*>(Vc);
    a->len = p->d_len + (int64_t)layer * NHl;
    a->off = p->d_off + (int64_t)layer * NHl;
    a->ioff = p->d_ioff + (int64_t)layer * NHl;
    a->work_o = p->d_work + p->work.work_o;
    a->work_ml = p->d_work + p->work.work_ml;
    a->warp_o = p->d_work + p->work.warp_o;
    a->warp_ml = p->d_work + p->work.warp_ml;
    if (!aligned16(a->work_o) || !aligned16(a->work_ml) || !aligned16(a->warp_o) || !aligned16(a->warp_ml))
        return fail(DKV_ERR_INVALID_ARG, "split-K workspace regions are not 16-byte aligned");
    a->out = out;
    a->slab_count = p->d_slab_count;
    a->merge_extra = fault("merge") ? 1 : 0;
    a->status = p->d_status;
    a->B = p->B;
    a->H = p->s.H;
    a->Hkv = p->s.H_kv;
    a->G = p->G;
    a->Q = 1;
    a->NC = p->G;
    a->reserve = p->reserve;
    a->append = with_new ? 1 : 0;
    const float sc = scale > 0.f ? scale : 1.0f / std::sqrt((float)dkv::kHeadDim);
    a->qscale = sc * 1.4426950408889634f;  // base-2 softmax: exp(x) = exp2(x log2 e)
    a->nctas = launch_ctas(p, layer, p->cfg);
    return DKV_OK;
}

// The split-K pass of one layer, with the merge fused in or not.
dkv_status launch_split_k(const dkv_plan* p, const dkv::DecodeArgs& a, bool fused, cudaStream_t stream)
{
    const char* what = fused ? "decode kernel" : "decode partial kernel";
    if (p->use_mma) {
        dkv::CacheMaps maps;
        const cudaError_t e = dkv::make_cache_maps(a.Kc, a.Vc, p->total_rows, &maps, fault("copy"));
        if (e != cudaSuccess) return cuda_fail(e, "tensor maps of the packed caches");
        return launched(fused ? dkv::launch_decode_mma_fused(a, maps, p->cfg, stream)
                              : dkv::launch_decode_mma_partial(a, maps, p->cfg, stream),
                        what);
    }
    return launched(fused ? dkv::launch_decode_fused(a, p->cfg, stream) : dkv::launch_decode_partial(a, p->cfg, stream),
                    what);
}

}  // namespace

dkv_status dkv_decode_attn(const dkv_plan* p, int32_t layer, const void* q, const void* k_new, const void* v_new,
                           const int32_t* n_appended, void* Kc, void* Vc, float scale, float* out,
                           cudaStream_t stream)
{
    dkv::DecodeArgs a;
    dkv_status st = decode_args(p, layer, q, k_new, v_new, k_new != nullptr, n_appended, Kc, Vc, scale, out,
                                true, true, &a);
    if (st != DKV_OK) return st;
    st = launch_split_k(p, a, true, stream);
    return st == DKV_OK ? ok() : st;
}

dkv_status dkv_decode_multi(const dkv_plan* p, int32_t layer, const void* q, int32_t num_queries,
                            const int32_t* n_appended, void* Kc, void* Vc, float scale, float* out,
                            cudaStream_t stream)
{
    dkv::DecodeArgs a;
    dkv_status st = decode_args(p, layer, q, nullptr, nullptr, 0, n_appended, Kc, Vc, scale, out, true, true, &a);
    if (st != DKV_OK) return st;
    if (num_queries < 1 || num_queries * p->G > dkv::kMaxCols)
        return fail(DKV_ERR_INVALID_ARG, "num_queries=%d: need 1 <= Q and Q*G <= %d (G=%d)", num_queries,
                    dkv::kMaxCols, p->G);
    if (!p->use_mma)
        return fail(DKV_ERR_INVALID_ARG, "multi-query decode needs the tensor-core kernel (a cache of < 2^31 rows)");
    a.Q = num_queries;
    a.NC = num_queries * p->G;
    // Q = 1 runs the decode step's kernel; more queries the multi-query kernels.
    const dkv::DecodeConfig& cfg = num_queries == 1 ? p->cfg : (a.NC > 8 ? p->cfg_multi : p->cfg_multi1);
    a.nctas = launch_ctas(p, layer, cfg);
    dkv::CacheMaps maps;
    const cudaError_t e = dkv::make_cache_maps(a.Kc, a.Vc, p->total_rows, &maps, fault("copy"));
    if (e != cudaSuccess) return cuda_fail(e, "tensor maps of the packed caches");
    st = launched(dkv::launch_decode_mma_fused(a, maps, cfg, stream), "multi-query decode kernel");
    return st == DKV_OK ? ok() : st;
}

dkv_status dkv_decode_partial(const dkv_plan* p, int32_t layer, const void* q, const void* k_new,
                              const void* v_new, const int32_t* n_appended, void* Kc, void* Vc, float scale,
                              cudaStream_t stream)
{
    dkv::DecodeArgs a;
    dkv_status st = decode_args(p, layer, q, k_new, v_new, k_new != nullptr, n_appended, Kc, Vc, scale,
                                nullptr, true, false, &a);
    if (st != DKV_OK) return st;
    st = launch_split_k(p, a, false, stream);
    return st == DKV_OK ? ok() : st;
}

dkv_status dkv_decode_combine(const dkv_plan* p, int32_t layer, const int32_t* n_appended, int32_t with_new_token,
                              float* out, cudaStream_t stream)
{
    dkv::DecodeArgs a;
    dkv_status st = decode_args(p, layer, nullptr, nullptr, nullptr, with_new_token, n_appended, nullptr,
                                nullptr, 1.f, out, false, true, &a);
    if (st != DKV_OK) return st;
    st = launched(dkv::launch_decode_combine(a, stream), "decode combine kernel");
    return st == DKV_OK ? ok() : st;
}

int64_t dkv_budget(double rho, int32_t L, int32_t H, int32_t D)
{
    if (!(rho >= 0.0 && rho <= 1.0) || L < 0 || H < 0 || D < 0) return -1;
    return (int64_t)std::floor(rho * (double)L * (double)H * (double)D + 0.5);
}

int64_t dkv_topk_workspace_bytes(void) { return dkv::topk_workspace_bytes(); }

dkv_status dkv_topk_mask(const float* P, int64_t n, int64_t K, uint8_t* M, void* workspace,
                         int64_t workspace_bytes, cudaStream_t stream)
{
    if (n < 0 || n >= ((int64_t)1 << 31)) return fail(DKV_ERR_INVALID_ARG, "n=%lld out of [0, 2^31)", (long long)n);
    if (K < 0 || K > n) return fail(DKV_ERR_INVALID_ARG, "K=%lld out of [0, n=%lld]", (long long)K, (long long)n);
    if (n > 0 && (!P || !M)) return fail(DKV_ERR_INVALID_ARG, "NULL P or M");
    if (n > 0 && K > 0 && K < n) {
        if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 3u) != 0 ||
            workspace_bytes < dkv::topk_workspace_bytes())
            return fail(DKV_ERR_INVALID_ARG, "workspace: need %lld bytes, 4-byte aligned",
                        (long long)dkv::topk_workspace_bytes());
    }
    const dkv_status st = launched(dkv::launch_topk(P, n, K, M, workspace, stream, fault("barrier")), "top-k kernels");
    return st == DKV_OK ? ok() : st;
}

dkv_status dkv_advance(const dkv_plan* p, int32_t* n_appended, cudaStream_t stream)
{
    if (!p || !n_appended) return fail(DKV_ERR_INVALID_ARG, "NULL plan or n_appended");
    dkv_status st = launched(dkv::launch_advance(n_appended, p->B, p->reserve, p->d_status, stream),
                             "advance kernel");
    return st == DKV_OK ? ok() : st;
}

dkv_status dkv_plan_status(const dkv_plan* p, int32_t* word, int32_t clear, cudaStream_t stream)
{
    if (!p || !word) return fail(DKV_ERR_INVALID_ARG, "NULL plan or word");
    cudaError_t e;
    if ((e = cudaMemcpyAsync(word, p->d_status, 4, cudaMemcpyDeviceToHost, stream)) != cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess)
        return cuda_fail(e, "read status word");
    if (clear && (e = cudaMemsetAsync(p->d_status, 0, 4, stream)) != cudaSuccess) return cuda_fail(e, "clear status");
    return ok();
}

void dkv_free(dkv_plan* p)
{
    if (!p) return;
    cudaDeviceSynchronize();
    release(p);
}

}  // extern "C"
