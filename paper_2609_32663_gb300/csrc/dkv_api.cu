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
    void* d_arena = nullptr;    // one allocation: the map's metadata and counters (the workspace too, dense plans)
    void* d_arena2 = nullptr;   // map plans: the index list and the workspace, sized after the map's one sync
    int32_t* d_len = nullptr;   // [NH]
    int64_t* d_off = nullptr;   // [NH+1]
    int64_t* d_ioff = nullptr;  // [NH+1]
    int32_t* d_idx = nullptr;   // [kept]
    int32_t* d_status = nullptr;
    float* d_work = nullptr;    // split-K partials
    int32_t* d_slab_count = nullptr;  // [B*H_kv][cols][2] arrival / written counters of the fused combine
    dkv::DecodeConfig cfg{};         // the decode step's kernel (cfg_f32 or cfg_mma)
    dkv::DecodeConfig cfg_f32{};     // fp32 kernel (caches of 2^31 rows or more)
    dkv::DecodeConfig cfg_mma{};     // tensor-core kernel of the decode step
    dkv::DecodeConfig cfg_multi1{};  // multi-query, one column tile (tensor-core plans)
    dkv::DecodeConfig cfg_multi{};   // multi-query, two column tiles (tensor-core plans)
    dkv::DecodeConfig cfg_tc{};      // multi-query, 17 to 64 columns on tcgen05 (tensor-core plans)
    dkv::WorkspaceLayout work{};     // carve-up of d_work
    int cols_cap = 0;                // columns the workspace and counters are sized for
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
    cudaFree(p->d_arena);
    cudaFree(p->d_arena2);
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

// Byte offsets of the plan's device arrays inside its one allocation, each on a
// 256-byte boundary.
struct ArenaLayout {
    size_t bytes = 0;
    template <class T>
    size_t take(size_t count)
    {
        const size_t off = (bytes + 255) / 256 * 256;
        bytes = off + std::max<size_t>(count, 1) * sizeof(T);
        return off;
    }
};

template <class T>
T* at(void* base, size_t off)
{
    return reinterpret_cast<T*>(static_cast<unsigned char*>(base) + off);
}

// Launch configurations of every decode kernel a plan may run (host queries,
// no device work), and the split-K workspace that serves all of them: slots for
// the largest grid plus the slabs of a layer, warp records for the largest grid
// x warps, kMaxCols columns.
dkv_status plan_configs(dkv_plan* p)
{
    cudaGetDevice(&p->device);
    cudaError_t e;
    if ((e = dkv::decode_config(p->G, p->B, &p->cfg_f32)) != cudaSuccess) return cuda_fail(e, "decode_config");
    if ((e = dkv::decode_config_mma(p->G, p->B, 0, &p->cfg_mma)) != cudaSuccess ||
        (e = dkv::decode_config_mma(p->G, p->B, 1, &p->cfg_multi1)) != cudaSuccess ||
        (e = dkv::decode_config_mma(p->G, p->B, 2, &p->cfg_multi)) != cudaSuccess)
        return cuda_fail(e, "decode_config (tensor cores)");
    if ((e = dkv::decode_config_tc(p->G, p->B, &p->cfg_tc)) != cudaSuccess) return cuda_fail(e, "decode_config (tcgen05)");
    // Warp records: the mma.sync and fp32 kernels (up to kMaxCols columns); CTA
    // partials: every kernel, up to kTcMaxCols columns (the tcgen05 kernel).
    int64_t ctas = p->cfg_tc.nctas, warp_records = 0;
    for (const dkv::DecodeConfig* c : {&p->cfg_f32, &p->cfg_mma, &p->cfg_multi1, &p->cfg_multi}) {
        ctas = std::max<int64_t>(ctas, c->nctas);
        warp_records = std::max<int64_t>(warp_records, (int64_t)c->nctas * c->nwarps);
    }
    p->cols_cap = dkv::kMaxCols;
    const int64_t NHl = (int64_t)p->B * p->s.H_kv;
    p->work = dkv::workspace_layout(ctas + NHl, dkv::kTcMaxCols, warp_records, dkv::kMaxCols);
    return DKV_OK;
}

// Places the counters (status word, then the fused combine's slab counters) as
// one int32 block that a single memset zeroes, and the split-K workspace.
struct ZeroBlock {
    size_t off = 0, count = 0;
};
ZeroBlock take_zeroed(ArenaLayout& lay, const dkv_plan* p, size_t extra)
{
    ZeroBlock z;
    z.count = 1 + (size_t)2 * p->B * p->s.H_kv * p->cols_cap + extra;
    z.off = lay.take<int32_t>(z.count);
    return z;
}

void place_zeroed(dkv_plan* p, const ZeroBlock& z)
{
    p->d_status = at<int32_t>(p->d_arena, z.off);
    p->d_slab_count = p->d_status + 1;
}

// The decode kernel of a plan whose row count is known.
void choose_kernel(dkv_plan* p)
{
    p->use_mma = p->total_rows >= 1 && p->total_rows <= dkv::kMaxMmaRows;
    p->cfg = p->use_mma ? p->cfg_mma : p->cfg_f32;
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
//
// Device work, all on `stream`: one allocation for the plan's metadata and
// counters (the map's inputs M and Tc live there too), one memset of the
// counters, the copies of M and Tc, the runs kernel (and, in place, the slab
// order), one read of the totals -- the only synchronisation -- then a second
// allocation, sized by the totals, for the index list and the split-K
// workspace, and the index list's write. The call returns without waiting for
// the write: later calls on `stream` are ordered after it.
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
    const int64_t NH64 = (int64_t)s->L * B * s->H_kv;
    if (NH64 > 0x7fffffffLL) return fail(DKV_ERR_INVALID_ARG, "L*B*H_kv=%lld slabs (> 2^31-1)", (long long)NH64);
    const int NH = (int)NH64;

    dkv_plan* p = new (std::nothrow) dkv_plan();
    if (!p) return fail(DKV_ERR_OOM, "host allocation of the plan failed");
    p->s = *s;
    p->B = B;
    p->G = s->H / s->H_kv;
    p->reserve = reserve_rows;
    p->inplace_stride = inplace_stride;
    p->T_stride = inplace_stride;
    auto bail = [&](dkv_status e) {
        release(p);
        return e;
    };
    p->cols_cap = dkv::kMaxCols;

    ArenaLayout lay;
    const size_t o_len = lay.take<int32_t>((size_t)NH), o_off = lay.take<int64_t>((size_t)NH + 1),
                 o_ioff = lay.take<int64_t>((size_t)NH + 1), o_nruns = lay.take<int32_t>((size_t)NH),
                 o_runs = lay.take<int2>((size_t)NH * (s->D + 2)), o_tail = lay.take<int64_t>((size_t)3 + s->L),
                 o_M = lay.take<uint8_t>(nM), o_Tc = lay.take<int32_t>((size_t)B),
                 o_order = inplace_stride > 0 ? lay.take<int32_t>((size_t)NH + 1) : 0;
    const ZeroBlock zb = take_zeroed(lay, p, 1);  // + the runs kernel's CTA counter
    if ((st = dalloc(reinterpret_cast<unsigned char**>(&p->d_arena), lay.bytes, "plan metadata")) != DKV_OK)
        return bail(st);
    p->d_len = at<int32_t>(p->d_arena, o_len);
    p->d_off = at<int64_t>(p->d_arena, o_off);
    p->d_ioff = at<int64_t>(p->d_arena, o_ioff);
    p->d_order = inplace_stride > 0 ? at<int32_t>(p->d_arena, o_order) : nullptr;
    place_zeroed(p, zb);

    cudaError_t e;
    if ((e = cudaMemsetAsync(p->d_status, 0, zb.count * sizeof(int32_t), stream)) != cudaSuccess)
        return bail(cuda_fail(e, "clear counters"));
    if (nM && (e = cudaMemcpyAsync(at<uint8_t>(p->d_arena, o_M), M_host, nM, cudaMemcpyHostToDevice, stream)) !=
                  cudaSuccess)
        return bail(cuda_fail(e, "copy pattern"));
    if ((e = cudaMemcpyAsync(at<int32_t>(p->d_arena, o_Tc), ctx_len_host, (size_t)B * 4, cudaMemcpyHostToDevice,
                             stream)) != cudaSuccess)
        return bail(cuda_fail(e, "copy ctx_len"));

    dkv::MapArgs ma{};
    ma.M = at<uint8_t>(p->d_arena, o_M);
    ma.Tc = at<int32_t>(p->d_arena, o_Tc);
    ma.runs = at<int2>(p->d_arena, o_runs);
    ma.nruns = at<int32_t>(p->d_arena, o_nruns);
    ma.len = p->d_len;
    ma.off = p->d_off;
    ma.ioff = p->d_ioff;
    ma.idx = nullptr;
    ma.tail = at<int64_t>(p->d_arena, o_tail);
    ma.done = reinterpret_cast<unsigned*>(p->d_status + zb.count - 1);
    ma.order = p->d_order;
    ma.L = s->L;
    ma.H = s->H;
    ma.Hkv = s->H_kv;
    ma.D = s->D;
    ma.B = B;
    ma.sink = s->sink;
    ma.recent = s->recent;
    ma.bin_width = s->bin_width;
    ma.reserve = reserve_rows;
    ma.NH = NH;
    ma.stride = inplace_stride;
    ma.status = p->d_status;
    if ((st = launched(dkv::launch_map(ma, stream), "map kernels")) != DKV_OK) return bail(st);
    // The one synchronisation: the totals (rows, kept rows, longest slab, rows of each layer).
    std::vector<int64_t> tail((size_t)3 + s->L);
    if ((e = cudaMemcpyAsync(tail.data(), ma.tail, sizeof(int64_t) * tail.size(), cudaMemcpyDeviceToHost, stream)) !=
            cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess)
        return bail(cuda_fail(e, "map: read totals"));
    p->total_rows = tail[0];
    p->kept_rows = tail[1];
    p->layer_rows.assign(tail.begin() + 3, tail.end());
    if ((st = plan_configs(p)) != DKV_OK) return bail(st);
    ArenaLayout lay2;
    const size_t o_idx = lay2.take<int32_t>((size_t)p->kept_rows), o_work = lay2.take<float>((size_t)p->work.total);
    if ((st = dalloc(reinterpret_cast<unsigned char**>(&p->d_arena2), lay2.bytes, "index list and workspace")) !=
        DKV_OK)
        return bail(st);
    p->d_idx = at<int32_t>(p->d_arena2, o_idx);
    p->d_work = at<float>(p->d_arena2, o_work);
    ma.idx = p->d_idx;
    if ((st = launched(dkv::launch_map_write(ma, (int)tail[2], stream), "map write kernel")) != DKV_OK)
        return bail(st);
    choose_kernel(p);
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
    auto bail = [&](dkv_status e) {
        release(p);
        return e;
    };
    if ((st = plan_configs(p)) != DKV_OK) return bail(st);
    // The uncompressed layout is given by the arguments: slab h holds the
    // sequence's Tc[b] rows at row h * T_stride.
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
    p->layer_rows.assign((size_t)s->L, 0);
    for (int h = 0; h < NH; ++h) p->layer_rows[(size_t)h / (B * s->H_kv)] += len[h];
    ArenaLayout lay;
    const size_t o_len = lay.take<int32_t>((size_t)NH), o_off = lay.take<int64_t>((size_t)NH + 1),
                 o_ioff = lay.take<int64_t>((size_t)NH + 1);
    const ZeroBlock zb = take_zeroed(lay, p, 0);
    const size_t o_work = lay.take<float>((size_t)p->work.total);
    if ((st = dalloc(reinterpret_cast<unsigned char**>(&p->d_arena), lay.bytes, "plan metadata")) != DKV_OK)
        return bail(st);
    p->d_len = at<int32_t>(p->d_arena, o_len);
    p->d_off = at<int64_t>(p->d_arena, o_off);
    p->d_ioff = at<int64_t>(p->d_arena, o_ioff);
    p->d_work = at<float>(p->d_arena, o_work);
    place_zeroed(p, zb);
    cudaError_t e;
    if ((e = cudaMemsetAsync(p->d_status, 0, zb.count * sizeof(int32_t), stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(p->d_len, len.data(), (size_t)NH * 4, cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(p->d_off, off.data(), (size_t)(NH + 1) * 8, cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaMemcpyAsync(p->d_ioff, ioff.data(), (size_t)(NH + 1) * 8, cudaMemcpyHostToDevice, stream)) != cudaSuccess ||
        (e = cudaStreamSynchronize(stream)) != cudaSuccess)
        return bail(cuda_fail(e, "dense plan upload"));
    choose_kernel(p);
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
    a.status = p->d_status;
    a.rows_cap = (int64_t)a.NH * p->inplace_stride;
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
    a.status = p->d_status;
    a.rows_cap = p->total_rows;
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
    a->rows_cap = p->total_rows;
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
    if (num_queries < 1 || (int64_t)num_queries * p->G > dkv::kTcMaxCols)
        return fail(DKV_ERR_INVALID_ARG, "num_queries=%d: need 1 <= Q and Q*G <= %d (G=%d)", num_queries,
                    dkv::kTcMaxCols, p->G);
    if (!p->use_mma)
        return fail(DKV_ERR_INVALID_ARG, "multi-query decode needs the tensor-core kernel (a cache of < 2^31 rows)");
    a.Q = num_queries;
    a.NC = num_queries * p->G;
    if (a.NC > dkv::kMaxCols) {
        // More columns than the mma.sync kernels' accumulator registers hold: the
        // tcgen05 kernel (accumulators in TMEM).
        a.nctas = p->cfg_tc.nctas;
        dkv::CacheMaps maps;
        const cudaError_t e = dkv::make_cache_maps(a.Kc, a.Vc, p->total_rows, &maps, fault("copy"), 16);
        if (e != cudaSuccess) return cuda_fail(e, "tensor maps of the packed caches");
        st = launched(dkv::launch_decode_tc(a, maps, p->cfg_tc, stream), "multi-query decode kernel (tcgen05)");
        return st == DKV_OK ? ok() : st;
    }
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
