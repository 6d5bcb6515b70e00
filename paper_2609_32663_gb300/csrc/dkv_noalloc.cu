// dkv_decode_attn_noalloc: decode attention for callers that may not allocate
// device memory. Some hosts own every byte of device memory themselves -- a
// serving engine or plugin framework that hands out buffers from its own pool
// and forbids cudaMalloc/cudaFree (they synchronise the whole device and would
// fragment the pool mid-run). Such a caller cannot create a dkv_plan, whose
// split-K workspace comes from cudaMalloc. This entry point takes the plan's
// metadata as caller-provided device arrays and keeps its split-K partials in
// a fixed, file-scope device array instead of allocated memory.
//
// The array is part of the library image: every GPU that loads libdkv.so holds
// it (kScratchBytes) until the process exits. All calls share it and it keeps
// whatever the previous call left there; the kernels write every partial they
// later read, so nothing in it needs clearing except the fallback status word,
// which each call zeroes. Calls whose kernels overlap on the GPU (different
// streams, or different host threads) race on the array.
#include "dkv.h"
#include "dkv_internal.cuh"

#include <cuda.h>

#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <map>
#include <mutex>
#include <tuple>
#include <vector>

namespace {

// 8 MiB: split-K records of (CTAs + sequences x KV heads + warps of the grid) x
// group size x 130 floats, plus one status word at the end.
constexpr size_t kScratchBytes = size_t(8) << 20;
constexpr size_t kStatusOffset = kScratchBytes - 256;

static __device__ __align__(256) unsigned char g_decode_scratch[kScratchBytes];

// Per CUDA context (not per device ordinal: a context that is destroyed and
// made again, e.g. after cudaDeviceReset, loads the library's module again and
// the array moves), looked up by the context's process-unique ID:
//   - the device address of g_decode_scratch (in host code the symbol names a
//     host-side stand-in, never the device memory);
//   - the fp32 decode kernel's launch configuration for each (G, B), so that a
//     call does not set kernel attributes and query occupancy every time.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

std::mutex g_setup_mu;
std::vector<std::pair<unsigned long long, void*>> g_scratch_addr;  // (context ID, device address)
std::map<std::tuple<unsigned long long, int, int>, dkv::DecodeConfig> g_configs;  // (context ID, G, B)

template <class F>
F driver_fn(const char* name)
{
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) != cudaSuccess ||
        q != cudaDriverEntryPointSuccess)
        return nullptr;
    return reinterpret_cast<F>(p);
}

// ID of the calling thread's current context; the runtime's primary context of
// the current device is made current first if none is.
cudaError_t current_context_id(unsigned long long* id)
{
    static const CtxGetCurrentFn get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
    static const CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
    if (!get_current || !get_id) return cudaErrorNotSupported;
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS) return cudaErrorDeviceUninitialized;
    if (!ctx) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaSetDevice(dev);  // initialises the device's primary context
        if (e != cudaSuccess) return e;
        if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return cudaErrorDeviceUninitialized;
    }
    return get_id(ctx, id) == CUDA_SUCCESS ? cudaSuccess : cudaErrorDeviceUninitialized;
}

// The device address of the array and the launch configuration for (G, B) in
// the current context, looked up on the context's first call.
cudaError_t setup_for_current_context(int G, int B, void** scratch, dkv::DecodeConfig* cfg)
{
    unsigned long long id = 0;
    cudaError_t e = current_context_id(&id);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lk(g_setup_mu);
    void* addr = nullptr;
    for (const auto& kv : g_scratch_addr)
        if (kv.first == id) addr = kv.second;
    if (!addr) {
        e = cudaGetSymbolAddress(&addr, g_decode_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr.emplace_back(id, addr);
    }
    const auto key = std::make_tuple(id, G, B);
    auto it = g_configs.find(key);
    if (it == g_configs.end()) {
        dkv::DecodeConfig c{};
        if ((e = dkv::decode_config(G, B, &c)) != cudaSuccess) return e;
        it = g_configs.emplace(key, c).first;
    }
    *scratch = addr;
    *cfg = it->second;
    return cudaSuccess;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

namespace dkv {
dkv_status set_error(dkv_status st, const char* msg);  // dkv_api.cu
}

extern "C" dkv_status dkv_decode_attn_noalloc(const dkv_shape* s, int32_t B, int32_t layer, int32_t reserve_rows,
                                              const int32_t* d_len, const int64_t* d_off, const int64_t* d_ioff,
                                              const void* q, const void* k_new, const void* v_new,
                                              const int32_t* n_appended, void* Kc, void* Vc, float scale,
                                              float* out, int32_t* status, cudaStream_t stream)
{
    char msg[256];
    auto bad = [&](dkv_status st, const char* fmt, ...) {
        va_list ap;
        va_start(ap, fmt);
        vsnprintf(msg, sizeof msg, fmt, ap);
        va_end(ap);
        return dkv::set_error(st, msg);
    };
    if (!s) return bad(DKV_ERR_INVALID_ARG, "shape is NULL");
    if (s->L < 1 || s->H < 1 || s->H_kv < 1 || s->H % s->H_kv != 0 || s->H / s->H_kv > 8)
        return bad(DKV_ERR_INVALID_ARG, "bad head geometry H=%d H_kv=%d", s->H, s->H_kv);
    if (s->head_dim != dkv::kHeadDim) return bad(DKV_ERR_INVALID_ARG, "head_dim=%d: only 128", s->head_dim);
    if (B < 1 || B > 512) return bad(DKV_ERR_INVALID_ARG, "B=%d out of [1, 512]", B);
    if (layer < 0 || layer >= s->L) return bad(DKV_ERR_INVALID_ARG, "layer=%d out of [0, %d)", layer, s->L);
    if (reserve_rows < 0) return bad(DKV_ERR_INVALID_ARG, "reserve_rows=%d < 0", reserve_rows);
    if (!d_len || !d_off || !d_ioff || !q || !Kc || !Vc || !out)
        return bad(DKV_ERR_INVALID_ARG, "NULL metadata, q, Kc, Vc or out");
    if ((k_new == nullptr) != (v_new == nullptr))
        return bad(DKV_ERR_INVALID_ARG, "k_new and v_new must both be given or both be NULL");
    if (!aligned16(q) || !aligned16(Kc) || !aligned16(Vc) || !aligned16(out) || !aligned16(k_new) ||
        !aligned16(v_new))
        return bad(DKV_ERR_INVALID_ARG, "q/k_new/v_new/Kc/Vc/out must be 16-byte aligned");
    if (!std::isfinite(scale)) return bad(DKV_ERR_INVALID_ARG, "scale is not finite");

    const int G = s->H / s->H_kv;
    void* scratch = nullptr;
    dkv::DecodeConfig cfg{};
    cudaError_t e = setup_for_current_context(G, B, &scratch, &cfg);
    if (e != cudaSuccess) return bad(DKV_ERR_CUDA, "scratch set-up: %s", cudaGetErrorString(e));
    const int NHl = B * s->H_kv;
    const dkv::WorkspaceLayout lay = dkv::decode_workspace(cfg.nctas, cfg.nwarps, G, NHl);
    const size_t need = (size_t)lay.total * sizeof(float);
    if (need > kStatusOffset)
        return bad(DKV_ERR_INVALID_ARG,
                   "split-K partials need %zu bytes (%lld slots x G=%d); the static scratch holds %zu", need,
                   (long long)cfg.nctas + NHl, G, (size_t)kStatusOffset);

    float* work = static_cast<float*>(scratch);
    int32_t* status_word = status;
    if (!status_word) {
        status_word = reinterpret_cast<int32_t*>(static_cast<unsigned char*>(scratch) + kStatusOffset);
        if ((e = cudaMemsetAsync(status_word, 0, sizeof(int32_t), stream)) != cudaSuccess)
            return bad(DKV_ERR_CUDA, "clear status word: %s", cudaGetErrorString(e));
    }

    dkv::DecodeArgs a{};
    a.q = static_cast<const uint16_t*>(q);
    a.k_new = static_cast<const uint16_t*>(k_new);
    a.v_new = static_cast<const uint16_t*>(v_new);
    a.n_app = n_appended;
    a.Kc = static_cast<uint16_t*>(Kc);
    a.Vc = static_cast<uint16_t*>(Vc);
    a.len = d_len + (int64_t)layer * NHl;
    a.off = d_off + (int64_t)layer * NHl;
    a.ioff = d_ioff + (int64_t)layer * NHl;
    a.work_o = work + lay.work_o;
    a.work_ml = work + lay.work_ml;
    a.warp_o = work + lay.warp_o;
    a.warp_ml = work + lay.warp_ml;
    if (!aligned16(a.work_o) || !aligned16(a.work_ml) || !aligned16(a.warp_o) || !aligned16(a.warp_ml))
        return bad(DKV_ERR_INVALID_ARG, "split-K workspace regions are not 16-byte aligned");
    a.out = out;
    a.status = status_word;
    a.B = B;
    a.H = s->H;
    a.Hkv = s->H_kv;
    a.G = G;
    a.Q = 1;
    a.NC = G;
    a.reserve = reserve_rows;
    a.append = k_new ? 1 : 0;
    const float sc = scale > 0.f ? scale : 1.0f / std::sqrt((float)dkv::kHeadDim);
    a.qscale = sc * 1.4426950408889634f;
    a.nctas = cfg.nctas;
    if ((e = dkv::launch_decode_partial(a, cfg, stream)) != cudaSuccess)
        return bad(DKV_ERR_CUDA, "decode partial kernel: %s", cudaGetErrorString(e));
    if ((e = dkv::launch_decode_combine(a, stream)) != cudaSuccess)
        return bad(DKV_ERR_CUDA, "decode combine kernel: %s", cudaGetErrorString(e));
    return dkv::set_error(DKV_OK, "");
}
