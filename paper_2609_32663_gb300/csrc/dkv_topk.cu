// Exact-budget pattern export (Eq. 3, App. A.3): M = TopKMask(P, K), the K
// largest of the n entries of P set to 1. Ties go to the lower flat index and
// NaN ranks below every number (+0 and -0 tie).
//
// Radix select over an order-preserving 32-bit key of each value:
//   pass p = 0..3   histogram of key digit p (bits 31-24, 23-16, 15-8, 7-0) over
//                   the keys that match the threshold's digits found so far;
//                   the next launch's prologue scans that histogram from the top
//                   to find the threshold's next digit and the rank left in it;
//   count           per CTA, the keys equal to the full threshold T;
//   mark            M[i] = key > T, or key == T and i is among the first k ties
//                   in index order (CTA prefix of the counts, then block scans).
// Each launch streams P once (4 n bytes); mark also writes M (n bytes).
#include "dkv.h"
#include "dkv_internal.cuh"

#include <cstdint>

namespace dkv {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kTkThreads = 256;
constexpr int kTkMaxCtas = 4096;
constexpr int kTkPerCta = 4096;  // entries per CTA before the grid grows

// Workspace (uint32): histograms [4][256], selection state [5] x (prefix, rank),
// per-CTA tie counts [kTkMaxCtas].
constexpr int kWsHist = 0;
constexpr int kWsState = 4 * 256;
constexpr int kWsTies = kWsState + 16;
constexpr int kWsWords = kWsTies + kTkMaxCtas;

__device__ __forceinline__ uint32_t order_key(float x)
{
    if (x != x) return 0u;  // NaN: below every number
    uint32_t u = __float_as_uint(x);
    if (u == 0x80000000u) u = 0u;  // -0 ranks as +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// State of pass p: threshold digits above pass p (prefix) and the rank (1-based,
// from the top) still sought among the keys that share them.
struct Sel {
    uint32_t prefix;
    uint32_t rank;
};

// Digit of pass p: bits [24 - 8p, 32 - 8p); keys "match" when their bits above
// that digit equal the prefix.
__device__ __forceinline__ uint32_t digit_of(uint32_t key, int p) { return (key >> (24 - 8 * p)) & 255u; }
__device__ __forceinline__ bool matches(uint32_t key, uint32_t prefix, int p)
{
    return p == 0 || (key >> (32 - 8 * p)) == (prefix >> (32 - 8 * p));
}

// State of pass p + 1 from the state and histogram of pass p: the digit d where
// the running count from the top first reaches the rank. One warp.
__device__ Sel next_sel(Sel s, const uint32_t* hist, int p, int lane)
{
    // Lane l owns bins 255 - 8 l .. 248 - 8 l (descending).
    uint32_t c[8], sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        c[i] = hist[255 - 8 * lane - i];
        sum += c[i];
    }
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
    }
    const uint32_t excl = incl - sum;
    const unsigned hit = __ballot_sync(kFull, excl < s.rank && incl >= s.rank);
    const int src = hit ? __ffs(hit) - 1 : 0;  // hit != 0: the rank lies within the matching keys
    uint32_t digit = 0, rank = 0;
    if (lane == src) {
        uint32_t cum = excl;
        for (int i = 0; i < 8; ++i) {
            if (cum + c[i] >= s.rank) {
                digit = 255u - 8u * lane - i;
                rank = s.rank - cum;
                break;
            }
            cum += c[i];
        }
    }
    digit = __shfl_sync(kFull, digit, src);
    rank = __shfl_sync(kFull, rank, src);
    return Sel{s.prefix | (digit << (24 - 8 * p)), rank};
}

// The selection state this launch works with: pass 0 starts from (0, K);
// later launches derive it from the previous pass and record it.
__device__ Sel load_sel(uint32_t* ws, int p, uint32_t K, Sel* sh)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) {
        Sel s{0u, K};
        if (p > 0) {
            const Sel prev{ws[kWsState + 2 * (p - 1)], ws[kWsState + 2 * (p - 1) + 1]};
            s = next_sel(prev, ws + kWsHist + 256 * (p - 1), p - 1, lane);
        }
        if (lane == 0) {
            *sh = s;
            if (blockIdx.x == 0) {
                ws[kWsState + 2 * p] = s.prefix;
                ws[kWsState + 2 * p + 1] = s.rank;
            }
        }
    }
    __syncthreads();
    return *sh;
}

__global__ void __launch_bounds__(kTkThreads) topk_hist_kernel(const float* P, int64_t n, uint32_t K, int p,
                                                               uint32_t* ws)
{
    __shared__ uint32_t h[256];
    __shared__ Sel sh;
    for (int i = threadIdx.x; i < 256; i += blockDim.x) h[i] = 0;
    const Sel s = load_sel(ws, p, K, &sh);
    const int lane = threadIdx.x & 31;
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i0 = (int64_t)blockIdx.x * blockDim.x; i0 < n; i0 += stride) {
        const int64_t i = i0 + threadIdx.x;
        bool take = false;
        uint32_t d = 0;
        if (i < n) {
            const uint32_t key = order_key(__ldg(P + i));
            take = matches(key, s.prefix, p);
            d = digit_of(key, p);
        }
        // Warp-aggregated increments: keys of a pattern share their top digits.
        const unsigned act = __ballot_sync(kFull, take);
        if (take) {
            const unsigned same = __match_any_sync(act, d);
            if (lane == __ffs(same) - 1) atomicAdd(&h[d], (uint32_t)__popc(same));
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 256; i += blockDim.x)
        if (h[i]) atomicAdd(ws + kWsHist + 256 * p + i, h[i]);
}

// Contiguous index range of CTA c.
__device__ __forceinline__ void cta_range(int64_t n, int64_t* lo, int64_t* hi)
{
    const int64_t per = (n + gridDim.x - 1) / gridDim.x;
    *lo = min(n, per * blockIdx.x);
    *hi = min(n, *lo + per);
}

__global__ void __launch_bounds__(kTkThreads) topk_count_kernel(const float* P, int64_t n, uint32_t K,
                                                                uint32_t* ws)
{
    __shared__ Sel sh;
    __shared__ uint32_t wsum[kTkThreads / 32];
    const Sel s = load_sel(ws, 4, K, &sh);  // the full threshold T and the ties to take
    int64_t lo, hi;
    cta_range(n, &lo, &hi);
    uint32_t cnt = 0;
    for (int64_t i = lo + threadIdx.x; i < hi; i += blockDim.x) cnt += order_key(__ldg(P + i)) == s.prefix;
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) cnt += __shfl_xor_sync(kFull, cnt, o);
    if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = cnt;
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t t = 0;
        for (int w = 0; w < kTkThreads / 32; ++w) t += wsum[w];
        ws[kWsTies + blockIdx.x] = t;
    }
}

__global__ void __launch_bounds__(kTkThreads) topk_mark_kernel(const float* P, int64_t n, uint8_t* M,
                                                               const uint32_t* ws)
{
    __shared__ uint32_t wsum[kTkThreads / 32];
    __shared__ uint32_t base_sh;
    const uint32_t T = ws[kWsState + 8], take = ws[kWsState + 9];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) {  // ties in the CTAs before this one
        uint32_t b = 0;
        for (int c = lane; c < (int)blockIdx.x; c += 32) b += ws[kWsTies + c];
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) b += __shfl_xor_sync(kFull, b, o);
        if (lane == 0) base_sh = b;
    }
    __syncthreads();
    uint32_t carry = base_sh;
    int64_t lo, hi;
    cta_range(n, &lo, &hi);
    for (int64_t i0 = lo; i0 < hi; i0 += blockDim.x) {
        const int64_t i = i0 + threadIdx.x;
        uint32_t key = 0;
        bool tie = false;
        if (i < hi) {
            key = order_key(__ldg(P + i));
            tie = key == T;
        }
        // Exclusive rank of this tie within the round, in index order.
        const unsigned bal = __ballot_sync(kFull, tie);
        const uint32_t in_warp = __popc(bal & ((1u << lane) - 1u));
        if (lane == 0) wsum[warp] = __popc(bal);
        __syncthreads();
        uint32_t before = 0, round_total = 0;
#pragma unroll
        for (int w = 0; w < kTkThreads / 32; ++w) {
            before += (w < warp) ? wsum[w] : 0u;
            round_total += wsum[w];
        }
        if (i < hi) M[i] = (key > T || (tie && carry + before + in_warp < take)) ? 1 : 0;
        carry += round_total;
        __syncthreads();  // wsum is rewritten next round
    }
}

}  // namespace

int64_t topk_workspace_bytes() { return (int64_t)kWsWords * 4; }

cudaError_t launch_topk(const float* P, int64_t n, int64_t K, uint8_t* M, void* workspace, cudaStream_t st)
{
    cudaError_t e;
    if (n == 0) return cudaSuccess;
    if (K == 0 || K == n) return cudaMemsetAsync(M, K == n ? 1 : 0, (size_t)n, st);
    uint32_t* ws = static_cast<uint32_t*>(workspace);
    if ((e = cudaMemsetAsync(ws, 0, sizeof(uint32_t) * kWsWords, st)) != cudaSuccess) return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const int64_t want = (n + kTkPerCta - 1) / kTkPerCta;
    const int grid = (int)(want < 1 ? 1 : (want > 4 * sms ? 4 * sms : want));
    for (int p = 0; p < 4; ++p) {
        topk_hist_kernel<<<grid, kTkThreads, 0, st>>>(P, n, (uint32_t)K, p, ws);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    topk_count_kernel<<<grid, kTkThreads, 0, st>>>(P, n, (uint32_t)K, ws);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    topk_mark_kernel<<<grid, kTkThreads, 0, st>>>(P, n, M, ws);
    return cudaGetLastError();
}

}  // namespace dkv
