// Exact-budget pattern export (Eq. 3, App. A.3): M = TopKMask(P, K), the K
// largest of the n entries of P set to 1. Ties go to the lower flat index and
// NaN ranks below every number (+0 and -0 tie).
//
// One cooperative launch: a radix select over an order-preserving 32-bit key of
// each value, in phases separated by grid barriers. CTA c owns the contiguous
// index range [lo_c, hi_c) (its warps equal parts of it) and reads it in
// phases 1, 2, 3 and 5 (from L2 after the first, while P fits there).
//   1  histogram of key bits 31-21 (2048 bins);
//   2  every CTA scans that histogram from the top for the bin holding rank K
//      (digit d1, rank k1 left inside it), then histograms bits 20-10 of the
//      keys whose top bits are d1;
//   3  likewise d2, k2, and a histogram of bits 9-0 of the keys matching d1 d2,
//      one per warp range;
//   4  d3 completes the threshold key T; k3 = ties at T to take; the keys equal
//      to T per warp range are bin d3 of that warp's histogram, and each CTA
//      publishes its total;
//   5  M[i] = key > T, or key == T and i is among the first k3 such indices
//      (prefix of the CTA counts, then block scans in index order).
// Histograms build in shared memory; a thread counts runs of equal bins in a
// register and adds a run when its bin changes (patterns are smooth, so runs
// are long), and a CTA adds its nonzero bins to the global histogram.
#include "dkv.h"
#include "dkv_internal.cuh"

#include <cstdint>
#include <mutex>

namespace dkv {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kTkThreads = 512;
constexpr int kTkWarps = kTkThreads / 32;
constexpr int kTkMaxCtas = 2048;
constexpr int kTkMinPerCta = 2048;        // entries per CTA before the grid grows
constexpr int kTkSpins = 1 << 24;         // bound on barrier polls (each an L2 round trip), and 2 s
constexpr int kTkSmem = kTkWarps * 1024 * 4;  // per-warp histograms of the last digit

// Workspace (uint32): status, barrier counter, histograms of the three digit
// passes, per-CTA tie counts.
constexpr int kWsStatus = 0;
constexpr int kWsBarrier = 1;
constexpr int kWsH1 = 16;
constexpr int kWsH2 = kWsH1 + 2048;
constexpr int kWsH3 = kWsH2 + 2048;
constexpr int kWsTies = kWsH3 + 1024;
constexpr int kWsZeroed = kWsTies;  // words cleared before each launch
constexpr int kWsWords = kWsTies + kTkMaxCtas;

__device__ __forceinline__ uint32_t order_key(float x)
{
    if (x != x) return 0u;  // NaN: below every number
    uint32_t u = __float_as_uint(x);
    if (u == 0x80000000u) u = 0u;  // -0 ranks as +0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__device__ __forceinline__ uint32_t ld_acquire(const uint32_t* p)
{
    uint32_t v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Grid barrier number `phase` (1, 2, ...): every CTA arrives once per phase on
// a counter zeroed before the launch. Bounded: false after kTkSpins polls (the
// status word is then set), and the caller returns.
__device__ bool grid_barrier(uint32_t* ws, uint32_t phase, uint32_t expected, int* ok_sh)
{
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t* ctr = ws + kWsBarrier;
        __threadfence();  // this CTA's histogram and count writes, ordered by the CTA barrier above
        asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
        const uint32_t target = phase * expected;
        int ok = 0;
        unsigned long long t0;
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
        for (int i = 0; i < kTkSpins; ++i) {
            if (ld_acquire(ctr) >= target) {
                ok = 1;
                break;
            }
            if ((i & 255) == 255) {  // and at most 2 s
                unsigned long long t;
                asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
                if (t - t0 > 2000000000ull) break;
            }
        }
        if (!ok) atomicOr(ws + kWsStatus, 1u);
        __threadfence();
        *ok_sh = ok;
    }
    __syncthreads();
    return *ok_sh != 0;
}

// Adds the run (bin, cnt) of this thread to the shared histogram.
__device__ __forceinline__ void flush_run(uint32_t* h, uint32_t bin, uint32_t cnt)
{
    if (cnt) atomicAdd(h + bin, cnt);
}

// Keys of the warp's range [wlo, whi) in steps of 32 consecutive entries, eight
// steps' loads issued together (P is read from L2 after the first phase, and
// one load per lane in flight would leave the loop latency bound). f(i, key)
// sees every entry of the range once, in index order within a lane.
template <class F>
__device__ __forceinline__ void for_keys(const float* P, int64_t wlo, int64_t whi, int lane, F f)
{
    constexpr int U = 8;
    for (int64_t i0 = wlo; i0 < whi; i0 += 32 * U) {
        float v[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t i = i0 + 32 * u + lane;
            v[u] = i < whi ? __ldg(P + i) : 0.f;
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            const int64_t i = i0 + 32 * u + lane;
            f(i, i < whi, order_key(v[u]));
        }
    }
}

// Histogram of digit (key >> shift) & mask over the warp ranges' keys whose
// bits above the digit equal `prefix` (all keys when pbits == 0), added to the
// global histogram g. PER_WARP: each warp counts into its own hw[warp][nbins]
// (kept for the caller) and the CTA sums them; else one shared h[nbins].
template <bool PER_WARP>
__device__ void histogram(const float* P, int64_t wlo, int64_t whi, int lane, uint32_t* h, int nbins, int shift,
                          uint32_t mask, int pbits, uint32_t prefix, uint32_t* g)
{
    const int nh = PER_WARP ? kTkWarps * nbins : nbins;
    for (int i = threadIdx.x; i < nh; i += blockDim.x) h[i] = 0;
    __syncthreads();
    uint32_t* mine = PER_WARP ? h + (threadIdx.x >> 5) * nbins : h;
    uint32_t run_bin = 0, run_cnt = 0;
    const int pshift = 32 - pbits;
    for_keys(P, wlo, whi, lane, [&](int64_t, bool in, uint32_t key) {
        if (!in || (pbits && (key >> pshift) != prefix)) return;
        const uint32_t bin = (key >> shift) & mask;
        if (bin != run_bin) {
            flush_run(mine, run_bin, run_cnt);
            run_bin = bin;
            run_cnt = 0;
        }
        ++run_cnt;
    });
    flush_run(mine, run_bin, run_cnt);
    __syncthreads();
    for (int i = threadIdx.x; i < nbins; i += blockDim.x) {
        uint32_t c = h[i];
        if (PER_WARP)
            for (int w = 1; w < kTkWarps; ++w) c += h[w * nbins + i];
        if (c) atomicAdd(g + i, c);
    }
}

// The bin of the global histogram g[nbins] that holds rank `rank` (1-based,
// counted from the largest bin down), and the rank left inside it. Every CTA
// computes it from the same counts. Thread t owns bins nbins-1-q t .. nbins-q-q t
// (q = nbins / blockDim, descending).
__device__ void select_bin(const uint32_t* g, int nbins, uint32_t rank, uint32_t* scratch, uint32_t* bin_out,
                           uint32_t* rank_out)
{
    const int q = nbins / kTkThreads;  // 4 or 2
    const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
    uint32_t c[4], sum = 0;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        c[i] = i < q ? __ldcg(g + nbins - 1 - q * t - i) : 0u;
        sum += c[i];
    }
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t v = __shfl_up_sync(kFull, incl, o);
        if (lane >= o) incl += v;
    }
    if (lane == 31) scratch[warp] = incl;
    __syncthreads();
    uint32_t before = 0;
    for (int w = 0; w < warp; ++w) before += scratch[w];
    const uint32_t excl = before + incl - sum;
    if (excl < rank && excl + sum >= rank) {  // exactly one thread: the rank lies in its bins
        uint32_t cum = excl;
        for (int i = 0; i < q; ++i) {
            if (cum + c[i] >= rank) {
                *bin_out = (uint32_t)(nbins - 1 - q * t - i);
                *rank_out = rank - cum;
                break;
            }
            cum += c[i];
        }
    }
    __syncthreads();
}

// arrivals: the CTAs each grid barrier counts, gridDim.x (one more only under
// fault injection, so that the first barrier's wait runs out).
__global__ void __launch_bounds__(kTkThreads) topk_kernel(const float* __restrict__ P, int n, uint32_t K,
                                                          uint8_t* __restrict__ M, uint32_t* ws, uint32_t arrivals)
{
    extern __shared__ uint32_t h[];  // [kTkWarps][1024]: phase 3's per-warp histograms; [2048] before
    __shared__ uint32_t scratch[kTkWarps];
    __shared__ uint32_t wties[kTkWarps];
    __shared__ uint32_t sel_bin, sel_rank, base_sh;
    __shared__ int ok_sh;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // CTA c owns [lo, hi); warp w of it owns the w-th of kTkWarps equal parts.
    const int64_t per = ((int64_t)n + gridDim.x - 1) / gridDim.x;
    const int64_t lo = min((int64_t)n, per * blockIdx.x), hi = min((int64_t)n, lo + per);
    const int64_t wlo = lo + (hi - lo) * warp / kTkWarps, whi = lo + (hi - lo) * (warp + 1) / kTkWarps;

    // 1: top 11 bits
    histogram<false>(P, wlo, whi, lane, h, 2048, 21, 2047u, 0, 0u, ws + kWsH1);
    if (!grid_barrier(ws, 1, arrivals, &ok_sh)) return;
    select_bin(ws + kWsH1, 2048, K, scratch, &sel_bin, &sel_rank);
    const uint32_t d1 = sel_bin, k1 = sel_rank;
    // 2: bits 20-10 of the keys in bin d1
    histogram<false>(P, wlo, whi, lane, h, 2048, 10, 2047u, 11, d1, ws + kWsH2);
    if (!grid_barrier(ws, 2, arrivals, &ok_sh)) return;
    select_bin(ws + kWsH2, 2048, k1, scratch, &sel_bin, &sel_rank);
    const uint32_t p22 = (d1 << 11) | sel_bin, k2 = sel_rank;
    // 3: bits 9-0 of the keys matching the 22-bit prefix, per warp
    histogram<true>(P, wlo, whi, lane, h, 1024, 0, 1023u, 22, p22, ws + kWsH3);
    if (!grid_barrier(ws, 3, arrivals, &ok_sh)) return;
    select_bin(ws + kWsH3, 1024, k2, scratch, &sel_bin, &sel_rank);
    const uint32_t T = (p22 << 10) | sel_bin, take = sel_rank;  // take the first `take` keys equal to T
    // 4: keys equal to T per warp range (bin d3 of the warp's histogram) and per CTA
    if (lane == 0) wties[warp] = h[warp * 1024 + sel_bin];
    __syncthreads();
    if (threadIdx.x == 0) {
        uint32_t s = 0;
        for (int w = 0; w < kTkWarps; ++w) s += wties[w];
        ws[kWsTies + blockIdx.x] = s;
    }
    if (!grid_barrier(ws, 4, arrivals, &ok_sh)) return;
    // 5: mark. Ties before this warp's range: the earlier CTAs', then the
    // earlier warps' of this CTA; within the range, ballots in index order.
    if (warp == 0) {
        uint32_t b = 0;
        for (int c = lane; c < (int)blockIdx.x; c += 32) b += __ldcg(ws + kWsTies + c);
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) b += __shfl_xor_sync(kFull, b, o);
        if (lane == 0) base_sh = b;
    }
    __syncthreads();
    uint32_t carry = base_sh;
    for (int w = 0; w < warp; ++w) carry += wties[w];
    const unsigned below = (1u << lane) - 1u;
    for_keys(P, wlo, whi, lane, [&](int64_t i, bool in, uint32_t key) {
        const bool tie = in && key == T;
        const unsigned bal = __ballot_sync(kFull, tie);
        if (in) M[i] = (key > T || (tie && carry + __popc(bal & below) < take)) ? 1 : 0;
        carry += __popc(bal);
    });
}

}  // namespace

int64_t topk_workspace_bytes() { return (int64_t)kWsWords * 4; }

cudaError_t launch_topk(const float* P, int64_t n, int64_t K, uint8_t* M, void* workspace, cudaStream_t st,
                        bool phantom_cta)
{
    cudaError_t e;
    if (n == 0) return cudaSuccess;
    if (K == 0 || K == n) return cudaMemsetAsync(M, K == n ? 1 : 0, (size_t)n, st);
    uint32_t* ws = static_cast<uint32_t*>(workspace);
    if ((e = cudaMemsetAsync(ws, 0, sizeof(uint32_t) * kWsZeroed, st)) != cudaSuccess) return e;
    // Device capacity, looked up once per device (the host cost of these calls
    // would otherwise dominate small exports).
    static std::mutex mu;
    static int cached_dev = -1, cached_cap = 0;
    int dev = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    int64_t cap = 0;
    {
        std::lock_guard<std::mutex> lock(mu);
        if (cached_dev != dev) {
            int sms = 0, per_sm = 0;
            if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
            if ((e = cudaFuncSetAttribute(topk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTkSmem)) !=
                cudaSuccess)
                return e;
            if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, topk_kernel, kTkThreads, kTkSmem)) !=
                cudaSuccess)
                return e;
            cached_cap = sms * (per_sm < 1 ? 1 : per_sm);
            cached_dev = dev;
        }
        cap = cached_cap;
    }
    // Every CTA must be resident at once (grid barriers): at most the device's
    // capacity, and no more CTAs than ranges of kTkMinPerCta entries.
    const int64_t want = (n + kTkMinPerCta - 1) / kTkMinPerCta;
    int grid = (int)(want < cap ? want : cap);
    if (grid > kTkMaxCtas) grid = kTkMaxCtas;
    if (grid < 1) grid = 1;
    int nn = (int)n;
    uint32_t KK = (uint32_t)K;
    uint32_t arrivals = (uint32_t)grid + (phantom_cta ? 1u : 0u);
    void* args[] = {(void*)&P, (void*)&nn, (void*)&KK, (void*)&M, (void*)&ws, (void*)&arrivals};
    return cudaLaunchCooperativeKernel((const void*)topk_kernel, dim3(grid), dim3(kTkThreads), args, kTkSmem, st);
}

}  // namespace dkv
