// One-time prune-and-pack (Sec. 3.4): Kc[off[h] + r] = K[h][idx[ioff[h] + r]],
// same for V, for every kept row r < len[h] of every slab h. A pure byte copy.
//
// The flat kept-row space [0, kept) is cut into 8-row pieces, one per warp; a
// half-warp moves one 256-byte row as 16 lanes x 16 bytes, so each warp
// instruction moves 512 contiguous bytes of K (or V). Every lane issues all of
// its 8 loads (K and V of 4 row pairs) before its stores to keep 128 bytes per
// lane in flight. Dropped rows are never read.
#include "dkv_internal.cuh"

namespace dkv {
namespace {

constexpr int kThreads = 256;
constexpr int kPairs = 4;                     // row pairs per warp
constexpr int kRowsPerWarp = 2 * kPairs;
constexpr int kRowsPerCta = kRowsPerWarp * (kThreads / 32);

__device__ __forceinline__ uint4 ld_stream(const uint4* p)
{
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

__device__ __forceinline__ void st_stream(uint4* p, const uint4& v)
{
    asm volatile("st.global.L1::no_allocate.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x),
                 "r"(v.y), "r"(v.z), "r"(v.w)
                 : "memory");
}

// Last slab h with ioff[h] <= row (skips empty slabs, whose ioff repeats).
__device__ __forceinline__ int slab_of(const int64_t* __restrict__ ioff, int NH, int64_t row)
{
    int lo = 0, hi = NH - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (ioff[mid] <= row)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

__global__ void __launch_bounds__(kThreads) compact_kernel(const CompactArgs a)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int half = lane >> 4, sub = lane & 15;
    const int64_t r0 = ((int64_t)blockIdx.x * (kThreads / 32) + warp) * kRowsPerWarp;
    if (r0 >= a.kept) return;
    int h = slab_of(a.ioff, a.NH, r0);

    uint4 kv[kPairs], vv[kPairs];
    int64_t dst[kPairs];
#pragma unroll
    for (int i = 0; i < kPairs; ++i) {
        const int64_t row = r0 + 2 * i + half;
        dst[i] = -1;
        if (row < a.kept) {
            int hr = h;
            while (a.ioff[hr + 1] <= row) ++hr;
            const int32_t ix = a.idx[row];
            const int64_t d = a.off[hr] + (row - a.ioff[hr]);
            if (in_bounds(ix >= 0 && ix < a.T_stride && d >= 0 && d < a.rows_cap, a.status)) {
                const int64_t src = (int64_t)hr * a.T_stride + ix;
                dst[i] = d;
                kv[i] = ld_stream(reinterpret_cast<const uint4*>(a.K + src * kHeadDim) + sub);
                vv[i] = ld_stream(reinterpret_cast<const uint4*>(a.V + src * kHeadDim) + sub);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < kPairs; ++i) {
        if (dst[i] >= 0) {
            st_stream(reinterpret_cast<uint4*>(a.Kc + dst[i] * kHeadDim) + sub, kv[i]);
            st_stream(reinterpret_cast<uint4*>(a.Vc + dst[i] * kHeadDim) + sub, vv[i]);
        }
    }
}

}  // namespace

// In-place prune-and-pack: slab h's kept rows move from rows h * T_stride +
// idx[r] to rows h * T_stride + r of the same buffer. idx is ascending, so
// idx[r] >= r: a row only moves towards the slab's start, and rows before the
// first dropped position stay where they are.
//
// One CTA per SM streams whole slabs, claimed from a list sorted by length
// (longest first) so the last slabs to start are short. A slab's moving rows
// go in chunks of kIpRows, in order: every thread loads its pieces of the
// chunk's source rows into registers, a CTA barrier waits for all of them,
// then the rows are stored at their destinations. A chunk's sources lie at or
// after its own first destination and after every earlier chunk's
// destinations, and the next chunk's stores come after this chunk's barrier,
// so no row is overwritten before it has been read. The index entries of the
// next chunk are loaded with this chunk's rows, off the critical path. Row
// loads bypass L1 (the buffer is written by this kernel).
namespace {

constexpr int kIpThreads = 512;
constexpr int kIpPer = 16;                               // 16-byte pieces per thread per chunk
constexpr int kIpWarps = kIpThreads / 32;
constexpr int kIpRows = kIpThreads * kIpPer / 32;        // rows per chunk (a row is 32 pieces: K, V)

// Warp-wide search for the first row r in [0, n) with idx[r] > r (the predicate
// is monotone: idx[r] - r is non-decreasing); n if none. Each round probes 32
// evenly spaced rows, so a 64K-row slab takes four dependent loads.
__device__ int first_moving_row(const int32_t* idx, int n, int lane)
{
    int lo = 0, hi = n;  // answer in [lo, hi]
    while (hi - lo > 0) {
        const int step = (hi - lo + 31) / 32;
        const int x = lo + lane * step;
        const bool p = x < hi && __ldg(idx + x) > x;
        const unsigned m = __ballot_sync(0xffffffffu, p);
        if (step == 1) return m ? lo + __ffs(m) - 1 : hi;
        if (m) {
            const int j = __ffs(m) - 1;  // x_j satisfies it, x_{j-1} does not
            hi = lo + j * step;
            lo = j ? lo + (j - 1) * step + 1 : lo;
        } else {
            lo += (hi - 1 - lo) / step * step + 1;  // past the last probed row
        }
    }
    return lo;
}

__global__ void __launch_bounds__(kIpThreads, 1)
    compact_inplace_kernel(const CompactArgs a, const int32_t* __restrict__ order, int32_t* claim)
{
    __shared__ int sh_h, sh_lo;
    uint16_t* K = const_cast<uint16_t*>(a.K);
    uint16_t* V = const_cast<uint16_t*>(a.V);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int kv = (lane >> 4) & 1, c = lane & 15;  // a warp moves whole rows: K pieces, then V pieces
    for (;;) {
        __syncthreads();  // the previous slab's values of sh_h / sh_lo are no longer read
        if (warp == 0) {
            int h = -1, lo = 0;
            int s = 0;
            if (lane == 0) s = atomicAdd(claim, 1);
            s = __shfl_sync(0xffffffffu, s, 0);
            if (s < a.NH) {
                h = __ldg(order + s);
                lo = first_moving_row(a.idx + __ldg(a.ioff + h), __ldg(a.len + h), lane);
            }
            if (lane == 0) {
                sh_h = h;
                sh_lo = lo;
            }
        }
        __syncthreads();
        const int h = sh_h;
        if (h < 0) return;
        const int n = __ldg(a.len + h);
        const int32_t* idx = a.idx + __ldg(a.ioff + h);
        const int64_t base = (int64_t)h * a.T_stride;
        int r0 = sh_lo;
        // Piece i of this thread: row r0 + warp + kIpWarps * i of the chunk.
        int nxt[kIpPer];
#pragma unroll
        for (int i = 0; i < kIpPer; ++i) {
            const int r = r0 + warp + kIpWarps * i;
            nxt[i] = r < n ? __ldg(idx + r) : -1;
        }
        for (; r0 < n; r0 += kIpRows) {
            uint4 v[kIpPer];
            int cur[kIpPer];
#pragma unroll
            for (int i = 0; i < kIpPer; ++i) {
                cur[i] = nxt[i];
                // A row only moves towards its slab's start, inside the slab's region.
                if (cur[i] >= 0 &&
                    !in_bounds(cur[i] >= r0 + warp + kIpWarps * i && cur[i] < a.T_stride, a.status))
                    cur[i] = -1;
                if (cur[i] >= 0) {
                    const uint16_t* src = (kv ? V : K) + (base + cur[i]) * kHeadDim;
                    v[i] = __ldcg(reinterpret_cast<const uint4*>(src) + c);
                }
            }
#pragma unroll
            for (int i = 0; i < kIpPer; ++i) {
                const int r = r0 + kIpRows + warp + kIpWarps * i;
                nxt[i] = r < n ? __ldg(idx + r) : -1;
            }
            __syncthreads();  // every source row of this chunk is read
#pragma unroll
            for (int i = 0; i < kIpPer; ++i) {
                if (cur[i] >= 0) {
                    const int64_t dst = base + r0 + warp + kIpWarps * i;
                    reinterpret_cast<uint4*>((kv ? V : K) + dst * kHeadDim)[c] = v[i];
                }
            }
        }
    }
}

}  // namespace

cudaError_t launch_compact_inplace(const CompactArgs& a, const int32_t* order, int32_t* claim, cudaStream_t st)
{
    if (a.kept == 0 || a.NH == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaMemsetAsync(claim, 0, sizeof(int32_t), st)) != cudaSuccess) return e;
    const int grid = a.NH < sms ? a.NH : sms;
    compact_inplace_kernel<<<grid, kIpThreads, 0, st>>>(a, order, claim);
    return cudaGetLastError();
}

cudaError_t launch_compact(const CompactArgs& a, cudaStream_t st)
{
    if (a.kept == 0) return cudaSuccess;
    const int64_t blocks = (a.kept + kRowsPerCta - 1) / kRowsPerCta;
    compact_kernel<<<(unsigned)blocks, kThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace dkv
