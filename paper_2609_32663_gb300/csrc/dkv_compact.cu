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
            const int64_t src = (int64_t)hr * a.T_stride + a.idx[row];
            dst[i] = a.off[hr] + (row - a.ioff[hr]);
            kv[i] = ld_stream(reinterpret_cast<const uint4*>(a.K + src * kHeadDim) + sub);
            vv[i] = ld_stream(reinterpret_cast<const uint4*>(a.V + src * kHeadDim) + sub);
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
// first dropped position stay where they are. One CTA walks a slab in chunks of
// kInChunk rows: it loads the chunk's source rows into registers, waits at a
// barrier for all of them, then stores. A chunk's sources lie at or after its
// own destinations and strictly after the previous chunks' destinations, and
// the next chunk's destinations come after this chunk's barrier, so no row is
// overwritten before it has been read. Loads bypass L1 (the buffer is written
// by this kernel).
constexpr int kInThreads = 256;
constexpr int kInChunk = 64;                               // rows per chunk
constexpr int kInPer = kInChunk * 2 * 16 / kInThreads;     // 16-byte pieces per thread per chunk (K and V)

__global__ void __launch_bounds__(kInThreads) compact_inplace_kernel(const CompactArgs a)
{
    uint16_t* K = const_cast<uint16_t*>(a.K);
    uint16_t* V = const_cast<uint16_t*>(a.V);
    for (int h = blockIdx.x; h < a.NH; h += gridDim.x) {
        const int n = a.len[h];
        const int32_t* idx = a.idx + a.ioff[h];
        const int64_t base = (int64_t)h * a.T_stride;
        // First row that moves: idx[r] - r is non-decreasing, so a binary search.
        int lo = 0, hi = n;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (__ldg(idx + mid) > mid)
                hi = mid;
            else
                lo = mid + 1;
        }
        for (int r0 = lo; r0 < n; r0 += kInChunk) {
            uint4 v[kInPer];
            int64_t dst[kInPer];
#pragma unroll
            for (int k = 0; k < kInPer; ++k) {
                const int piece = threadIdx.x + k * kInThreads;  // (row, K/V, 16-byte chunk)
                const int r = r0 + piece / 32, kv = (piece / 16) & 1, c = piece & 15;
                dst[k] = -1;
                if (r < n) {
                    const uint16_t* src = (kv ? V : K) + (base + __ldg(idx + r)) * kHeadDim;
                    v[k] = __ldcg(reinterpret_cast<const uint4*>(src) + c);
                    dst[k] = ((base + r) * kHeadDim) / 8 + c;  // in uint4 units
                }
            }
            __syncthreads();  // every source row of this chunk is read
#pragma unroll
            for (int k = 0; k < kInPer; ++k) {
                const int piece = threadIdx.x + k * kInThreads;
                const int kv = (piece / 16) & 1;
                if (dst[k] >= 0) reinterpret_cast<uint4*>(kv ? V : K)[dst[k]] = v[k];
            }
        }
    }
}

cudaError_t launch_compact_inplace(const CompactArgs& a, cudaStream_t st)
{
    if (a.kept == 0 || a.NH == 0) return cudaSuccess;
    int dev = 0, sms = 0;
    cudaError_t e;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const int grid = a.NH < 8 * sms ? a.NH : 8 * sms;
    compact_inplace_kernel<<<grid, kInThreads, 0, st>>>(a);
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
