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

cudaError_t launch_compact(const CompactArgs& a, cudaStream_t st)
{
    if (a.kept == 0) return cudaSuccess;
    const int64_t blocks = (a.kept + kRowsPerCta - 1) / kRowsPerCta;
    compact_kernel<<<(unsigned)blocks, kThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace dkv
