// Pattern -> positions map (Sec. 3.4, Eqs. 4-5 and the GQA union).
//
// Four stream-ordered kernels, no device-wide waits:
//   union_kernel   U[l][g][d] = OR_j M[l][g*G + j][d]       (GQA union of bins)
//   count_kernel   per (slab, chunk of 8192 positions): kept count via warp ballot
//   scan_kernel    one CTA: per-slab lengths, chunk bases, slab offsets (int64)
//   write_kernel   recomputes the keep bits, ballot + popc + CTA scan -> idx
// keep(p) = p < S  or  p >= Tc - R  or  U[l][g][(Tc - R - 1 - p) / W].
#include "dkv_internal.cuh"

namespace dkv {
namespace {

__global__ void union_kernel(const uint8_t* __restrict__ M, uint8_t* __restrict__ U, int L, int H,
                             int Hkv, int D)
{
    const int G = H / Hkv;
    const int64_t n = (int64_t)L * Hkv * D;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int d = (int)(i % D);
        const int64_t lg = i / D;  // l*Hkv + g
        const uint8_t* row = M + (lg * G) * D + d;
        uint8_t u = 0;
        for (int j = 0; j < G; ++j) u |= row[(int64_t)j * D];
        U[i] = u;
    }
}

// Retention decision of KV head slab (layer, g) at position p of a Tc-token context.
__device__ __forceinline__ bool keep_pos(const uint8_t* __restrict__ Urow, int p, int Tc, int S,
                                         int R, int W)
{
    if (p < S || p >= Tc - R) return true;
    return Urow[(Tc - R - 1 - p) / W] != 0;
}

struct SlabView {
    const uint8_t* Urow;
    int Tc;
};

__device__ __forceinline__ SlabView slab_view(const MapArgs& a, int h)
{
    const int g = h % a.Hkv;
    const int b = (h / a.Hkv) % a.B;
    const int l = h / (a.Hkv * a.B);
    return SlabView{a.U + ((int64_t)l * a.Hkv + g) * a.D, a.Tc[b]};
}

constexpr int kMapThreads = 256;
constexpr int kMapIters = kMapChunk / kMapThreads;  // 32 positions per thread

__global__ void __launch_bounds__(kMapThreads) count_kernel(const MapArgs a)
{
    const int h = blockIdx.x, c = blockIdx.y;
    const SlabView v = slab_view(a, h);
    const int base = c * kMapChunk;
    int cnt = 0;
    if (base < v.Tc) {
        for (int k = 0; k < kMapIters; ++k) {
            const int p = base + k * kMapThreads + threadIdx.x;
            const bool kp = p < v.Tc && keep_pos(v.Urow, p, v.Tc, a.sink, a.recent, a.bin_width);
            const unsigned bal = __ballot_sync(0xffffffffu, kp);
            cnt += __popc(bal);  // identical in every lane of the warp
        }
    }
    __shared__ int warp_cnt[kMapThreads / 32];
    if ((threadIdx.x & 31) == 0) warp_cnt[threadIdx.x >> 5] = cnt;
    __syncthreads();
    if (threadIdx.x == 0) {
        int s = 0;
        for (int w = 0; w < kMapThreads / 32; ++w) s += warp_cnt[w];
        a.chunk_cnt[(int64_t)h * a.nchunks + c] = s;
    }
}

// One CTA. Pass 1: slab lengths, and chunk counts turned into exclusive chunk
// bases in place. Pass 2: exclusive scans of len+reserve (off) and len (ioff)
// over the flat slab order, as a CTA-wide scan of per-thread partial sums.
constexpr int kScanThreads = 1024;

__global__ void __launch_bounds__(kScanThreads) scan_kernel(const MapArgs a)
{
    for (int h = threadIdx.x; h < a.NH; h += kScanThreads) {
        int32_t* cc = a.chunk_cnt + (int64_t)h * a.nchunks;
        int s = 0;
        for (int c = 0; c < a.nchunks; ++c) {
            const int n = cc[c];
            cc[c] = s;
            s += n;
        }
        a.len[h] = s;
    }
    __syncthreads();

    const int per = (a.NH + kScanThreads - 1) / kScanThreads;
    const int h0 = min(a.NH, (int)threadIdx.x * per);
    const int h1 = min(a.NH, h0 + per);
    int64_t s_off = 0, s_ioff = 0;
    for (int h = h0; h < h1; ++h) {
        s_off += (int64_t)a.len[h] + a.reserve;
        s_ioff += a.len[h];
    }
    __shared__ int64_t sh_off[kScanThreads], sh_ioff[kScanThreads];
    sh_off[threadIdx.x] = s_off;
    sh_ioff[threadIdx.x] = s_ioff;
    __syncthreads();
    // Hillis-Steele inclusive scan over the per-thread sums.
    for (int d = 1; d < kScanThreads; d <<= 1) {
        int64_t vo = 0, vi = 0;
        if ((int)threadIdx.x >= d) {
            vo = sh_off[threadIdx.x - d];
            vi = sh_ioff[threadIdx.x - d];
        }
        __syncthreads();
        sh_off[threadIdx.x] += vo;
        sh_ioff[threadIdx.x] += vi;
        __syncthreads();
    }
    int64_t run_off = sh_off[threadIdx.x] - s_off;
    int64_t run_ioff = sh_ioff[threadIdx.x] - s_ioff;
    for (int h = h0; h < h1; ++h) {
        a.off[h] = a.stride > 0 ? (int64_t)h * a.stride : run_off;  // in place: the slab's own dense rows
        a.ioff[h] = run_ioff;
        run_off += (int64_t)a.len[h] + a.reserve;
        run_ioff += a.len[h];
    }
    if (threadIdx.x == kScanThreads - 1) {
        a.off[a.NH] = a.stride > 0 ? (int64_t)a.NH * a.stride : sh_off[kScanThreads - 1];
        a.ioff[a.NH] = sh_ioff[kScanThreads - 1];
    }
}

__global__ void __launch_bounds__(kMapThreads) write_kernel(const MapArgs a)
{
    const int h = blockIdx.x, c = blockIdx.y;
    const SlabView v = slab_view(a, h);
    const int base = c * kMapChunk;
    if (base >= v.Tc) return;  // uniform over the CTA
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    __shared__ int warp_cnt[kMapThreads / 32];
    int64_t out = a.ioff[h] + a.chunk_cnt[(int64_t)h * a.nchunks + c];
    for (int k = 0; k < kMapIters; ++k) {
        const int p = base + k * kMapThreads + threadIdx.x;
        const bool kp = p < v.Tc && keep_pos(v.Urow, p, v.Tc, a.sink, a.recent, a.bin_width);
        const unsigned bal = __ballot_sync(0xffffffffu, kp);
        if (lane == 0) warp_cnt[warp] = __popc(bal);
        __syncthreads();
        int before = 0, total = 0;
#pragma unroll
        for (int w = 0; w < kMapThreads / 32; ++w) {
            const int n = warp_cnt[w];
            before += (w < warp) ? n : 0;
            total += n;
        }
        if (kp) a.idx[out + before + __popc(bal & ((1u << lane) - 1u))] = p;
        out += total;
        __syncthreads();  // warp_cnt is rewritten by the next iteration
    }
}

}  // namespace

cudaError_t launch_map(const MapArgs& a, cudaStream_t st)
{
    const int64_t nu = (int64_t)a.L * a.Hkv * a.D;
    if (nu > 0) {
        const int blocks = (int)((nu + 255) / 256 < 4096 ? (nu + 255) / 256 : 4096);
        union_kernel<<<blocks, 256, 0, st>>>(a.M, a.U, a.L, a.H, a.Hkv, a.D);
    }
    dim3 grid(a.NH, a.nchunks);
    count_kernel<<<grid, kMapThreads, 0, st>>>(a);
    scan_kernel<<<1, kScanThreads, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_map_write(const MapArgs& a, cudaStream_t st)
{
    dim3 grid(a.NH, a.nchunks);
    write_kernel<<<grid, kMapThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace dkv
