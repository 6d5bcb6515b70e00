// Pattern -> positions map (Sec. 3.4, Eqs. 4-5 and the GQA union).
//
// keep(p) = p < S  or  p >= Tc - R  or  U[l][g][(Tc - R - 1 - p) / W],  with
// U[l][g][d] = OR_j M[l][g G + j][d]. Between the sink and the recent window the
// decision is constant over the W positions of a distance bin, so a slab's kept
// positions are a few runs of consecutive positions: the sink, each kept bin the
// context reaches (far bins first: token order), the recent window. The map is
// built per bin instead of per position:
//
//   runs_kernel   one warp per slab (layer, sequence, KV head). Lanes take 32
//                 bins at a time in token order: the GQA union of the bin's query
//                 heads, its positions clipped to the context, a warp ballot over
//                 the kept bins and a prefix scan of their lengths, which place
//                 each kept bin's run (first output row, first position) in the
//                 slab's run list and give the slab's length. The last CTA to
//                 finish scans the lengths over the flat slab order into slab
//                 offsets (len + reserve, or h * stride in place), index offsets,
//                 and the totals the host reads (rows, kept rows, longest slab,
//                 kept rows per layer).
//   order_kernel  (in place only) the slabs by length, longest first, ties by
//                 index: slab h goes to its rank among all slabs.
//   write_kernel  one CTA per (slab, kMapChunk output rows): output row r of slab h
//                 is the position runs[i].pos + (r - runs[i].row) of the run i
//                 holding r; lanes take consecutive rows, so the index list is
//                 written with coalesced stores, and no position is visited
//                 twice. Dropped positions are never touched.
#include "dkv_internal.cuh"

namespace dkv {
namespace {

constexpr unsigned kFullMask = 0xffffffffu;
constexpr int kRunsThreads = 256;  // 8 slabs per CTA, one a warp
constexpr int kWriteThreads = 256;

__global__ void __launch_bounds__(kRunsThreads) runs_kernel(const MapArgs a)
{
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.x * (kRunsThreads / 32) + warp;
    if (h < a.NH) {
        const int g = h % a.Hkv;
        const int b = (h / a.Hkv) % a.B;
        const int l = h / (a.Hkv * a.B);
        const int G = a.H / a.Hkv;
        const int Tc = a.Tc[b];
        const int S = a.sink, R = a.recent, W = a.bin_width;
        int2* run = a.runs + (int64_t)h * (a.D + 2);
        int n = 0, out = 0;
        if (Tc <= S + R) {
            // Sink and recent window cover the whole context: one run.
            if (Tc > 0) {
                if (lane == 0) run[0] = make_int2(0, 0);
                n = 1;
            }
            out = Tc;
        } else {
            const int C = Tc - S - R;          // positions between sink and recent window
            const int nb = (int)(((int64_t)C + W - 1) / W);  // bins the context reaches (<= D: checked on the host)
            if (lane == 0) run[0] = make_int2(0, 0);  // the sink
            n = 1;
            out = S;
            const uint8_t* Mg = a.M + ((int64_t)l * a.H + (int64_t)g * G) * a.D;
            for (int k0 = 0; k0 < nb; k0 += 32) {
                const int k = k0 + lane;  // k-th bin in token order: d = nb - 1 - k
                bool on = false;
                int len = 0, lo = 0;
                if (k < nb) {
                    const int d = nb - 1 - k;
                    uint8_t u = 0;
                    for (int j = 0; j < G; ++j) u |= __ldg(Mg + (int64_t)j * a.D + d);
                    on = u != 0;
                    len = min(W, C - d * W);                  // positions of bin d inside the context
                    lo = (int)max((int64_t)S, (int64_t)Tc - R - (int64_t)(d + 1) * W);  // its first position
                }
                const unsigned kept = __ballot_sync(kFullMask, on);
                int incl = on ? len : 0;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int v = __shfl_up_sync(kFullMask, incl, o);
                    if (lane >= o) incl += v;
                }
                if (on) {
                    const int rank = __popc(kept & ((1u << lane) - 1u));
                    run[n + rank] = make_int2(out + incl - len, lo);
                }
                n += __popc(kept);
                out += __shfl_sync(kFullMask, incl, 31);
            }
            if (lane == 0) run[n] = make_int2(out, Tc - R);  // the recent window
            n += 1;
            out += R;
        }
        if (lane == 0) {
            a.len[h] = out;
            a.nruns[h] = n;
        }
    }

    // The last CTA to finish scans the slab lengths.
    __shared__ bool last;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        last = atomicAdd(a.done, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    constexpr int T = kRunsThreads;
    const int per = (a.NH + T - 1) / T;
    const int h0 = min(a.NH, (int)threadIdx.x * per), h1 = min(a.NH, h0 + per);
    int64_t s_off = 0, s_ioff = 0;
    int mx = 0;
    for (int h = h0; h < h1; ++h) {
        const int n = __ldcg(a.len + h);
        s_off += (int64_t)n + a.reserve;
        s_ioff += n;
        mx = max(mx, n);
    }
    __shared__ int64_t sh_off[T], sh_ioff[T];
    __shared__ int sh_max[T];
    sh_off[threadIdx.x] = s_off;
    sh_ioff[threadIdx.x] = s_ioff;
    sh_max[threadIdx.x] = mx;
    __syncthreads();
    // Hillis-Steele inclusive scan over the per-thread sums (and a max).
    for (int d = 1; d < T; d <<= 1) {
        int64_t vo = 0, vi = 0;
        int vm = 0;
        if ((int)threadIdx.x >= d) {
            vo = sh_off[threadIdx.x - d];
            vi = sh_ioff[threadIdx.x - d];
            vm = sh_max[threadIdx.x - d];
        }
        __syncthreads();
        sh_off[threadIdx.x] += vo;
        sh_ioff[threadIdx.x] += vi;
        sh_max[threadIdx.x] = max(sh_max[threadIdx.x], vm);
        __syncthreads();
    }
    int64_t run_off = sh_off[threadIdx.x] - s_off;
    int64_t run_ioff = sh_ioff[threadIdx.x] - s_ioff;
    for (int h = h0; h < h1; ++h) {
        const int n = __ldcg(a.len + h);
        a.off[h] = a.stride > 0 ? (int64_t)h * a.stride : run_off;  // in place: the slab's own dense rows
        a.ioff[h] = run_ioff;
        run_off += (int64_t)n + a.reserve;
        run_ioff += n;
    }
    if (threadIdx.x == T - 1) {
        const int64_t total = a.stride > 0 ? (int64_t)a.NH * a.stride : sh_off[T - 1];
        a.off[a.NH] = total;
        a.ioff[a.NH] = sh_ioff[T - 1];
        a.tail[0] = total;
        a.tail[1] = sh_ioff[T - 1];
        a.tail[2] = sh_max[T - 1];
    }
    __syncthreads();  // every ioff is written (this CTA's own global writes)
    // Kept rows of each layer: NHl = B * Hkv slabs per layer.
    const int NHl = a.B * a.Hkv;
    for (int l = threadIdx.x; l < a.L; l += T) a.tail[3 + l] = a.ioff[(l + 1) * NHl] - a.ioff[l * NHl];
}

// In-place plans: order[rank(h)] = h, rank = slabs longer than h, or as long
// with a lower index (a stable sort by length, longest first).
__global__ void __launch_bounds__(256) order_kernel(const int32_t* __restrict__ len, int NH, int32_t* order)
{
    __shared__ int tile[1024];
    const int h = blockIdx.x * blockDim.x + threadIdx.x;
    const int mine = h < NH ? len[h] : 0;
    int rank = 0;
    for (int t0 = 0; t0 < NH; t0 += 1024) {
        const int n = min(1024, NH - t0);
        __syncthreads();
        for (int i = threadIdx.x; i < n; i += blockDim.x) tile[i] = len[t0 + i];
        __syncthreads();
        if (h < NH)
            for (int i = 0; i < n; ++i) {
                const int x = tile[i];
                rank += (x > mine || (x == mine && t0 + i < h)) ? 1 : 0;
            }
    }
    if (h < NH) order[rank] = h;
}

// A slab's runs are staged in shared memory when they fit (D + 2 <= 2048 covers
// every pattern of the benchmark workloads); otherwise they are read from L2.
constexpr int kRunsSmem = 2048;

__global__ void __launch_bounds__(kWriteThreads) write_kernel(const MapArgs a)
{
    __shared__ int2 srun[kRunsSmem];
    const int h = blockIdx.x;
    const int n_h = __ldg(a.len + h);
    const int r0 = blockIdx.y * kMapChunk;
    if (r0 >= n_h) return;  // uniform over the CTA
    const int nr = __ldg(a.nruns + h);
    const int2* grun = a.runs + (int64_t)h * (a.D + 2);
    const bool staged = nr <= kRunsSmem;
    if (staged)
        for (int i = threadIdx.x; i < nr; i += kWriteThreads) srun[i] = __ldg(grun + i);
    __syncthreads();
    const int2* run = staged ? srun : grun;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // Bounds-checked build: the slab's indices lie inside the list, and every
    // position inside its sequence's context (checked per row below).
    const int Tcb = __ldg(a.Tc + (h / a.Hkv) % a.B);
    if (!in_bounds(__ldg(a.ioff + h) + n_h <= __ldg(a.ioff + a.NH), a.status)) return;  // uniform
    int32_t* dst = a.idx + __ldg(a.ioff + h);
    // Lane rows: base + 32 k, k < 32 (the warp covers 1024 consecutive rows).
    const int base = r0 + warp * (kMapChunk / (kWriteThreads / 32)) + lane;
    if (base >= n_h) return;
    // Run holding `base`: the last run whose first row is <= base.
    int lo = 0, hi = nr - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (run[mid].x <= base)
            lo = mid;
        else
            hi = mid - 1;
    }
    int i = lo;
    int2 cur = run[i];
    int next = i + 1 < nr ? run[i + 1].x : n_h;
#pragma unroll 4
    for (int k = 0; k < 32; ++k) {
        const int r = base + 32 * k;
        if (r >= n_h) break;
        while (r >= next) {
            ++i;
            cur = run[i];
            next = i + 1 < nr ? run[i + 1].x : n_h;
        }
        const int pos = cur.y + (r - cur.x);
        if (in_bounds(pos >= 0 && pos < Tcb, a.status)) dst[r] = pos;
    }
}

}  // namespace

cudaError_t launch_map(const MapArgs& a, cudaStream_t st)
{
    if (a.NH < 1) return cudaErrorInvalidValue;
    const int grid = (a.NH + kRunsThreads / 32 - 1) / (kRunsThreads / 32);
    runs_kernel<<<grid, kRunsThreads, 0, st>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !a.order) return e;
    order_kernel<<<(a.NH + 255) / 256, 256, 0, st>>>(a.len, a.NH, a.order);
    return cudaGetLastError();
}

cudaError_t launch_map_write(const MapArgs& a, int max_len, cudaStream_t st)
{
    if (max_len < 1) return cudaSuccess;  // no kept rows: nothing to write
    dim3 grid(a.NH, (max_len + kMapChunk - 1) / kMapChunk);
    write_kernel<<<grid, kWriteThreads, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace dkv
