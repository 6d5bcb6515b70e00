// Pieces shared by the decode kernels (split-K over the packed cache, Sec. 3.4):
// programmatic-dependent-launch wrappers (the mbarrier and bulk-copy ones are in
// dkv_ptx.cuh), the per-call slab table, the stream-K row partition over the slabs of one layer, the tile cursor of a
// warp, and the end of a CTA's pass: merging the warp states that share a slab
// and the fused cross-CTA merge (the last CTA to finish a (slab, head) merges
// every CTA's partial of it).
#pragma once

#include "dkv_internal.cuh"
#include "dkv_ptx.cuh"

#include <math.h>

namespace dkv {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kMaxB = 512;
constexpr float kSlack = 8.f;        // lazy-rescale threshold of the online softmax (log2 units)
constexpr int PRE = 1;               // tiles a warp fetches before waiting for the previous kernel

// Programmatic dependent launch: let the next kernel in the stream start its
// prologue, and wait for the previous kernel's results before reading them.
__device__ __forceinline__ void pdl_launch_dependents()
{
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void pdl_wait()
{
    asm volatile("griddepcontrol.wait;" ::: "memory");
}

// ------------------------------------------------------------ partition
// Per-call sequence table in shared memory: NA[b] = rows already appended
// (clamped to the reserve), NP[b] = exclusive prefix over b of the extra rows
// e_b = NA[b] + (this call appends to b ? 1 : 0). Layer rows fit in int32.
//
// When the layer has fewer than kSlabCache slabs, the table also holds the
// slabs' row prefix IO[h] = ioff[h] - ioff[0] ([NHl+1]) and cache offsets
// OFF[h] = off[h] ([NHl]), so that finding a warp's rows and streaming them
// reads no plan metadata from global memory: a CTA that starts after the
// previous kernel has drained (the last ones to get an SM) would otherwise pay
// a chain of dependent L2 round trips, under full HBM load, before its first
// copy. IO and OFF are null for larger layers (read from global memory then).
constexpr int kSlabCache = 1024;
struct SeqTable {
    int32_t* NA;   // [B]
    int32_t* NP;   // [B+1]
    int32_t* IO;   // [NHl+1] or null
    int64_t* OFF;  // [NHl] or null
};

// Bytes of the table at an 8-byte aligned base: OFF, IO, NA, NP.
__host__ __device__ constexpr int seq_table_bytes(int B) { return kSlabCache * 8 + kSlabCache * 4 + (2 * B + 1) * 4; }

__device__ __forceinline__ SeqTable seq_table_at(unsigned char* base, const DecodeArgs& a)
{
    SeqTable t;
    const bool cached = a.B * a.Hkv < kSlabCache;
    t.OFF = cached ? reinterpret_cast<int64_t*>(base) : nullptr;
    t.IO = cached ? reinterpret_cast<int32_t*>(base + kSlabCache * 8) : nullptr;
    t.NA = reinterpret_cast<int32_t*>(base + kSlabCache * 12);
    t.NP = t.NA + a.B;
    return t;
}

// Fill IO and OFF (when cached) with the threads [t0, t0 + nt) of the CTA; the
// caller's barrier publishes them.
__device__ __forceinline__ void load_slab_cache(const DecodeArgs& a, SeqTable t, int t0, int nt)
{
    if (!t.IO) return;
    const int NHl = a.B * a.Hkv;
    const int64_t i0 = __ldg(a.ioff);
    for (int h = (int)threadIdx.x - t0; h <= NHl; h += nt) {
        t.IO[h] = (int)(__ldg(a.ioff + h) - i0);
        if (h < NHl) t.OFF[h] = __ldg(a.off + h);
    }
}

__device__ void build_seq_table(const DecodeArgs& a, SeqTable t, bool report)
{
    // Called by one full warp.
    const int lane = threadIdx.x & 31;
    int carry = 0;
    for (int b0 = 0; b0 < a.B; b0 += 32) {
        const int b = b0 + lane;
        int na = 0, e = 0;
        if (b < a.B) {
            const int raw = a.n_app ? a.n_app[b] : 0;
            na = min(max(raw, 0), a.reserve);
            const bool app = a.append && raw >= 0 && raw < a.reserve;
            if (a.append && !app && report) atomicOr(a.status, 0x1 /* DKV_DEV_APPEND_OVERFLOW */);
            e = na + (app ? 1 : 0);
            t.NA[b] = na;
        }
        int incl = e;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += v;
        }
        if (b < a.B) t.NP[b] = carry + incl - e;
        carry += __shfl_sync(kFull, incl, 31);
    }
    if (lane == 0) t.NP[a.B] = carry;
}

// First layer row of slab h (h in [0, B*Hkv]) within this call.
__device__ __forceinline__ int slab_start(const DecodeArgs& a, const SeqTable& t, int h)
{
    const int b = h / a.Hkv, g = h - b * a.Hkv;
    int p = (t.IO ? t.IO[h] : (int)(a.ioff[h] - a.ioff[0])) + a.Hkv * t.NP[b];
    if (g) p += g * (t.NP[b + 1] - t.NP[b]);
    return p;
}

__device__ __forceinline__ int part_start(int w, int R, int P)
{
    // floor(w R / P) without a 64-bit division: R = q P + r, so w R / P = w q + w r / P,
    // and w r < P^2 fits 32 bits (P is a CTA count).
    const unsigned q = (unsigned)R / (unsigned)P, r = (unsigned)R - q * (unsigned)P;
    return (int)((unsigned)w * q + ((unsigned)w * r) / (unsigned)P);
}

// Largest part w with part_start(w) <= x, for 0 <= x < R. part_start(w) <= x
// exactly when w R < (x + 1) P, so w = floor(((x + 1) P - 1) / R): a float
// estimate of that quotient, then exact integer steps (a chain of integer
// divisions here would put ~0.5 us on the end of every launch).
__device__ __forceinline__ int part_of(int x, int R, int P)
{
    const int64_t num = (int64_t)(x + 1) * P - 1;
    int w = (int)((float)num * __fdividef(1.f, (float)R));
    while ((int64_t)(w + 1) * R <= num) ++w;
    while (w > 0 && (int64_t)w * R > num) --w;
    return min(w, P - 1);
}

// Last slab h in [0, NHl) with slab_start(h) <= x.
__device__ int slab_containing(const DecodeArgs& a, const SeqTable& t, int NHl, int x)
{
    int lo = 0, hi = NHl - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (slab_start(a, t, mid) <= x)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

// ------------------------------------------------------------ softmax helpers
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Tile cursor of one warp over its row range, with the current slab's constants.
struct Cursor {
    int h;         // slab; == hend when exhausted
    int s0, s1;    // the warp's rows of this slab, [s0, s1) (layer rows)
    int p0;        // slab_start(h)
    int x;         // first row of the current tile
    int n_h;       // rows of the slab in this call
    int app;       // this call appends the slab's last row from k_new/v_new
    int64_t base;  // off[h]: cache row of the slab's first row
};

__device__ __forceinline__ void cursor_seek(Cursor& cu, const DecodeArgs& a, const SeqTable& t, int hend, int wA,
                                            int wB)
{
    while (cu.h < hend) {
        cu.p0 = slab_start(a, t, cu.h);
        const int p1 = slab_start(a, t, cu.h + 1);
        cu.s0 = max(wA, cu.p0);
        cu.s1 = min(wB, p1);
        if (cu.s0 < cu.s1) {
            const int b = cu.h / a.Hkv;
            const int e = t.NP[b + 1] - t.NP[b];
            cu.n_h = (t.IO ? t.IO[cu.h + 1] - t.IO[cu.h] : a.len[cu.h]) + e;
            cu.app = (a.append && e > t.NA[b]) ? 1 : 0;
            cu.base = t.OFF ? t.OFF[cu.h] : a.off[cu.h];
            cu.x = cu.s0;
            return;
        }
        ++cu.h;
    }
}

template <int TR>
__device__ __forceinline__ void cursor_next(Cursor& cu, const DecodeArgs& a, const SeqTable& t, int hend, int wA,
                                            int wB)
{
    cu.x += TR;
    if (cu.x < cu.s1) return;
    ++cu.h;
    cursor_seek(cu, a, t, hend, wA, wB);
}

// Number of CTAs whose row range overlaps [p0, p1) (p0 < p1), and the first and
// last of them.
__device__ __forceinline__ int ctas_of_slab(int p0, int p1, int R, int P, int* c0_out, int* c1_out)
{
    const int c0 = part_of(p0, R, P), c1 = part_of(p1 - 1, R, P);
    int n = c1 - c0 + 1;
    if (R < P) {  // some CTAs have no rows (never when every CTA gets at least one)
        n = 0;
        for (int cc = c0; cc <= c1; ++cc) n += part_start(cc, R, P) < part_start(cc + 1, R, P) ? 1 : 0;
    }
    *c0_out = c0;
    *c1_out = c1;
    return n;
}

// Output row of column c of slab (b, g): query c / G, head g G + c % G of out [B][Q][H][128].
template <int G>
__device__ __forceinline__ int64_t out_row(const DecodeArgs& a, int b, int g, int c)
{
    const int qi = c / G, j = c - qi * G;
    return ((int64_t)b * a.Q + qi) * a.H + g * G + j;
}

// out row of column c = O / L; O, L of the column for the lane's 4 dims.
template <int G>
__device__ __forceinline__ void write_out(const DecodeArgs& a, int b, int g, int c, float4 O, float L, int lane)
{
    const float inv = L > 0.f ? 1.f / L : 0.f;
    float4* dst = reinterpret_cast<float4*>(a.out + out_row<G>(a, b, g, c) * kHeadDim);
    dst[lane] = make_float4(O.x * inv, O.y * inv, O.z * inv, O.w * inv);
}

// Fused combine of head j of slab h by one warp of the last CTA to finish the
// slab: the CTA partials in slots c + h, c in [c0, c1], which come from other
// SMs (L2 loads). Every lane loads the (m, l) and its 4 dims of o of KB partials
// at once, then merges them in registers; batches chain online. Measured: a
// load round at the end of a launch takes ~1.5 us and grows with the bytes in
// flight, so one round of 20-24 partials costs more than two smaller ones; of
// 8, 10, 12, 16, 20 and 24, KB = 12 was fastest.
template <int G, int KB, int NCC>
__device__ void merge_slab_head(const DecodeArgs& a, int h, int j, int c0, int c1, int R, int lane)
{
    const int b = h / a.Hkv, g = h - b * a.Hkv;
    const int P = a.nctas;
    const bool all_live = R >= P;
    float M = -INFINITY, L = 0.f;
    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int k0 = c0; k0 <= c1; k0 += KB) {
        float2 ml[KB];
        float4 v[KB];
#pragma unroll
        for (int u = 0; u < KB; ++u) {
            const int cc = k0 + u;
            const bool ok = cc <= c1 && (all_live || part_start(cc, R, P) < part_start(cc + 1, R, P));
            const int64_t sj = ((int64_t)cc + h) * (NCC ? NCC : a.NC) + j;
            ml[u] = ok ? __ldcg(reinterpret_cast<const float2*>(a.work_ml + sj * 2)) : make_float2(-INFINITY, 0.f);
            v[u] = ok ? __ldcg(reinterpret_cast<const float4*>(a.work_o + sj * kHeadDim) + lane)
                      : make_float4(0.f, 0.f, 0.f, 0.f);
        }
        float Mb = M;
#pragma unroll
        for (int u = 0; u < KB; ++u) Mb = fmaxf(Mb, ml[u].x);
        const float fo = (M == -INFINITY) ? 0.f : ex2(M - Mb);
        L *= fo;
        O.x *= fo;
        O.y *= fo;
        O.z *= fo;
        O.w *= fo;
#pragma unroll
        for (int u = 0; u < KB; ++u) {
            const float f = (ml[u].x == -INFINITY) ? 0.f : ex2(ml[u].x - Mb);
            L = fmaf(f, ml[u].y, L);
            O.x = fmaf(f, v[u].x, O.x);
            O.y = fmaf(f, v[u].y, O.y);
            O.z = fmaf(f, v[u].z, O.z);
            O.w = fmaf(f, v[u].w, O.w);
        }
        M = Mb;
    }
    write_out<G>(a, b, g, j, O, L, lane);
}

// End of one CTA's split-K pass, after its warps' ranges are done and a CTA
// barrier. NCC: the number of columns per slab when fixed at compile time (the
// decode step: G), 0 to take a.NC. meta: seg_first[NW], seg_last[NW] (first / last slab of warp w, -1 if
// none), then the layer rows [p0, p1) of each entry (2 w: first, 2 w + 1: last)
// as p0[2 NW], p1[2 NW], recorded while streaming so the end of the pass reads
// no plan metadata from global memory;
// the first slab's state is in the warp record (c, w) of warp_o / warp_ml, the
// last slab's in warp w's own ring at ring + w * warp_ring_bytes (o[G][128] then
// (m, l)[G]). The states of each slab are merged; a slab wholly inside this CTA
// is written out (fused), otherwise the CTA writes its partial to slot c + h.
// Fused, the CTA counts itself in for each (slab, head) before merging its
// warps' states; the last CTA to arrive waits until the others have written
// their partials and merges them all. A CTA writes its partial right after it
// arrives, with no wait in between, so the last arriver's wait always ends.
template <int G, int NW, bool FUSED, int NCC>
__device__ void cta_tail(const DecodeArgs& a, const unsigned char* ring, int warp_ring_bytes,
                         const int32_t* meta, int c, int R, int warp, int lane)
{
    const int32_t* seg_first = meta;
    const int32_t* seg_last = meta + NW;
    const int32_t* seg_p0 = meta + 2 * NW;
    const int32_t* seg_p1 = meta + 4 * NW;
    // Entry e (lane e) is the first (even e) or last (odd e) slab of warp e/2, -1 if
    // none; entries list their slabs in non-decreasing order. Task t = (slab #t/G,
    // head t%G) for the distinct slabs; warp w takes tasks w, w+NW, ...
    static_assert(2 * NW <= 32, "one entry per lane");
    const int h_e = (lane < 2 * NW) ? ((lane & 1) ? seg_last[lane >> 1] : seg_first[lane >> 1]) : -1;
    const int p0_e = h_e >= 0 ? seg_p0[lane] : 0, p1_e = h_e >= 0 ? seg_p1[lane] : 0;
    // Slab of the nearest valid entry before this one (-1 if none): one ballot
    // and one shuffle.
    const unsigned valid = __ballot_sync(kFull, h_e >= 0);
    const unsigned below = valid & ((1u << lane) - 1u);
    const int hprev = __shfl_sync(kFull, h_e, below ? 31 - __clz(below) : 0);
    const int prev = below ? hprev : -1;
    const unsigned fresh = __ballot_sync(kFull, h_e >= 0 && h_e != prev);
    const int nslab = __popc(fresh);
    const int NC = NCC ? NCC : a.NC;  // columns (query x head) per slab; NCC: known at compile time
    // Task t = (slab #si, column j), t = si NC + j; warp w takes t = w, w + NW, ...
    // (si, j) advance by additions: no division on this latency-bound path.
    int si = 0, j = warp - NW;
    for (int t = warp; t < nslab * NC; t += NW) {
        j += NW;
        while (j >= NC) {
            j -= NC;
            ++si;
        }
        unsigned m = fresh;
        for (int k = 0; k < si; ++k) m &= m - 1;
        const int e0 = __ffs(m) - 1;
        const int h = __shfl_sync(kFull, h_e, e0);
        const int hp0 = __shfl_sync(kFull, p0_e, e0), hp1 = __shfl_sync(kFull, p1_e, e0);
        const unsigned same = __ballot_sync(kFull, h_e == h);
        int c0h = 0, c1h = 0;
        const int nct = FUSED ? ctas_of_slab(hp0, hp1, R, a.nctas, &c0h, &c1h) : 0;
        // Count this CTA in for (slab, head) now, so that the atomic's round trip
        // overlaps the merge below. Counter pair: arrivals, then partials written.
        int32_t* ctr = FUSED ? a.slab_count + ((int64_t)h * NC + j) * 2 : nullptr;
        int old = 0;
        if (FUSED && nct > 1 && lane == 0)
            asm volatile("atom.relaxed.gpu.global.add.s32 %0, [%1], 1;" : "=r"(old) : "l"(ctr) : "memory");
        float M = -INFINITY;
#pragma unroll
        for (int f = 0; f < 2 * NW; ++f) {
            if (!((same >> f) & 1u)) continue;
            const int w = f >> 1;
            const float* ml = (f & 1) ? reinterpret_cast<const float*>(ring + w * warp_ring_bytes) + NC * kHeadDim
                                      : a.warp_ml + ((int64_t)c * NW + w) * NC * 2;
            M = fmaxf(M, ml[2 * j]);
        }
        float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
        float L = 0.f;
#pragma unroll
        for (int f = 0; f < 2 * NW; ++f) {
            if (!((same >> f) & 1u)) continue;
            const int w = f >> 1;
            const float* ob = (f & 1) ? reinterpret_cast<const float*>(ring + w * warp_ring_bytes)
                                      : a.warp_o + ((int64_t)c * NW + w) * NC * kHeadDim;
            const float* ml = (f & 1) ? ob + NC * kHeadDim : a.warp_ml + ((int64_t)c * NW + w) * NC * 2;
            const float2 mlj = *reinterpret_cast<const float2*>(ml + 2 * j);
            const float fct = (mlj.x == -INFINITY) ? 0.f : ex2(mlj.x - M);
            L = fmaf(mlj.y, fct, L);
            const float4 v = reinterpret_cast<const float4*>(ob + j * kHeadDim)[lane];
            O.x = fmaf(v.x, fct, O.x);
            O.y = fmaf(v.y, fct, O.y);
            O.z = fmaf(v.z, fct, O.z);
            O.w = fmaf(v.w, fct, O.w);
        }
        if (FUSED && nct == 1) {
            write_out<G>(a, h / a.Hkv, h % a.Hkv, j, O, L, lane);  // the slab lies wholly in this CTA
            continue;
        }
        const int64_t slot = (int64_t)c + h;
        reinterpret_cast<float4*>(a.work_o + (slot * NC + j) * kHeadDim)[lane] = O;
        if (lane == 0) *reinterpret_cast<float2*>(a.work_ml + (slot * NC + j) * 2) = make_float2(M, L);
        if (!FUSED) continue;
        __syncwarp();
        if (__shfl_sync(kFull, old, 0) != nct - 1) {
            // Not the last: release the partial just written to the last arriver.
            if (lane == 0) asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(ctr + 1) : "memory");
            continue;
        }
        // The last arriver: acquire the other CTAs' partials once all are written
        // (a bounded wait: every CTA that arrived is resident and writes next),
        // make the counters ready for the next call, and merge.
        int ok = 1;
        if (lane == 0) {
            ok = 0;
            const unsigned long long t0 = global_ns();
            for (int i = 1; i < kWaitSpins; ++i) {
                int n;
                asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(n) : "l"(ctr + 1) : "memory");
                if (n == nct - 1 + a.merge_extra) {
                    ok = 1;
                    break;
                }
                if ((i & 63) == 0 && global_ns() - t0 > kWaitNs) break;
            }
            if (!ok) atomicOr(a.status, 0x4 /* DKV_DEV_MERGE_TIMEOUT */);
            ctr[0] = 0;
            ctr[1] = 0;
        }
        ok = __shfl_sync(kFull, ok, 0);
        __syncwarp();
        if (ok) merge_slab_head<G, 12, NCC>(a, h, j, c0h, c1h, R, lane);
    }
}

// Launch with programmatic stream serialization: the kernel may start while the
// previous kernel in the stream drains, and waits (griddepcontrol.wait) before
// it reads that kernel's results.
template <class K, class... Args>
cudaError_t launch_pdl(K kernel, int grid, int block, int smem, cudaStream_t st, const Args&... args)
{
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(grid);
    lc.blockDim = dim3(block);
    lc.dynamicSmemBytes = smem;
    lc.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, kernel, args...);
}

}  // namespace
}  // namespace dkv
