// Decode-step attention over the packed cache (Sec. 3.4), split-K.
//
// Work split ("stream-K" over rows). For one layer, the rows of all slabs
// h = b*Hkv + g are laid end to end: slab h owns global rows
// [P(h), P(h+1)), n_h = len[h] + appended[b] (+1 for this step's token).
// CTA c of P CTAs takes rows [A(c), A(c+1)), A(c) = floor(c*R/P), so every CTA
// streams the same number of bytes whatever the slab lengths. It writes one
// partial (m, l, o) per slab it touches into slot c + h; the slots are
// distinct because CTA ranges and slabs are both in row order. The combine
// kernel then merges, for each (b, q-head), the partials of the CTAs that
// cover its slab.
//
// Inside a CTA, each warp owns a ring of NS stages and fetches its tiles of
// TR rows (K and V, 256 bytes a row) with cp.async.bulk into shared memory,
// completing on an mbarrier; tiles of a slab segment go round-robin to the
// warps. A half-warp takes one row, a lane 8 dims: q.k is 8 FMAs per lane and
// a 4-step xor-shuffle sum over the half, then an online softmax in base 2
// (q is pre-scaled by scale*log2 e), and o += p v on the lane's 8 dims. At the
// end of each slab segment the warps' states merge in shared memory.
#include "dkv_internal.cuh"

#include <math.h>

namespace dkv {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kMaxB = 1024;
constexpr int kWaitSpins = 1 << 22;  // bound on mbarrier polls (each poll may suspend)

// ------------------------------------------------------------ PTX helpers
__device__ __forceinline__ uint32_t smem_u32(const void* p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: false when the phase did not complete within kWaitSpins polls.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity)
{
    for (int i = 0; i < kWaitSpins; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    return false;
}

__device__ __forceinline__ uint64_t evict_first_policy()
{
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar, uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4& r, float* f)
{
    const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

// ------------------------------------------------------------ partition
// Per-call sequence table in shared memory: NA[b] = rows already appended
// (clamped to the reserve), NP[b] = exclusive prefix over b of the extra rows
// e_b = NA[b] + (this call appends to b ? 1 : 0).
struct SeqTable {
    int32_t* NA;  // [B]
    int32_t* NP;  // [B+1]
};

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

// First global row of slab h (h in [0, B*Hkv]) within this layer call.
__device__ __forceinline__ int64_t slab_start(const DecodeArgs& a, const SeqTable& t, int h)
{
    const int b = h / a.Hkv, g = h - b * a.Hkv;
    int64_t p = (a.ioff[h] - a.ioff[0]) + (int64_t)a.Hkv * t.NP[b];
    if (g) p += (int64_t)g * (t.NP[b + 1] - t.NP[b]);
    return p;
}

__device__ __forceinline__ int64_t cta_start(int c, int64_t R, int P)
{
    return ((int64_t)c * R) / P;
}

// Largest c with cta_start(c) <= x, for 0 <= x < R.
__device__ __forceinline__ int cta_of(int64_t x, int64_t R, int P)
{
    int c = (int)((x * P) / R);
    while (c + 1 < P && cta_start(c + 1, R, P) <= x) ++c;
    while (c > 0 && cta_start(c, R, P) > x) --c;
    return c;
}

// Last slab h in [0, NHl) with slab_start(h) <= x.
__device__ int slab_containing(const DecodeArgs& a, const SeqTable& t, int NHl, int64_t x)
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

// ------------------------------------------------------------ partial kernel
template <int G, int NW, int NS, int TR>
struct DecodeSmem {
    static constexpr int kStageBytes = 2 * TR * kRowBytes;  // K tile then V tile
    static constexpr int kRingBytes = NW * NS * kStageBytes;
    static constexpr int kBarBytes = NW * NS * 8;
    static constexpr int kMergeFloats = NW * G * (kHeadDim + 2);
    static constexpr int kFixedBytes = kRingBytes + kBarBytes + kMergeFloats * 4;
    static int bytes(int B) { return kFixedBytes + (2 * B + 1) * 4; }
};

// Tile cursor of one warp over the CTA's slab segments.
struct Cursor {
    int h;        // slab; == hend when exhausted
    int64_t s0;   // segment global rows [s0, s1)
    int64_t s1;
    int64_t p0;   // slab_start(h)
    int t;        // tile index within the segment
};

template <int TR, int NW>
__device__ __forceinline__ void cursor_seek(Cursor& cu, const DecodeArgs& a, const SeqTable& t,
                                            int hend, int64_t A, int64_t Bc, int warp)
{
    // Advance from cu.h (inclusive) to the first slab whose segment has a tile for `warp`.
    while (cu.h < hend) {
        cu.p0 = slab_start(a, t, cu.h);
        const int64_t p1 = slab_start(a, t, cu.h + 1);
        cu.s0 = max(A, cu.p0);
        cu.s1 = min(Bc, p1);
        cu.t = warp;
        if (cu.s0 + (int64_t)warp * TR < cu.s1) return;
        ++cu.h;
    }
}

template <int TR, int NW>
__device__ __forceinline__ void cursor_next(Cursor& cu, const DecodeArgs& a, const SeqTable& t,
                                            int hend, int64_t A, int64_t Bc, int warp)
{
    cu.t += NW;
    if (cu.s0 + (int64_t)cu.t * TR < cu.s1) return;
    ++cu.h;
    cursor_seek<TR, NW>(cu, a, t, hend, A, Bc, warp);
}

template <int G, int NW, int NS, int TR>
__global__ void __launch_bounds__(NW * 32, 1) decode_partial_kernel(const DecodeArgs a)
{
    using SM = DecodeSmem<G, NW, NS, TR>;
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char* ring = smem;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SM::kRingBytes);
    float* mrg = reinterpret_cast<float*>(smem + SM::kRingBytes + SM::kBarBytes);
    SeqTable tab;
    tab.NA = reinterpret_cast<int32_t*>(smem + SM::kFixedBytes);
    tab.NP = tab.NA + a.B;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int half = lane >> 4, sub = lane & 15;
    const int NHl = a.B * a.Hkv;
    const int c = blockIdx.x;

    if (warp == 0) build_seq_table(a, tab, c == 0);
    if (lane == 0) {
        for (int s = 0; s < NS; ++s) mbar_init(smem_u32(&bars[warp * NS + s]), 1);
        fence_proxy_async_smem();
    }
    __syncthreads();

    const int64_t R = slab_start(a, tab, NHl);
    if (R == 0) return;
    const int64_t A = cta_start(c, R, a.nctas), Bc = cta_start(c + 1, R, a.nctas);
    if (A >= Bc) return;
    const int hfirst = slab_containing(a, tab, NHl, A);
    const int hend = slab_containing(a, tab, NHl, Bc - 1) + 1;

    const uint64_t pol = evict_first_policy();
    unsigned char* my_ring = ring + warp * NS * SM::kStageBytes;
    uint64_t* my_bars = bars + warp * NS;

    // Issue cursor (lane 0 uses it; every lane tracks it identically).
    Cursor ld{hfirst, 0, 0, 0, 0};
    cursor_seek<TR, NW>(ld, a, tab, hend, A, Bc, warp);
    Cursor cp = ld;

    auto issue = [&](const Cursor& cu, int stage) {
        const int64_t x0 = cu.s0 + (int64_t)cu.t * TR;
        const int cnt = (int)min((int64_t)TR, cu.s1 - x0);
        const int r0 = (int)(x0 - cu.p0);  // local row within the slab
        const int b = cu.h / a.Hkv;
        const int n_h = a.len[cu.h] + (tab.NP[b + 1] - tab.NP[b]);
        const bool app = a.append && (tab.NP[b + 1] - tab.NP[b]) > tab.NA[b];
        const int ncopy = (app && r0 + cnt == n_h) ? cnt - 1 : cnt;  // new token comes from k_new
        const uint32_t bar = smem_u32(&my_bars[stage]);
        unsigned char* dst = my_ring + stage * SM::kStageBytes;
        const uint32_t bytes = (uint32_t)ncopy * kRowBytes;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(bar, 2 * bytes);
        if (ncopy > 0) {
            const int64_t row = a.off[cu.h] + r0;
            bulk_g2s(smem_u32(dst), a.Kc + row * kHeadDim, bytes, bar, pol);
            bulk_g2s(smem_u32(dst + TR * kRowBytes), a.Vc + row * kHeadDim, bytes, bar, pol);
        }
    };

    // A bounded wait that runs out marks the warp dead: it stops issuing and
    // computing but keeps walking the segments so the CTA barriers stay matched.
    bool dead = false;
    int inflight = 0;  // tiles issued and not yet consumed
    int dead_stage = 0, dead_inflight = 0;
    uint32_t dead_phase = 0;
    if (lane == 0) {
        Cursor it = ld;
        for (int s = 0; s < NS && it.h < hend; ++s) {
            issue(it, s);
            cursor_next<TR, NW>(it, a, tab, hend, A, Bc, warp);
        }
    }
    for (int s = 0; s < NS && ld.h < hend; ++s) {
        ++inflight;
        cursor_next<TR, NW>(ld, a, tab, hend, A, Bc, warp);
    }
    int stage = 0;
    uint32_t phase = 0;

    for (int h = hfirst; h < hend; ++h) {
        {
            const int64_t p0 = slab_start(a, tab, h), p1 = slab_start(a, tab, h + 1);
            if (max(A, p0) >= min(Bc, p1)) continue;  // empty slab: nothing to merge (uniform)
        }
        const int b = h / a.Hkv, g = h - b * a.Hkv;
        // q rows of this group: lane holds dims [8*sub, 8*sub + 8) of every head j.
        float q[G][8];
#pragma unroll
        for (int j = 0; j < G; ++j) {
            const uint4 r = *reinterpret_cast<const uint4*>(
                a.q + ((int64_t)b * a.H + g * G + j) * kHeadDim + 8 * sub);
            bf16x8_to_f32(r, q[j]);
#pragma unroll
            for (int e = 0; e < 8; ++e) q[j][e] *= a.qscale;
        }
        float m[G], l[G], o[G][8];
#pragma unroll
        for (int j = 0; j < G; ++j) {
            m[j] = -INFINITY;
            l[j] = 0.f;
#pragma unroll
            for (int e = 0; e < 8; ++e) o[j][e] = 0.f;
        }

        while (cp.h == h) {
            const int64_t x0 = cp.s0 + (int64_t)cp.t * TR;
            const int cnt = (int)min((int64_t)TR, cp.s1 - x0);
            const int r0 = (int)(x0 - cp.p0);
            unsigned char* kt = my_ring + stage * SM::kStageBytes;
            unsigned char* vt = kt + TR * kRowBytes;
            if (!dead) {
                // Every lane observes the completed phase itself (acquire) before reading.
                const bool ok = __all_sync(kFull, mbar_wait(smem_u32(&my_bars[stage]), phase));
                if (ok) {
                    --inflight;
                } else {
                    dead = true;
                    dead_stage = stage;
                    dead_phase = phase;
                    dead_inflight = inflight;
                    if (lane == 0) atomicOr(a.status, 0x2 /* DKV_DEV_TMA_TIMEOUT */);
                }
            }
            if (!dead) {
                const int n_h = a.len[h] + (tab.NP[b + 1] - tab.NP[b]);
                const bool app = a.append && (tab.NP[b + 1] - tab.NP[b]) > tab.NA[b];
                if (app && r0 + cnt == n_h) {
                    // This step's token: into the tile from k_new/v_new, and into the
                    // slab's next free row for later steps.
                    const int rr = cnt - 1;
                    const uint16_t* src = (half ? a.v_new : a.k_new) + ((int64_t)b * a.Hkv + g) * kHeadDim;
                    const uint4 v = *(reinterpret_cast<const uint4*>(src) + sub);
                    *reinterpret_cast<uint4*>((half ? vt : kt) + rr * kRowBytes + sub * 16) = v;
                    uint16_t* dstg = (half ? a.Vc : a.Kc) + (a.off[h] + (n_h - 1)) * kHeadDim;
                    *(reinterpret_cast<uint4*>(dstg) + sub) = v;
                    fence_proxy_async_smem();  // order these generic writes before later bulk copies
                    __syncwarp();
                }

                // Pass 1: scores of this tile, s[i][j] for rows 2i + half.
                float s[TR / 2][G];
#pragma unroll
                for (int i = 0; i < TR / 2; ++i) {
                    const int row = 2 * i + half;
                    const bool valid = row < cnt;
                    const uint4 kr = *reinterpret_cast<const uint4*>(kt + row * kRowBytes + sub * 16);
                    float kf[8];
                    bf16x8_to_f32(kr, kf);
#pragma unroll
                    for (int j = 0; j < G; ++j) {
                        float d = 0.f;
#pragma unroll
                        for (int e = 0; e < 8; ++e) d = fmaf(q[j][e], kf[e], d);
                        d += __shfl_xor_sync(kFull, d, 8);
                        d += __shfl_xor_sync(kFull, d, 4);
                        d += __shfl_xor_sync(kFull, d, 2);
                        d += __shfl_xor_sync(kFull, d, 1);
                        s[i][j] = valid ? d : -INFINITY;
                    }
                }
                // Online softmax, per half (each half keeps its own running state).
                float p[TR / 2][G];
#pragma unroll
                for (int j = 0; j < G; ++j) {
                    float tmax = s[0][j];
#pragma unroll
                    for (int i = 1; i < TR / 2; ++i) tmax = fmaxf(tmax, s[i][j]);
                    const float mnew = fmaxf(m[j], tmax);
                    const bool grow = mnew > m[j];
                    if (__any_sync(kFull, grow)) {
                        const float alpha = grow ? exp2f(m[j] - mnew) : 1.f;
                        l[j] *= alpha;
#pragma unroll
                        for (int e = 0; e < 8; ++e) o[j][e] *= alpha;
                    }
                    m[j] = mnew;
                    const float mref = (mnew == -INFINITY) ? 0.f : mnew;
                    float ls = 0.f;
#pragma unroll
                    for (int i = 0; i < TR / 2; ++i) {
                        p[i][j] = exp2f(s[i][j] - mref);
                        ls += p[i][j];
                    }
                    l[j] += ls;
                }
                // Pass 2: o += p v.
#pragma unroll
                for (int i = 0; i < TR / 2; ++i) {
                    const int row = 2 * i + half;
                    float vf[8];
                    if (row < cnt) {
                        const uint4 vr = *reinterpret_cast<const uint4*>(vt + row * kRowBytes + sub * 16);
                        bf16x8_to_f32(vr, vf);
                    } else {
#pragma unroll
                        for (int e = 0; e < 8; ++e) vf[e] = 0.f;
                    }
#pragma unroll
                    for (int j = 0; j < G; ++j)
#pragma unroll
                        for (int e = 0; e < 8; ++e) o[j][e] = fmaf(p[i][j], vf[e], o[j][e]);
                }
            }
            __syncwarp();
            // Refill this stage with the tile NS ahead.
            if (!dead && ld.h < hend) {
                if (lane == 0) issue(ld, stage);
                ++inflight;
                cursor_next<TR, NW>(ld, a, tab, hend, A, Bc, warp);
            }
            cursor_next<TR, NW>(cp, a, tab, hend, A, Bc, warp);
            if (++stage == NS) {
                stage = 0;
                phase ^= 1u;
            }
        }

        // Merge the two halves of the warp (same dims, different rows).
#pragma unroll
        for (int j = 0; j < G; ++j) {
            const float mo = __shfl_xor_sync(kFull, m[j], 16);
            const float lo = __shfl_xor_sync(kFull, l[j], 16);
            const float mm = fmaxf(m[j], mo);
            const float fa = (m[j] == -INFINITY) ? 0.f : exp2f(m[j] - mm);
            const float fb = (mo == -INFINITY) ? 0.f : exp2f(mo - mm);
            l[j] = l[j] * fa + lo * fb;
#pragma unroll
            for (int e = 0; e < 8; ++e) {
                const float oo = __shfl_xor_sync(kFull, o[j][e], 16);
                o[j][e] = o[j][e] * fa + oo * fb;
            }
            m[j] = mm;
        }
        float* mw = mrg + warp * G * (kHeadDim + 2);
        if (half == 0) {
#pragma unroll
            for (int j = 0; j < G; ++j) {
#pragma unroll
                for (int e = 0; e < 8; ++e) mw[j * (kHeadDim + 2) + 8 * sub + e] = o[j][e];
                if (sub == 0) {
                    mw[j * (kHeadDim + 2) + kHeadDim] = m[j];
                    mw[j * (kHeadDim + 2) + kHeadDim + 1] = l[j];
                }
            }
        }
        __syncthreads();
        // Merge the NW warp states into the CTA's partial for slab h.
        const int64_t slot = (int64_t)c + h;
        for (int i = threadIdx.x; i < G * kHeadDim; i += NW * 32) {
            const int j = i / kHeadDim, d = i - j * kHeadDim;
            float M = -INFINITY;
            for (int w = 0; w < NW; ++w) M = fmaxf(M, mrg[(w * G + j) * (kHeadDim + 2) + kHeadDim]);
            float O = 0.f, Lsum = 0.f;
            for (int w = 0; w < NW; ++w) {
                const float* st = mrg + (w * G + j) * (kHeadDim + 2);
                const float f = (st[kHeadDim] == -INFINITY) ? 0.f : exp2f(st[kHeadDim] - M);
                O = fmaf(st[d], f, O);
                Lsum = fmaf(st[kHeadDim + 1], f, Lsum);
            }
            a.work_o[(slot * G + j) * kHeadDim + d] = O;
            if (d == 0) {
                a.work_ml[(slot * G + j) * 2] = M;
                a.work_ml[(slot * G + j) * 2 + 1] = Lsum;
            }
        }
        __syncthreads();  // mrg is rewritten by the next segment
    }

    // After a timeout, wait (with the same bound) for the copies this warp still has in flight.
    if (dead && lane == 0) {
        for (int k = 0; k < dead_inflight; ++k) {
            mbar_wait(smem_u32(&my_bars[dead_stage]), dead_phase);
            if (++dead_stage == NS) {
                dead_stage = 0;
                dead_phase ^= 1u;
            }
        }
    }
}

// ------------------------------------------------------------ combine kernel
constexpr int kCombineWarps = 8;

__global__ void __launch_bounds__(kCombineWarps * 32) decode_combine_kernel(const DecodeArgs a)
{
    extern __shared__ int32_t csmem[];
    SeqTable tab{csmem, csmem + a.B};
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) build_seq_table(a, tab, false);
    __syncthreads();

    const int pair = blockIdx.x * kCombineWarps + warp;  // (b, q-head)
    if (pair >= a.B * a.H) return;
    const int b = pair / a.H, hq = pair - b * a.H;
    const int g = hq / a.G, j = hq - g * a.G;
    const int h = b * a.Hkv + g;
    const int NHl = a.B * a.Hkv;
    const int64_t R = slab_start(a, tab, NHl);
    const int64_t p0 = slab_start(a, tab, h), p1 = slab_start(a, tab, h + 1);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (p1 > p0) {
        const int c0 = cta_of(p0, R, a.nctas), c1 = cta_of(p1 - 1, R, a.nctas);
        float M = -INFINITY;
        for (int c = c0; c <= c1; ++c) {
            if (cta_start(c, R, a.nctas) == cta_start(c + 1, R, a.nctas)) continue;
            M = fmaxf(M, a.work_ml[(((int64_t)c + h) * a.G + j) * 2]);
        }
        float Lsum = 0.f;
        for (int c = c0; c <= c1; ++c) {
            if (cta_start(c, R, a.nctas) == cta_start(c + 1, R, a.nctas)) continue;
            const int64_t sj = ((int64_t)c + h) * a.G + j;
            const float mc = a.work_ml[sj * 2], lc = a.work_ml[sj * 2 + 1];
            const float f = (mc == -INFINITY) ? 0.f : exp2f(mc - M);
            Lsum = fmaf(lc, f, Lsum);
            const float4 v = *reinterpret_cast<const float4*>(a.work_o + sj * kHeadDim + 4 * lane);
            acc.x = fmaf(v.x, f, acc.x);
            acc.y = fmaf(v.y, f, acc.y);
            acc.z = fmaf(v.z, f, acc.z);
            acc.w = fmaf(v.w, f, acc.w);
        }
        const float inv = Lsum > 0.f ? 1.f / Lsum : 0.f;
        acc.x *= inv;
        acc.y *= inv;
        acc.z *= inv;
        acc.w *= inv;
    }
    *reinterpret_cast<float4*>(a.out + ((int64_t)b * a.H + hq) * kHeadDim + 4 * lane) = acc;
}

__global__ void advance_kernel(int32_t* n_app, int B, int reserve, int32_t* status)
{
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    if (n_app[b] < reserve)
        n_app[b] += 1;
    else
        atomicOr(status, 0x1 /* DKV_DEV_APPEND_OVERFLOW */);
}

// ------------------------------------------------------------ launch table
constexpr int kNW = 8;
constexpr int kNS = 4;
constexpr int kTR = 8;

template <int G>
cudaError_t launch_partial_g(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    decode_partial_kernel<G, kNW, kNS, kTR><<<cfg.nctas, kNW * 32, cfg.smem_bytes, st>>>(a);
    return cudaGetLastError();
}

template <int G>
cudaError_t config_g(int B, DecodeConfig* cfg)
{
    using SM = DecodeSmem<G, kNW, kNS, kTR>;
    const int smem = SM::bytes(B);
    cudaError_t e = cudaFuncSetAttribute(decode_partial_kernel<G, kNW, kNS, kTR>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
        return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(
             &per_sm, decode_partial_kernel<G, kNW, kNS, kTR>, kNW * 32, smem)) != cudaSuccess)
        return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    cfg->nctas = sms * per_sm;
    cfg->smem_bytes = smem;
    return cudaSuccess;
}

}  // namespace

cudaError_t decode_config(int G, int B, DecodeConfig* cfg)
{
    if (B < 1 || B > kMaxB) return cudaErrorInvalidValue;
    switch (G) {
        case 1: return config_g<1>(B, cfg);
        case 2: return config_g<2>(B, cfg);
        case 3: return config_g<3>(B, cfg);
        case 4: return config_g<4>(B, cfg);
        case 5: return config_g<5>(B, cfg);
        case 6: return config_g<6>(B, cfg);
        case 7: return config_g<7>(B, cfg);
        case 8: return config_g<8>(B, cfg);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_decode_partial(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    switch (a.G) {
        case 1: return launch_partial_g<1>(a, cfg, st);
        case 2: return launch_partial_g<2>(a, cfg, st);
        case 3: return launch_partial_g<3>(a, cfg, st);
        case 4: return launch_partial_g<4>(a, cfg, st);
        case 5: return launch_partial_g<5>(a, cfg, st);
        case 6: return launch_partial_g<6>(a, cfg, st);
        case 7: return launch_partial_g<7>(a, cfg, st);
        case 8: return launch_partial_g<8>(a, cfg, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_decode_combine(const DecodeArgs& a, cudaStream_t st)
{
    const int pairs = a.B * a.H;
    decode_combine_kernel<<<(pairs + kCombineWarps - 1) / kCombineWarps, kCombineWarps * 32,
                            (2 * a.B + 1) * 4, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_advance(int32_t* n_app, int B, int reserve, int32_t* status, cudaStream_t st)
{
    advance_kernel<<<(B + 127) / 128, 128, 0, st>>>(n_app, B, reserve, status);
    return cudaGetLastError();
}

}  // namespace dkv
