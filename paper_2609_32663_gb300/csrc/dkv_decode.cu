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

#include <type_traits>

namespace dkv {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kMaxB = 512;
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
__device__ __forceinline__ float ex2(float x)
{
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Packed pair of fp32 values (one 64-bit register pair) for fma.rn.f32x2.
__device__ __forceinline__ uint64_t pk(float lo, float hi)
{
    uint64_t d;
    asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(lo), "f"(hi));
    return d;
}

__device__ __forceinline__ float2 upk(uint64_t v)
{
    float2 r;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(r.x), "=f"(r.y) : "l"(v));
    return r;
}

__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c)
{
    uint64_t d;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
    return d;
}

__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b)
{
    uint64_t d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b)
{
    uint64_t d;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}

// bf16 pair (low element = lower dim) -> packed fp32 pair; exact.
__device__ __forceinline__ uint64_t bf2_to_f2(uint32_t w)
{
    return pk(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}

// Compile-time geometry of the partial kernel.
//   LPR lanes share one row (each owns DPL = 128/LPR dims, i.e. NCH 16-byte
//   chunks c = s + LPR*i of the row); a warp step covers RPS = 32/LPR rows; a
//   tile of TR rows takes STEPS steps. Scores: TR*G per tile, NSUM per lane.
template <int G_, int LPR_, int TR_, int NS_, int NW_>
struct PK {
    static constexpr int G = G_, LPR = LPR_, TR = TR_, NS = NS_, NW = NW_;
    static constexpr int RPS = 32 / LPR;
    static constexpr int DPL = kHeadDim / LPR;
    static constexpr int NCH = DPL / 8;
    static constexpr int STEPS = TR / RPS;
    static constexpr int NSUM = (TR * G + 31) / 32;
    static constexpr int GP = G <= 4 ? 4 : 8;  // p row stride (floats)
    // Reduction buffer red[j][r][step][s]: RS is the r stride, = LPR (mod 32), so
    // the 32 lanes of one store (fixed j, step) hit 32 distinct banks.
    static constexpr int RS0 = STEPS * LPR;
    static constexpr int RS = RS0 + ((LPR - RS0 % 32) + 32) % 32;
    static constexpr int JS = RPS * RS;
    static constexpr int kRedFloats = G * JS;
    static constexpr int kPFloats = TR * GP;
    static constexpr int kWarpScratch = (kRedFloats + kPFloats) * 4;
    static constexpr int kStageBytes = 2 * TR * kRowBytes;  // K tile then V tile
    static constexpr int kRingBytes = NW * NS * kStageBytes;
    static constexpr int kMergeBytes = NW * G * (kHeadDim + 2) * 4;
    static constexpr int kScratchBytes = (NW * kWarpScratch > kMergeBytes) ? NW * kWarpScratch : kMergeBytes;
    static constexpr int kBarBytes = NW * NS * 8;
    static constexpr int kFixedBytes = kRingBytes + kScratchBytes + kBarBytes;
    static int bytes(int B) { return kFixedBytes + (2 * B + 1) * 4; }
    static_assert(TR % RPS == 0 && 32 % TR == 0, "tile geometry");
    static_assert(RS % 4 == 0, "16-byte aligned reduction rows");
};

// Tile cursor of one warp over the CTA's slab segments, with the segment's
// constants cached (slab start row in the cache, rows, append flag).
struct Cursor {
    int h;        // slab; == hend when exhausted
    int64_t s0;   // segment global rows [s0, s1)
    int64_t s1;
    int64_t p0;   // slab_start(h)
    int64_t base; // off[h]: first cache row of the slab
    int n_h;      // rows of the slab in this call
    int app;      // this call appends the slab's last row from k_new/v_new
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
        if (cu.s0 + (int64_t)warp * TR < cu.s1) {
            const int b = cu.h / a.Hkv;
            const int e = t.NP[b + 1] - t.NP[b];
            cu.n_h = a.len[cu.h] + e;
            cu.app = (a.append && e > t.NA[b]) ? 1 : 0;
            cu.base = a.off[cu.h];
            return;
        }
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

template <class C>
__global__ void __launch_bounds__(C::NW * 32, 1) decode_partial_kernel(const DecodeArgs a)
{
    constexpr int G = C::G, LPR = C::LPR, TR = C::TR, NS = C::NS, NW = C::NW;
    constexpr int RPS = C::RPS, DPL = C::DPL, NCH = C::NCH, STEPS = C::STEPS, NSUM = C::NSUM;
    extern __shared__ __align__(128) unsigned char smem[];
    unsigned char* ring = smem;
    unsigned char* scratch = smem + C::kRingBytes;
    uint64_t* bars = reinterpret_cast<uint64_t*>(scratch + C::kScratchBytes);
    SeqTable tab;
    tab.NA = reinterpret_cast<int32_t*>(smem + C::kFixedBytes);
    tab.NP = tab.NA + a.B;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int r = lane / LPR, sl = lane % LPR;  // row within a step, dim slice
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
    unsigned char* my_ring = ring + warp * NS * C::kStageBytes;
    uint64_t* my_bars = bars + warp * NS;
    float* red = reinterpret_cast<float*>(scratch + warp * C::kWarpScratch);
    float* ps = red + C::kRedFloats;
    float* mrg = reinterpret_cast<float*>(scratch);

    Cursor ld{hfirst, 0, 0, 0, 0, 0, 0, 0};
    cursor_seek<TR, NW>(ld, a, tab, hend, A, Bc, warp);
    Cursor cp = ld;

    auto issue = [&](const Cursor& cu, int stage) {
        const int64_t x0 = cu.s0 + (int64_t)cu.t * TR;
        const int cnt = (int)min((int64_t)TR, cu.s1 - x0);
        const int r0 = (int)(x0 - cu.p0);
        const int ncopy = (cu.app && r0 + cnt == cu.n_h) ? cnt - 1 : cnt;  // new token comes from k_new
        const uint32_t bar = smem_u32(&my_bars[stage]);
        unsigned char* dst = my_ring + stage * C::kStageBytes;
        const uint32_t bytes = (uint32_t)ncopy * kRowBytes;
        fence_proxy_async_smem();
        mbar_arrive_expect_tx(bar, 2 * bytes);
        if (ncopy > 0) {
            const int64_t row = cu.base + r0;
            bulk_g2s(smem_u32(dst), a.Kc + row * kHeadDim, bytes, bar, pol);
            bulk_g2s(smem_u32(dst + TR * kRowBytes), a.Vc + row * kHeadDim, bytes, bar, pol);
        }
    };

    bool dead = false;
    int inflight = 0;
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
    const float cs = a.qscale;  // softmax scale * log2(e)

    for (int h = hfirst; h < hend; ++h) {
        {
            const int64_t p0 = slab_start(a, tab, h), p1 = slab_start(a, tab, h + 1);
            if (max(A, p0) >= min(Bc, p1)) continue;  // empty slab: nothing to merge (uniform)
        }
        const int b = h / a.Hkv, g = h - b * a.Hkv;
        // q of the group, unscaled, as packed fp32 pairs of the lane's dims.
        uint64_t q2[G][DPL / 2];
#pragma unroll
        for (int j = 0; j < G; ++j) {
            const uint16_t* qrow = a.q + ((int64_t)b * a.H + g * G + j) * kHeadDim;
#pragma unroll
            for (int i = 0; i < NCH; ++i) {
                const uint4 w = *reinterpret_cast<const uint4*>(qrow + 8 * (sl + LPR * i));
                q2[j][4 * i + 0] = bf2_to_f2(w.x);
                q2[j][4 * i + 1] = bf2_to_f2(w.y);
                q2[j][4 * i + 2] = bf2_to_f2(w.z);
                q2[j][4 * i + 3] = bf2_to_f2(w.w);
            }
        }
        // Running state: m per head (same in every lane), the lane's share of l
        // for its score slots, o for its dims of its rows.
        float m_all[G], m_my[NSUM], l_my[NSUM];
        uint64_t o2[G][DPL / 2];
#pragma unroll
        for (int j = 0; j < G; ++j) {
            m_all[j] = -INFINITY;
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) o2[j][i] = 0ull;
        }
#pragma unroll
        for (int u = 0; u < NSUM; ++u) {
            m_my[u] = -INFINITY;
            l_my[u] = 0.f;
        }

        while (cp.h == h) {
            const int64_t x0 = cp.s0 + (int64_t)cp.t * TR;
            const int cnt = (int)min((int64_t)TR, cp.s1 - x0);
            const int r0 = (int)(x0 - cp.p0);
            unsigned char* kt = my_ring + stage * C::kStageBytes;
            unsigned char* vt = kt + TR * kRowBytes;
            if (!dead) {
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
                if (cp.app && r0 + cnt == cp.n_h) {
                    // This step's token: into the tile from k_new/v_new, and into the
                    // slab's next free row for later steps.
                    const int half = lane >> 4, sub = lane & 15;
                    const int rr = cnt - 1;
                    const uint16_t* src = (half ? a.v_new : a.k_new) + ((int64_t)b * a.Hkv + g) * kHeadDim;
                    const uint4 v = *(reinterpret_cast<const uint4*>(src) + sub);
                    *reinterpret_cast<uint4*>((half ? vt : kt) + rr * kRowBytes + sub * 16) = v;
                    uint16_t* dstg = (half ? a.Vc : a.Kc) + (cp.base + (cp.n_h - 1)) * kHeadDim;
                    *(reinterpret_cast<uint4*>(dstg) + sub) = v;
                    fence_proxy_async_smem();  // order these generic writes before later bulk copies
                    __syncwarp();
                }

                // q.k partial sums over the lane's dims -> red[j][r][step][sl].
#pragma unroll
                for (int st = 0; st < STEPS; ++st) {
                    const int row = st * RPS + r;
                    uint64_t k2[DPL / 2];
#pragma unroll
                    for (int i = 0; i < NCH; ++i) {
                        const uint4 w = *reinterpret_cast<const uint4*>(kt + row * kRowBytes + 16 * (sl + LPR * i));
                        k2[4 * i + 0] = bf2_to_f2(w.x);
                        k2[4 * i + 1] = bf2_to_f2(w.y);
                        k2[4 * i + 2] = bf2_to_f2(w.z);
                        k2[4 * i + 3] = bf2_to_f2(w.w);
                    }
#pragma unroll
                    for (int j = 0; j < G; ++j) {
                        uint64_t acc = mul2(q2[j][0], k2[0]);
#pragma unroll
                        for (int i = 1; i < DPL / 2; ++i) acc = fma2(q2[j][i], k2[i], acc);
                        const float2 f = upk(acc);
                        red[j * C::JS + r * C::RS + st * LPR + sl] = f.x + f.y;
                    }
                }
                __syncwarp();
                // Full scores of the lane's slots: slot k = lane + 32u -> (row k % TR, head k / TR).
                float sc[NSUM];
#pragma unroll
                for (int u = 0; u < NSUM; ++u) {
                    const int k = lane + 32 * u;
                    const int row = k % TR, j = k / TR;
                    float v = -INFINITY;
                    if (j < G) {
                        const float4* src = reinterpret_cast<const float4*>(
                            red + j * C::JS + (row % RPS) * C::RS + (row / RPS) * LPR);
                        float4 acc = src[0];
#pragma unroll
                        for (int i = 1; i < LPR / 4; ++i) {
                            const float4 x = src[i];
                            acc.x += x.x;
                            acc.y += x.y;
                            acc.z += x.z;
                            acc.w += x.w;
                        }
                        const float d = (acc.x + acc.y) + (acc.z + acc.w);
                        if (row < cnt) v = d;
                    }
                    sc[u] = v;
                }
                // Tile max per head (over the TR lanes that hold that head), then
                // the new running max of every head in every lane.
                float mnew_my[NSUM];
#pragma unroll
                for (int u = 0; u < NSUM; ++u) {
                    float x = sc[u];
#pragma unroll
                    for (int o = TR / 2; o >= 1; o >>= 1) x = fmaxf(x, __shfl_xor_sync(kFull, x, o));
                    mnew_my[u] = fmaxf(m_my[u], x * cs);
                }
                float mnew_all[G];
                bool grow = false;
#pragma unroll
                for (int j = 0; j < G; ++j) {
                    mnew_all[j] = __shfl_sync(kFull, mnew_my[(j * TR) / 32], (j * TR) % 32);
                    grow |= mnew_all[j] > m_all[j];
                }
                if (__any_sync(kFull, grow)) {  // rare after the first tiles
#pragma unroll
                    for (int j = 0; j < G; ++j) {
                        const float al = (mnew_all[j] == -INFINITY) ? 1.f : ex2(m_all[j] - mnew_all[j]);
                        const uint64_t al2 = pk(al, al);
#pragma unroll
                        for (int i = 0; i < DPL / 2; ++i) o2[j][i] = mul2(o2[j][i], al2);
                        m_all[j] = mnew_all[j];
                    }
#pragma unroll
                    for (int u = 0; u < NSUM; ++u)
                        l_my[u] *= (mnew_my[u] == -INFINITY) ? 1.f : ex2(m_my[u] - mnew_my[u]);
                }
#pragma unroll
                for (int u = 0; u < NSUM; ++u) {
                    m_my[u] = mnew_my[u];
                    const int k = lane + 32 * u;
                    const int row = k % TR, j = k / TR;
                    const float p = (sc[u] == -INFINITY) ? 0.f : ex2(fmaf(sc[u], cs, -m_my[u]));
                    l_my[u] += p;
                    if (j < G) ps[row * C::GP + j] = p;
                }
                __syncwarp();
                // o += p v over the lane's dims.
#pragma unroll
                for (int st = 0; st < STEPS; ++st) {
                    const int row = st * RPS + r;
                    float pj[C::GP];
#pragma unroll
                    for (int q4 = 0; q4 < C::GP / 4; ++q4) {
                        const float4 pv = *reinterpret_cast<const float4*>(ps + row * C::GP + 4 * q4);
                        pj[4 * q4 + 0] = pv.x;
                        pj[4 * q4 + 1] = pv.y;
                        pj[4 * q4 + 2] = pv.z;
                        pj[4 * q4 + 3] = pv.w;
                    }
                    uint64_t v2[DPL / 2];
                    const bool valid = row < cnt;
#pragma unroll
                    for (int i = 0; i < NCH; ++i) {
                        uint4 w = *reinterpret_cast<const uint4*>(vt + row * kRowBytes + 16 * (sl + LPR * i));
                        if (!valid) w = make_uint4(0u, 0u, 0u, 0u);  // stale bytes may not be finite
                        v2[4 * i + 0] = bf2_to_f2(w.x);
                        v2[4 * i + 1] = bf2_to_f2(w.y);
                        v2[4 * i + 2] = bf2_to_f2(w.z);
                        v2[4 * i + 3] = bf2_to_f2(w.w);
                    }
#pragma unroll
                    for (int j = 0; j < G; ++j) {
                        const uint64_t pp = pk(pj[j], pj[j]);
#pragma unroll
                        for (int i = 0; i < DPL / 2; ++i) o2[j][i] = fma2(pp, v2[i], o2[j][i]);
                    }
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

        // Warp state of this segment: o summed over the RPS row lanes (same m), l
        // summed over the TR lanes of each head, then broadcast per head.
#pragma unroll
        for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
            for (int j = 0; j < G; ++j)
#pragma unroll
                for (int i = 0; i < DPL / 2; ++i) {
                    const float2 f = upk(o2[j][i]);
                    o2[j][i] = add2(o2[j][i], pk(__shfl_xor_sync(kFull, f.x, o), __shfl_xor_sync(kFull, f.y, o)));
                }
        float l_all[G];
#pragma unroll
        for (int u = 0; u < NSUM; ++u) {
            float x = l_my[u];
#pragma unroll
            for (int o = TR / 2; o >= 1; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
            l_my[u] = x;
        }
#pragma unroll
        for (int j = 0; j < G; ++j) l_all[j] = __shfl_sync(kFull, l_my[(j * TR) / 32], (j * TR) % 32);

        __syncthreads();  // every warp is done with its red/ps scratch, which mrg overlaps
        float* mw = mrg + warp * G * (kHeadDim + 2);
        if (r == 0) {
#pragma unroll
            for (int j = 0; j < G; ++j) {
#pragma unroll
                for (int i = 0; i < NCH; ++i) {
                    // (kHeadDim + 2) floats per head is not 16-byte aligned: plain stores.
                    float* d = mw + j * (kHeadDim + 2) + 8 * (sl + LPR * i);
                    const float2 a0 = upk(o2[j][4 * i + 0]), a1 = upk(o2[j][4 * i + 1]);
                    const float2 a2 = upk(o2[j][4 * i + 2]), a3 = upk(o2[j][4 * i + 3]);
                    d[0] = a0.x; d[1] = a0.y; d[2] = a1.x; d[3] = a1.y;
                    d[4] = a2.x; d[5] = a2.y; d[6] = a3.x; d[7] = a3.y;
                }
                if (sl == 0) {
                    mw[j * (kHeadDim + 2) + kHeadDim] = m_all[j];
                    mw[j * (kHeadDim + 2) + kHeadDim + 1] = l_all[j];
                }
            }
        }
        __syncthreads();
        // Merge the NW warp states into the CTA's partial for slab h.
        const int64_t slot = (int64_t)c + h;
        for (int i = threadIdx.x; i < G * kHeadDim; i += NW * 32) {
            const int j = i / kHeadDim, d = i - j * kHeadDim;
            float M = -INFINITY;
#pragma unroll
            for (int w = 0; w < NW; ++w) M = fmaxf(M, mrg[(w * G + j) * (kHeadDim + 2) + kHeadDim]);
            float O = 0.f, Lsum = 0.f;
#pragma unroll
            for (int w = 0; w < NW; ++w) {
                const float* st = mrg + (w * G + j) * (kHeadDim + 2);
                const float f = (st[kHeadDim] == -INFINITY) ? 0.f : ex2(st[kHeadDim] - M);
                O = fmaf(st[d], f, O);
                Lsum = fmaf(st[kHeadDim + 1], f, Lsum);
            }
            a.work_o[(slot * G + j) * kHeadDim + d] = O;
            if (d == 0) {
                a.work_ml[(slot * G + j) * 2] = M;
                a.work_ml[(slot * G + j) * 2 + 1] = Lsum;
            }
        }
        __syncthreads();  // mrg (and the warps' scratch) is reused by the next segment
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
// One CTA per (b, q-head): kCombineWarps warps split the slab's partials,
// each keeps its loads in flight, then the CTA sums the warps' shares.
constexpr int kCombineWarps = 4;
constexpr int kCombineStride = kHeadDim + 4;  // floats per warp share: o[128], L, pad (16-byte rows)

__global__ void __launch_bounds__(kCombineWarps * 32) decode_combine_kernel(const DecodeArgs a)
{
    extern __shared__ int32_t csmem[];
    SeqTable tab{csmem, csmem + a.B};
    // [kCombineWarps][kCombineStride] floats after the table, at a 16-byte boundary.
    float* red = reinterpret_cast<float*>(csmem + (((2 * a.B + 1) + 3) & ~3));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp == 0) build_seq_table(a, tab, false);
    __syncthreads();

    const int pair = blockIdx.x;  // (b, q-head)
    const int b = pair / a.H, hq = pair - b * a.H;
    const int g = hq / a.G, j = hq - g * a.G;
    const int h = b * a.Hkv + g;
    const int NHl = a.B * a.Hkv;
    const int64_t R = slab_start(a, tab, NHl);
    const int64_t p0 = slab_start(a, tab, h), p1 = slab_start(a, tab, h + 1);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float Lw = 0.f;
    if (p1 > p0) {
        const int c0 = cta_of(p0, R, a.nctas), c1 = cta_of(p1 - 1, R, a.nctas);
        // Global max over the partials (lanes in parallel), same in every warp.
        float M = -INFINITY;
        for (int cc = c0 + lane; cc <= c1; cc += 32)
            if (cta_start(cc, R, a.nctas) < cta_start(cc + 1, R, a.nctas))
                M = fmaxf(M, a.work_ml[(((int64_t)cc + h) * a.G + j) * 2]);
#pragma unroll
        for (int o = 16; o >= 1; o >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, o));
#pragma unroll 4
        for (int cc = c0 + warp; cc <= c1; cc += kCombineWarps) {
            if (cta_start(cc, R, a.nctas) == cta_start(cc + 1, R, a.nctas)) continue;
            const int64_t sj = ((int64_t)cc + h) * a.G + j;
            const float mc = a.work_ml[sj * 2], lc = a.work_ml[sj * 2 + 1];
            const float f = (mc == -INFINITY) ? 0.f : ex2(mc - M);
            Lw = fmaf(lc, f, Lw);
            const float4 v = *reinterpret_cast<const float4*>(a.work_o + sj * kHeadDim + 4 * lane);
            acc.x = fmaf(v.x, f, acc.x);
            acc.y = fmaf(v.y, f, acc.y);
            acc.z = fmaf(v.z, f, acc.z);
            acc.w = fmaf(v.w, f, acc.w);
        }
    }
    float* rw = red + warp * kCombineStride;
    reinterpret_cast<float4*>(rw)[lane] = acc;
    if (lane == 0) rw[kHeadDim] = Lw;
    __syncthreads();
    if (warp == 0) {
        float4 o = make_float4(0.f, 0.f, 0.f, 0.f);
        float L = 0.f;
#pragma unroll
        for (int w = 0; w < kCombineWarps; ++w) {
            const float4 x = reinterpret_cast<const float4*>(red + w * kCombineStride)[lane];
            o.x += x.x;
            o.y += x.y;
            o.z += x.z;
            o.w += x.w;
            L += red[w * kCombineStride + kHeadDim];
        }
        const float inv = L > 0.f ? 1.f / L : 0.f;
        o.x *= inv;
        o.y *= inv;
        o.z *= inv;
        o.w *= inv;
        *reinterpret_cast<float4*>(a.out + ((int64_t)b * a.H + hq) * kHeadDim + 4 * lane) = o;
    }
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
// G <= 4: a quarter-warp per row (16 dims a lane), 16-row tiles, 3 stages.
// G >= 5: a half-warp per row (8 dims a lane), 8-row tiles, 5 stages.
template <int G>
using PKFor = typename std::conditional<(G <= 4), PK<G, 8, 16, 3, 8>, PK<G, 16, 8, 5, 8>>::type;

template <int G>
cudaError_t launch_partial_g(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    decode_partial_kernel<PKFor<G>><<<cfg.nctas, PKFor<G>::NW * 32, cfg.smem_bytes, st>>>(a);
    return cudaGetLastError();
}

template <int G>
cudaError_t config_g(int B, DecodeConfig* cfg)
{
    using C = PKFor<G>;
    const int smem = C::bytes(B);
    cudaError_t e = cudaFuncSetAttribute(decode_partial_kernel<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_partial_kernel<C>, C::NW * 32, smem)) !=
        cudaSuccess)
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
    const int smem = (2 * a.B + 1) * 4 + 16 + kCombineWarps * kCombineStride * 4;
    decode_combine_kernel<<<pairs, kCombineWarps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_advance(int32_t* n_app, int B, int reserve, int32_t* status, cudaStream_t st)
{
    advance_kernel<<<(B + 127) / 128, 128, 0, st>>>(n_app, B, reserve, status);
    return cudaGetLastError();
}

}  // namespace dkv
