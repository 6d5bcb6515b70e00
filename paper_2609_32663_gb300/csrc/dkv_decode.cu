// Decode-step attention over the packed cache (Sec. 3.4), split-K.
//
// Work split ("stream-K" over rows). For one layer, the rows of all slabs
// h = b*Hkv + g are laid end to end: slab h owns layer rows [P(h), P(h+1)),
// n_h = len[h] + appended[b] (+1 for this step's token). CTA c of P takes rows
// [A(c), A(c+1)), A(c) = floor(c*R/P), so every CTA streams the same number of
// bytes whatever the slab lengths; its warps split that range into equal
// contiguous pieces and run independently (no barrier until the end). Each CTA
// writes one partial (m, l, o) per slab it touches into slot c + h; the slots
// are distinct because CTA ranges and slabs are both in row order. The combine
// kernel merges, for each (b, q-head), the partials of the CTAs covering its slab.
//
// A warp fetches its tiles of TR rows (K and V, 256 bytes a row) with
// cp.async.bulk into its own ring of NS shared-memory stages, each completing
// on an mbarrier. LPR lanes share a row (16 or 8 dims each): q.k partial sums
// use packed f32x2 FMAs and are summed across the LPR lanes through a small
// shared-memory transpose; the softmax is online in base 2 (scores scaled by
// scale*log2 e) with one exp per (row, head); o += p v again in f32x2. A warp
// keeps the state of its last slab in registers; the state of a slab it leaves
// earlier goes to a per-warp record (first slab) or straight to the CTA's slot
// (a slab wholly inside the warp's range). Warps do not wait for each other
// until their ranges are done; then the CTA merges the states that share a slab.
#include "dkv_decode_common.cuh"

#include <math.h>

#include <type_traits>

namespace dkv {
namespace {

// (constants, partition and merge helpers: dkv_decode_common.cuh; PTX wrappers: dkv_ptx.cuh)

// ------------------------------------------------------------ partial kernel
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

__device__ __forceinline__ void bf8_to_f2x4(const uint4& w, uint64_t* out)
{
    out[0] = bf2_to_f2(w.x);
    out[1] = bf2_to_f2(w.y);
    out[2] = bf2_to_f2(w.z);
    out[3] = bf2_to_f2(w.w);
}

// Compile-time geometry of the partial kernel.
//   LPR lanes share one row; a lane owns DPL = 128/LPR dims, i.e. NCH 16-byte
//   chunks c = sl + LPR*i of the row; a warp step covers RPS = 32/LPR rows; a
//   tile of TR rows takes STEPS steps. A tile has TR*G scores, NSUM per lane:
//   slot u of lane l is (row l % TR, head l / TR + u * 32/TR).
template <int G_, int LPR_, int TR_, int NS_, int NW_>
struct PK {
    static constexpr int G = G_, LPR = LPR_, TR = TR_, NS = NS_, NW = NW_;
    static_assert(PRE <= NS, "the tiles fetched before the PDL wait fit the warp's ring");
    static constexpr int RPS = 32 / LPR;
    static constexpr int DPL = kHeadDim / LPR;
    static constexpr int NCH = DPL / 8;
    static constexpr int STEPS = TR / RPS;
    static constexpr int HPU = 32 / TR;  // heads per score slot index u
    static constexpr int NSUM = (G + HPU - 1) / HPU;
    static constexpr int GP = G <= 4 ? 4 : 8;  // p pairs per row in shared memory
    // Reduction buffer red[j][step][r][sl]: the 32 lanes of one store (fixed j,
    // step) write 32 consecutive floats; a score sums LPR consecutive floats.
    // The p pairs of a tile reuse the same bytes once the scores are read.
    static constexpr int kRedFloats = G * STEPS * 32;
    static constexpr int kPFloats = TR * GP * 2;
    static constexpr int kWarpScratch = ((kRedFloats > kPFloats ? kRedFloats : kPFloats) * 4 + 15) / 16 * 16;
    static constexpr int kStageBytes = 2 * TR * kRowBytes;  // K tile then V tile
    static constexpr int kRingBytes = NW * NS * kStageBytes;
    static constexpr int kScratchBytes = NW * kWarpScratch;
    static constexpr int kBarBytes = NW * NS * 8;
    static constexpr int kMetaBytes = NW * 6 * 4 + 16;  // first/last slab of each warp, their row bounds
    static constexpr int kFixedBytes = kRingBytes + kScratchBytes + kBarBytes + kMetaBytes;
    static constexpr int kStateFloats = G * (kHeadDim + 2);
    static int bytes(int B) { return kFixedBytes + seq_table_bytes(B); }
    static_assert(kFixedBytes + seq_table_bytes(kMaxB) <= 227 * 1024, "fits the opt-in shared memory of one CTA");
    static_assert(TR % RPS == 0 && 32 % TR == 0, "tile geometry");
    static_assert(kStateFloats * 4 <= NS * kStageBytes, "a warp's final state fits in its ring");
};

// Per-warp running state of one slab segment.
template <class C>
struct State {
    float m_all[C::G];       // running max per head (log2 domain), same in every lane
    float m_my[C::NSUM];     // running max of the heads of the lane's score slots
    float l_my[C::NSUM];     // the lane's share of the softmax denominator
    uint64_t o2[C::G][C::DPL / 2];  // unnormalised output, the lane's dims of its rows
};

// One tile: scores, online softmax, o += p v. FULL: all TR rows are valid.
template <class C, bool FULL>
__device__ __forceinline__ void tile_compute(State<C>& S, const uint64_t (&q2)[C::G][C::DPL / 2],
                                             const unsigned char* kt, const unsigned char* vt, float* red,
                                             float2* ps, int cnt, float cs, int lane)
{
    constexpr int G = C::G, LPR = C::LPR, TR = C::TR, RPS = C::RPS, DPL = C::DPL, NCH = C::NCH;
    constexpr int STEPS = C::STEPS, NSUM = C::NSUM, HPU = C::HPU;
    const int r = lane / LPR, sl = lane % LPR;

    // q.k partial sums over the lane's dims -> red[j][step][r][sl].
#pragma unroll
    for (int st = 0; st < STEPS; ++st) {
        const int row = st * RPS + r;
        uint64_t k2[DPL / 2];
#pragma unroll
        for (int i = 0; i < NCH; ++i)
            bf8_to_f2x4(*reinterpret_cast<const uint4*>(kt + row * kRowBytes + 16 * (sl + LPR * i)), k2 + 4 * i);
#pragma unroll
        for (int j = 0; j < G; ++j) {
            uint64_t acc = mul2(q2[j][0], k2[0]);
#pragma unroll
            for (int i = 1; i < DPL / 2; ++i) acc = fma2(q2[j][i], k2[i], acc);
            const float2 f = upk(acc);
            red[(j * STEPS + st) * 32 + lane] = f.x + f.y;
        }
    }
    __syncwarp();
    // Full scores of the lane's slots.
    const int row = lane % TR;
    float sc[NSUM];
#pragma unroll
    for (int u = 0; u < NSUM; ++u) {
        const int j = lane / TR + u * HPU;
        float v = -INFINITY;
        if (NSUM * HPU == G || j < G) {
            const float4* src = reinterpret_cast<const float4*>(red + (j * STEPS + row / RPS) * 32 +
                                                                 (row % RPS) * LPR);
            float4 acc = src[0];
#pragma unroll
            for (int i = 1; i < LPR / 4; ++i) {
                const float4 x = src[i];
                acc.x += x.x;
                acc.y += x.y;
                acc.z += x.z;
                acc.w += x.w;
            }
            v = (acc.x + acc.y) + (acc.z + acc.w);
            if (!FULL && row >= cnt) v = -INFINITY;
        }
        sc[u] = v;
    }
    // Lazy rescaling: the running max m of a head only moves when a score tops it
    // by more than kSlack (log2 units), so p = 2^(s - m) <= 2^kSlack and most tiles
    // need one vote instead of a cross-lane max. The first tile always moves m.
    bool over = false;
#pragma unroll
    for (int u = 0; u < NSUM; ++u) over |= sc[u] * cs > S.m_my[u] + kSlack;
    if (__any_sync(kFull, over)) {
        float mnew_my[NSUM];
#pragma unroll
        for (int u = 0; u < NSUM; ++u) {
            float x = sc[u];
#pragma unroll
            for (int o = TR / 2; o >= 1; o >>= 1) x = fmaxf(x, __shfl_xor_sync(kFull, x, o));
            mnew_my[u] = fmaxf(S.m_my[u], x * cs);
        }
#pragma unroll
        for (int j = 0; j < G; ++j) {
            const float mn = __shfl_sync(kFull, mnew_my[j / HPU], (j % HPU) * TR);
            const float al = (mn == -INFINITY) ? 1.f : ex2(S.m_all[j] - mn);
            const uint64_t al2 = pk(al, al);
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) S.o2[j][i] = mul2(S.o2[j][i], al2);
            S.m_all[j] = mn;
        }
#pragma unroll
        for (int u = 0; u < NSUM; ++u) {
            S.l_my[u] *= (mnew_my[u] == -INFINITY) ? 1.f : ex2(S.m_my[u] - mnew_my[u]);
            S.m_my[u] = mnew_my[u];
        }
    }
    __syncwarp();  // the p pairs below overwrite the reduction buffer
#pragma unroll
    for (int u = 0; u < NSUM; ++u) {
        const int j = lane / TR + u * HPU;
        const float mref = (S.m_my[u] == -INFINITY) ? 0.f : S.m_my[u];
        const float p = ex2(fmaf(sc[u], cs, -mref));  // exp2(-inf) = 0 for masked rows
        S.l_my[u] += p;
        if (NSUM * HPU == G || j < G) ps[row * C::GP + j] = make_float2(p, p);
    }
    __syncwarp();
    // o += p v over the lane's dims.
#pragma unroll
    for (int st = 0; st < STEPS; ++st) {
        const int vrow = st * RPS + r;
        uint64_t pp[C::GP];
#pragma unroll
        for (int q4 = 0; q4 < C::GP / 2; ++q4) {
            const ulonglong2 w = *reinterpret_cast<const ulonglong2*>(ps + vrow * C::GP + 2 * q4);
            pp[2 * q4] = w.x;
            pp[2 * q4 + 1] = w.y;
        }
        uint64_t v2[DPL / 2];
#pragma unroll
        for (int i = 0; i < NCH; ++i) {
            uint4 w = *reinterpret_cast<const uint4*>(vt + vrow * kRowBytes + 16 * (sl + LPR * i));
            if (!FULL && vrow >= cnt) w = make_uint4(0u, 0u, 0u, 0u);  // stale bytes may not be finite
            bf8_to_f2x4(w, v2 + 4 * i);
        }
#pragma unroll
        for (int j = 0; j < G; ++j)
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) S.o2[j][i] = fma2(pp[j], v2[i], S.o2[j][i]);
    }
}

// Final answer of a slab held by one warp: out = o / l for the lane's dims
// (lanes with r == 0 hold o after finish_state).
template <class C>
__device__ __forceinline__ void write_out_state(const DecodeArgs& a, const State<C>& S, const float (&l_all)[C::G],
                                                int b, int g, int lane)
{
    constexpr int G = C::G, LPR = C::LPR, NCH = C::NCH;
    const int r = lane / LPR, sl = lane % LPR;
    if (r != 0) return;
#pragma unroll
    for (int j = 0; j < G; ++j) {
        const float inv = l_all[j] > 0.f ? 1.f / l_all[j] : 0.f;
        float* dst = a.out + ((int64_t)b * a.H + g * G + j) * kHeadDim;
#pragma unroll
        for (int i = 0; i < NCH; ++i) {
            float4* d = reinterpret_cast<float4*>(dst + 8 * (sl + LPR * i));
            const float2 a0 = upk(S.o2[j][4 * i + 0]), a1 = upk(S.o2[j][4 * i + 1]);
            const float2 a2 = upk(S.o2[j][4 * i + 2]), a3 = upk(S.o2[j][4 * i + 3]);
            d[0] = make_float4(a0.x * inv, a0.y * inv, a1.x * inv, a1.y * inv);
            d[1] = make_float4(a2.x * inv, a2.y * inv, a3.x * inv, a3.y * inv);
        }
    }
}

// Writes a warp state (o over the lane's dims for the RPS row lanes already
// summed, m and l per head) as one record: o[G][128] at o_dst, (m, l)[G] at ml_dst.
template <class C>
__device__ __forceinline__ void store_state(const State<C>& S, const float (&l_all)[C::G], float* o_dst,
                                            float* ml_dst, int lane)
{
    constexpr int G = C::G, LPR = C::LPR, NCH = C::NCH;
    const int r = lane / LPR, sl = lane % LPR;
    if (r == 0) {
#pragma unroll
        for (int j = 0; j < G; ++j)
#pragma unroll
            for (int i = 0; i < NCH; ++i) {
                float4* d = reinterpret_cast<float4*>(o_dst + j * kHeadDim + 8 * (sl + LPR * i));
                const float2 a0 = upk(S.o2[j][4 * i + 0]), a1 = upk(S.o2[j][4 * i + 1]);
                const float2 a2 = upk(S.o2[j][4 * i + 2]), a3 = upk(S.o2[j][4 * i + 3]);
                d[0] = make_float4(a0.x, a0.y, a1.x, a1.y);
                d[1] = make_float4(a2.x, a2.y, a3.x, a3.y);
            }
    }
    if (lane == 0) {
#pragma unroll
        for (int j = 0; j < G; ++j) *reinterpret_cast<float2*>(ml_dst + 2 * j) = make_float2(S.m_all[j], l_all[j]);
    }
}

// Sums a segment's state over the RPS row lanes (o) and the TR lanes of each
// head (l); afterwards lanes with r == 0 hold o of their dims, l_all is per head.
template <class C>
__device__ __forceinline__ void finish_state(State<C>& S, float (&l_all)[C::G])
{
    constexpr int G = C::G, LPR = C::LPR, TR = C::TR, DPL = C::DPL, NSUM = C::NSUM, HPU = C::HPU;
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
        for (int j = 0; j < G; ++j)
#pragma unroll
            for (int i = 0; i < DPL / 2; ++i) {
                const float2 f = upk(S.o2[j][i]);
                S.o2[j][i] = add2(S.o2[j][i], pk(__shfl_xor_sync(kFull, f.x, o), __shfl_xor_sync(kFull, f.y, o)));
            }
#pragma unroll
    for (int u = 0; u < NSUM; ++u) {
        float x = S.l_my[u];
#pragma unroll
        for (int o = TR / 2; o >= 1; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
        S.l_my[u] = x;
    }
#pragma unroll
    for (int j = 0; j < G; ++j) l_all[j] = __shfl_sync(kFull, S.l_my[j / HPU], (j % HPU) * TR);
}

template <class C, bool FUSED>
__global__ void __launch_bounds__(C::NW * 32, 1) decode_partial_kernel(const DecodeArgs a)
{
    constexpr int G = C::G, LPR = C::LPR, TR = C::TR, NS = C::NS, NW = C::NW;
    constexpr int DPL = C::DPL, NCH = C::NCH, NSUM = C::NSUM;
    extern __shared__ __align__(128) unsigned char smem[];
    const SeqTable tab = seq_table_at(smem + C::kFixedBytes, a);
    int32_t* seg_first = reinterpret_cast<int32_t*>(smem + C::kRingBytes + C::kScratchBytes + C::kBarBytes);
    int32_t* seg_last = seg_first + NW;
    int32_t* seg_p0 = seg_first + 2 * NW;  // [2 NW] layer rows [p0, p1) of entry 2 w (first) / 2 w + 1 (last)
    int32_t* seg_p1 = seg_first + 4 * NW;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sl = lane % LPR;
    const int NHl = a.B * a.Hkv;
    const int c = blockIdx.x;
    uint64_t* my_bars = reinterpret_cast<uint64_t*>(smem + C::kRingBytes + C::kScratchBytes) + warp * NS;

    if (warp == 0)
        build_seq_table(a, tab, c == 0);
    else
        load_slab_cache(a, tab, 32, (NW - 1) * 32);
    if (lane == 0) {
        for (int s = 0; s < NS; ++s) mbar_init(smem_u32(&my_bars[s]), 1);
        fence_proxy_async_smem();
        seg_first[warp] = -1;
        seg_last[warp] = -1;
    }
    __syncthreads();  // table, barriers and slab entries are ready
    pdl_launch_dependents();

    const int R = slab_start(a, tab, NHl);
    if (FUSED && c == a.nctas - 1 && warp == 0) {
        // Slabs with no rows belong to no CTA: their outputs are zero (written by
        // the last CTA, which always runs; after the wait, as any write of out).
        pdl_wait();
        for (int h = 0; h < NHl; ++h)
            if (slab_start(a, tab, h) == slab_start(a, tab, h + 1))
                for (int j = 0; j < G; ++j)
                    write_out<G>(a, h / a.Hkv, h % a.Hkv, j, make_float4(0.f, 0.f, 0.f, 0.f), 0.f, lane);
    }
    const int A = part_start(c, R, a.nctas), Bc = part_start(c + 1, R, a.nctas);
    if (A >= Bc) return;  // uniform: this CTA has no rows
    const int wA = A + (int)(((int64_t)(Bc - A) * warp) / NW);
    const int wB = A + (int)(((int64_t)(Bc - A) * (warp + 1)) / NW);
    unsigned char* my_ring = smem + warp * NS * C::kStageBytes;
    State<C> S;
    float l_all[G];
    bool have_last = false;  // S holds the state of this warp's last slab

    if (wA < wB) {
        const int hfirst = slab_containing(a, tab, NHl, wA);
        const int hlast = slab_containing(a, tab, NHl, wB - 1);
        const int hend = hlast + 1;
        const uint64_t pol = evict_first_policy();
        float* red = reinterpret_cast<float*>(smem + C::kRingBytes + warp * C::kWarpScratch);
        float2* ps = reinterpret_cast<float2*>(red);

        Cursor ld;
        ld.h = hfirst;
        cursor_seek(ld, a, tab, hend, wA, wB);
        Cursor cp = ld;

        auto issue = [&](const Cursor& cu, int stage) {
            const int cnt = min(TR, cu.s1 - cu.x);
            const int r0 = cu.x - cu.p0;  // row within the slab
            int ncopy = (cu.app && r0 + cnt == cu.n_h) ? cnt - 1 : cnt;  // new token comes from k_new
            // Bounds-checked build: rows outside the cache are not copied (the stage's
            // barrier then expects no bytes, so its wait still completes).
            if (!in_bounds(cu.base + r0 >= 0 && (a.rows_cap == 0 || cu.base + r0 + ncopy <= a.rows_cap), a.status))
                ncopy = 0;
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

        // A bounded wait that runs out marks the warp dead: it stops issuing and
        // computing, drains its copies in flight, and leaves its partials unwritten.
        bool dead = false;
        int inflight = 0;
        if (lane == 0) {
            Cursor it = ld;
            for (int s = 0; s < PRE && it.h < hend; ++s) {
                issue(it, s);
                cursor_next<TR>(it, a, tab, hend, wA, wB);
            }
        }
        for (int s = 0; s < PRE && ld.h < hend; ++s) {
            ++inflight;
            cursor_next<TR>(ld, a, tab, hend, wA, wB);
        }
        // Everything above reads only the plan, n_appended and the cache rows of
        // earlier steps; q, k_new, v_new, the cache slots written here and the
        // workspace belong to the previous kernel's epoch.
        pdl_wait();
        if (lane == 0) {
            Cursor it = ld;
            for (int s = PRE; s < NS && it.h < hend; ++s) {
                issue(it, s);
                cursor_next<TR>(it, a, tab, hend, wA, wB);
            }
        }
        for (int s = PRE; s < NS && ld.h < hend; ++s) {
            ++inflight;
            cursor_next<TR>(ld, a, tab, hend, wA, wB);
        }
        int stage = 0;
        uint32_t phase = 0;
        const float cs = a.qscale;  // softmax scale * log2(e)

        while (cp.h < hend && !dead) {
            const int h = cp.h;
            const int p0h = cp.p0, p1h = cp.p0 + cp.n_h;  // the slab's layer rows
            const int b = h / a.Hkv, g = h - b * a.Hkv;
            // q of the group, unscaled, as packed fp32 pairs of the lane's dims.
            uint64_t q2[G][DPL / 2];
#pragma unroll
            for (int j = 0; j < G; ++j) {
                const uint16_t* qrow = a.q + ((int64_t)b * a.H + g * G + j) * kHeadDim;
#pragma unroll
                for (int i = 0; i < NCH; ++i)
                    bf8_to_f2x4(__ldg(reinterpret_cast<const uint4*>(qrow + 8 * (sl + LPR * i))), q2[j] + 4 * i);
            }
#pragma unroll
            for (int j = 0; j < G; ++j) {
                S.m_all[j] = -INFINITY;
#pragma unroll
                for (int i = 0; i < DPL / 2; ++i) S.o2[j][i] = 0ull;
            }
#pragma unroll
            for (int u = 0; u < NSUM; ++u) {
                S.m_my[u] = -INFINITY;
                S.l_my[u] = 0.f;
            }

            while (cp.h == h) {
                const int cnt = min(TR, cp.s1 - cp.x);
                const int r0 = cp.x - cp.p0;
                unsigned char* kt = my_ring + stage * C::kStageBytes;
                unsigned char* vt = kt + TR * kRowBytes;
                // Every lane observes the completed phase itself (acquire) before reading.
                if (!__all_sync(kFull, mbar_wait(smem_u32(&my_bars[stage]), phase))) {
                    dead = true;
                    if (lane == 0) atomicOr(a.status, 0x2 /* DKV_DEV_TMA_TIMEOUT */);
                    break;
                }
                --inflight;
                if (cp.app && r0 + cnt == cp.n_h) {
                    // This step's token: into the tile from k_new/v_new, and into the
                    // slab's next free row for later steps.
                    const int half = lane >> 4, sub = lane & 15;
                    const uint16_t* src = (half ? a.v_new : a.k_new) + ((int64_t)b * a.Hkv + g) * kHeadDim;
                    const uint4 v = __ldg(reinterpret_cast<const uint4*>(src) + sub);
                    *reinterpret_cast<uint4*>((half ? vt : kt) + (cnt - 1) * kRowBytes + sub * 16) = v;
                    const int64_t nrow = cp.base + (cp.n_h - 1);
                    if (in_bounds(nrow >= 0 && (a.rows_cap == 0 || nrow < a.rows_cap), a.status)) {
                        uint16_t* dstg = (half ? a.Vc : a.Kc) + nrow * kHeadDim;
                        *(reinterpret_cast<uint4*>(dstg) + sub) = v;
                    }
                    fence_proxy_async_smem();  // order these generic writes before later bulk copies
                    __syncwarp();
                }
                if (cnt == TR)
                    tile_compute<C, true>(S, q2, kt, vt, red, ps, cnt, cs, lane);
                else
                    tile_compute<C, false>(S, q2, kt, vt, red, ps, cnt, cs, lane);
                __syncwarp();
                // Refill this stage with the tile NS ahead.
                if (ld.h < hend) {
                    if (lane == 0) issue(ld, stage);
                    ++inflight;
                    cursor_next<TR>(ld, a, tab, hend, wA, wB);
                }
                cursor_next<TR>(cp, a, tab, hend, wA, wB);
                if (++stage == NS) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (dead) break;
            finish_state<C>(S, l_all);
            if (h == hlast) {
                have_last = true;  // merged with the other warps at the end
                if (lane == 0) {
                    seg_last[warp] = h;
                    seg_p0[2 * warp + 1] = p0h;
                    seg_p1[2 * warp + 1] = p1h;
                }
            } else if (h == hfirst) {
                const int64_t rec = (int64_t)c * NW + warp;  // this slab continues in an earlier warp
                store_state<C>(S, l_all, a.warp_o + rec * G * kHeadDim, a.warp_ml + rec * G * 2, lane);
                if (lane == 0) {
                    seg_first[warp] = h;
                    seg_p0[2 * warp] = p0h;
                    seg_p1[2 * warp] = p1h;
                }
            } else if (FUSED) {
                write_out_state<C>(a, S, l_all, b, g, lane);  // the whole slab lies in this warp's range
            } else {
                const int64_t slot = (int64_t)c + h;  // the whole slab lies in this warp's range
                store_state<C>(S, l_all, a.work_o + slot * G * kHeadDim, a.work_ml + slot * G * 2, lane);
            }
        }

        if (dead) {
            // After a timeout, wait (with the same bound) for the copies still in flight.
            if (lane == 0)
                for (int k = 0; k < inflight; ++k) {
                    mbar_wait(smem_u32(&my_bars[stage]), phase);
                    if (++stage == NS) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
        }
    }
    // The warp's own ring is idle now (every tile it issued was consumed): its
    // final state goes there. Then the CTA merges, all warps sharing the work
    // (one CTA per SM: warps that finish early have nothing else to run).
    if (have_last)
        store_state<C>(S, l_all, reinterpret_cast<float*>(my_ring), reinterpret_cast<float*>(my_ring) + G * kHeadDim,
                       lane);
    __syncthreads();
    pdl_wait();  // the merges write the workspace and out: the previous kernel must be done with them

    cta_tail<G, NW, FUSED, G>(a, smem, NS * C::kStageBytes, seg_first, c, R, warp, lane);
}

// ------------------------------------------------------------ combine kernel
// One CTA per (b, q-head): the CTA's threads find the max over the slab's
// partials, its warps split the partials (loads kept in flight), and the
// CTA sums the warps' shares.
constexpr int kCombineWarps = 8;
constexpr int kCombineStride = kHeadDim + 4;  // floats per warp share: o[128], L, pad (16-byte rows)

__global__ void __launch_bounds__(kCombineWarps * 32) decode_combine_kernel(const DecodeArgs a)
{
    extern __shared__ int32_t csmem[];
    SeqTable tab{csmem, csmem + a.B};
    // [kCombineWarps][kCombineStride] floats after the table, at a 16-byte boundary.
    float* red = reinterpret_cast<float*>(csmem + (((2 * a.B + 1) + 3) & ~3));
    __shared__ float wmax[kCombineWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    pdl_launch_dependents();
    if (warp == 0) build_seq_table(a, tab, false);
    __syncthreads();
    pdl_wait();  // the partials of the previous (partial) kernel

    const int pair = blockIdx.x;  // (b, q-head)
    const int b = pair / a.H, hq = pair - b * a.H;
    const int g = hq / a.G, j = hq - g * a.G;
    const int h = b * a.Hkv + g;
    const int NHl = a.B * a.Hkv;
    const int R = slab_start(a, tab, NHl);
    const int p0 = slab_start(a, tab, h), p1 = slab_start(a, tab, h + 1);
    float4* outp = reinterpret_cast<float4*>(a.out + ((int64_t)b * a.H + hq) * kHeadDim);
    if (p1 <= p0) {  // no rows: zeros (uniform over the CTA)
        if (warp == 0) outp[lane] = make_float4(0.f, 0.f, 0.f, 0.f);
        return;
    }
    const int P = a.nctas;
    const int c0 = part_of(p0, R, P), c1 = part_of(p1 - 1, R, P);
    float M = -INFINITY;
    for (int c = c0 + (int)threadIdx.x; c <= c1; c += kCombineWarps * 32)
        if (part_start(c, R, P) < part_start(c + 1, R, P))
            M = fmaxf(M, a.work_ml[(((int64_t)c + h) * a.G + j) * 2]);
#pragma unroll
    for (int o = 16; o >= 1; o >>= 1) M = fmaxf(M, __shfl_xor_sync(kFull, M, o));
    if (lane == 0) wmax[warp] = M;
    __syncthreads();
#pragma unroll
    for (int w = 0; w < kCombineWarps; ++w) M = fmaxf(M, wmax[w]);

    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    float Lw = 0.f;
#pragma unroll 4
    for (int c = c0 + warp; c <= c1; c += kCombineWarps) {
        if (part_start(c, R, P) == part_start(c + 1, R, P)) continue;
        const int64_t sj = ((int64_t)c + h) * a.G + j;
        const float2 ml = *reinterpret_cast<const float2*>(a.work_ml + sj * 2);
        const float f = (ml.x == -INFINITY) ? 0.f : ex2(ml.x - M);
        Lw = fmaf(ml.y, f, Lw);
        const float4 v = *reinterpret_cast<const float4*>(a.work_o + sj * kHeadDim + 4 * lane);
        acc.x = fmaf(v.x, f, acc.x);
        acc.y = fmaf(v.y, f, acc.y);
        acc.z = fmaf(v.z, f, acc.z);
        acc.w = fmaf(v.w, f, acc.w);
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
        outp[lane] = make_float4(o.x * inv, o.y * inv, o.z * inv, o.w * inv);
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
// G <= 4: 8 lanes a row (16 dims each), 16-row tiles, 3 stages, 8 warps.
// G >= 5: 16 lanes a row (8 dims each), 8-row tiles, 5 stages, 8 warps.
#ifndef DKV_CFG_SMALL_G
#define DKV_CFG_SMALL_G 8, 16, 3, 8
#endif
#ifndef DKV_CFG_LARGE_G
#define DKV_CFG_LARGE_G 16, 8, 5, 8
#endif
template <int G>
using PKFor = typename std::conditional<(G <= 4), PK<G, DKV_CFG_SMALL_G>, PK<G, DKV_CFG_LARGE_G>>::type;

template <int G, bool FUSED>
cudaError_t launch_partial_g(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    return launch_pdl(decode_partial_kernel<PKFor<G>, FUSED>, cfg.nctas, PKFor<G>::NW * 32, cfg.smem_bytes, st, a);
}

template <int G>
cudaError_t config_g(int B, DecodeConfig* cfg)
{
    using C = PKFor<G>;
    const int smem = C::bytes(B);
    cudaError_t e = cudaFuncSetAttribute(decode_partial_kernel<C, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(decode_partial_kernel<C, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_partial_kernel<C, true>, C::NW * 32, smem)) !=
        cudaSuccess)
        return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    // The small kernels between partial launches ask for the same shared-memory
    // carve-out, so the SMs need not reconfigure L1 between launches.
    if ((e = cudaFuncSetAttribute(decode_combine_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                  cudaSharedmemCarveoutMaxShared)) != cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(advance_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                                  cudaSharedmemCarveoutMaxShared)) != cudaSuccess)
        return e;
    cfg->nctas = sms * per_sm;
    cfg->nwarps = C::NW;
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

template <bool FUSED>
cudaError_t launch_partial_any(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    switch (a.G) {
        case 1: return launch_partial_g<1, FUSED>(a, cfg, st);
        case 2: return launch_partial_g<2, FUSED>(a, cfg, st);
        case 3: return launch_partial_g<3, FUSED>(a, cfg, st);
        case 4: return launch_partial_g<4, FUSED>(a, cfg, st);
        case 5: return launch_partial_g<5, FUSED>(a, cfg, st);
        case 6: return launch_partial_g<6, FUSED>(a, cfg, st);
        case 7: return launch_partial_g<7, FUSED>(a, cfg, st);
        case 8: return launch_partial_g<8, FUSED>(a, cfg, st);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_decode_partial(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    return launch_partial_any<false>(a, cfg, st);
}

cudaError_t launch_decode_fused(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st)
{
    return launch_partial_any<true>(a, cfg, st);
}

cudaError_t launch_decode_combine(const DecodeArgs& a, cudaStream_t st)
{
    const int pairs = a.B * a.H;
    const int smem = (2 * a.B + 1) * 4 + 16 + kCombineWarps * kCombineStride * 4;
    return launch_pdl(decode_combine_kernel, pairs, kCombineWarps * 32, smem, st, a);
}

cudaError_t launch_advance(int32_t* n_app, int B, int reserve, int32_t* status, cudaStream_t st)
{
    advance_kernel<<<(B + 127) / 128, 128, 0, st>>>(n_app, B, reserve, status);
    return cudaGetLastError();
}

}  // namespace dkv
