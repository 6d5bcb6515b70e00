// Decode-step attention over the packed cache (Sec. 3.4), split-K, with both
// contractions of a tile on the tensor cores.
//
// Work split, cursor, slab segments and merges are those of the fp32 kernel
// (dkv_decode_common.cuh). What differs is the tile: 16 rows of K and V reach a
// warp's ring as four 2-D TMA boxes (16 rows x 64 dims each, 128-byte swizzle,
// so ldmatrix reads them without bank conflicts), and per tile the warp runs
//   S   = K q^T      8 x mma.sync m16n8k16 (bf16 in, fp32 accumulate): the 16
//                    rows are the M side, the G query heads of the KV head the
//                    n = 8 columns (heads G..7 are zero),
//   P   = 2^(S*scale*log2 e - m) with the lazily rescaled running max m,
//   O^T += V^T P^T   8 x 2 mma.sync: V^T via ldmatrix.trans, P^T via movmatrix;
//                    P enters as a bf16 high part plus a bf16 remainder, two
//                    products, which keeps about 16 significant bits of P.
// The query is already bf16 and K is bf16, so S is exact products summed in
// fp32, as in the fp32 kernel; only the summation order differs.
//
// The boxes read whole 16-row tiles even at the end of a segment: the rows past
// it (another slab's rows, reserve rows, or zero fill past the end of the cache)
// get score -inf and their V rows are zeroed in shared memory before use.
#include "dkv_decode_common.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

#include <math.h>

#include <mutex>
#include <type_traits>

namespace dkv {
namespace {

constexpr int kMmaTR = 16;                // rows per tile: the m16 of the score product
constexpr int kBoxBytes = kMmaTR * 128;   // one TMA box: 16 rows x 64 bf16 dims
constexpr int kMmaStage = 4 * kBoxBytes;  // K dims 0-63, K dims 64-127, V dims 0-63, V dims 64-127

template <int G_, int NT_, int NS_, int NW_>
struct MK {
    static constexpr int G = G_, NT = NT_, NS = NS_, NW = NW_, TR = kMmaTR;
    static constexpr int kStageBytes = kMmaStage;
    static_assert(PRE <= NS, "the tiles fetched before the PDL wait fit the warp's ring");
    static constexpr int kWarpRing = NS * kStageBytes;
    static constexpr int kRingBytes = NW * kWarpRing;
    static constexpr int kBarBytes = NW * NS * 8;
    static constexpr int kMetaBytes = NW * 6 * 4 + 16;  // first/last slab of each warp, their row bounds
    static constexpr int kAlign = 1024;                  // swizzle atoms are 1024-byte aligned
    static constexpr int kFixedBytes = kRingBytes + kBarBytes + kMetaBytes;
    static int bytes(int B) { return kAlign + kFixedBytes + seq_table_bytes(B); }
    static_assert(kAlign + kFixedBytes + seq_table_bytes(kMaxB) <= 227 * 1024, "fits the opt-in shared memory of one CTA");
    static_assert(8 * NT * (kHeadDim + 2) * 4 <= kWarpRing, "a warp's final state fits in its ring");
};

// Stages per warp, warps per CTA. One column tile (the decode step): more warps
// hide more of a tile's latency chain (8 dependent score MMAs, softmax, 16
// output MMAs), and at the end of a pass the CTA's (slab, column) merge tasks
// spread over more warps, which counts for G > 4 (G tasks per slab). Multi-query
// with one column tile: Q G columns give up to 8 merge tasks per slab, so 16
// warps x 1 stage (measured against 12 x 2: 7-10 % faster at Q = 2). Two column
// tiles: twice the accumulators still fit 12 warps without spills, and two
// stages hold a 16-column final state; measured against 8 warps x 3 stages,
// 2 % faster at G = 7 and 0.3 % at G = 4.
#ifndef DKV_MMA_CFG_SMALL_G
#define DKV_MMA_CFG_SMALL_G 2, 12
#endif
#ifndef DKV_MMA_CFG_LARGE_G
#define DKV_MMA_CFG_LARGE_G 1, 16
#endif
#ifndef DKV_MMA_CFG_MULTI1
#define DKV_MMA_CFG_MULTI1 1, 16
#endif
#ifndef DKV_MMA_CFG_MULTI
#define DKV_MMA_CFG_MULTI 2, 12
#endif
// Right after the wait for the previous kernel, a warp has one tile landed and
// one in flight: half its ring. The rows of its next kL2Tiles tiles are
// prefetched into L2 then, to fill the memory pipe while its first tiles are
// computed. Measured (same-box A/B, us per step): llama8b-128k 1,091 -> 1,069
// with 1 or 2 tiles (1,076 with 3, 1,081 with 4); qwen7b-64k-b4-r20 716 -> 712;
// qwen7b-64k-b4-r50 1,285 with 2 tiles, 1,277 with 1. A warp with a short range
// gains nothing and its prefetches delay the copies its first tiles wait for:
// prefetching at llama8b-32k (3-4 tiles a warp) took 466 -> 516, so only warps
// with at least kL2MinRows rows prefetch (32K: 469 -> 471, none do). The same
// prefetches issued before the wait competed with the previous kernel's
// end-of-pass merge and measured slower at every size.
constexpr int kL2Tiles = 1;
constexpr int kL2MinRows = 64;

template <int G, int NT, bool MULTI>
using MKFor = typename std::conditional<
    (NT > 1), MK<G, NT, DKV_MMA_CFG_MULTI>,
    typename std::conditional<
        MULTI, MK<G, 1, DKV_MMA_CFG_MULTI1>,
        typename std::conditional<(G <= 4), MK<G, 1, DKV_MMA_CFG_SMALL_G>,
                                  MK<G, 1, DKV_MMA_CFG_LARGE_G>>::type>::type>::type;

// ------------------------------------------------------------ PTX wrappers
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar,
                                            uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(map), "r"(x), "r"(y), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4])
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4])
{
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

// d += a b, m16n8k16, bf16 operands, fp32 accumulators.
__device__ __forceinline__ void mma16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t movm_t(uint32_t x)
{
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

// bf16 pair (lo in the low half), round to nearest even.
__device__ __forceinline__ uint32_t bf16x2(float lo, float hi)
{
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    return d;
}

// Byte offset of 16-byte chunk ch (0..7) of row r in a 128-byte-swizzled box.
__device__ __forceinline__ int swz(int r, int ch) { return r * 128 + ((ch ^ (r & 7)) << 4); }

// ------------------------------------------------------------ per-warp state
// Columns: the n side of both products, NT tiles of 8. Column c is query c / G,
// head c % G of the KV head's group (the decode step has one query: c = head).
// Lane (gid = lane / 4, t = lane % 4) holds columns 8 nt + 2t and 8 nt + 2t + 1.
template <int NT>
struct MmaState {
    float m[NT][2];     // running max of the two columns (log2 domain), the same in all gid lanes
    float l[NT][2];     // this lane's share of their softmax denominators
    float o[NT][8][4];  // O^T: [tile][dim block db][(dim 16 db + gid, col 2t), (.., 2t+1), (dim +8, 2t), (.., 2t+1)]
};

template <int NT>
__device__ __forceinline__ void state_reset(MmaState<NT>& S)
{
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        S.m[nt][0] = S.m[nt][1] = -INFINITY;
        S.l[nt][0] = S.l[nt][1] = 0.f;
#pragma unroll
        for (int db = 0; db < 8; ++db) S.o[nt][db][0] = S.o[nt][db][1] = S.o[nt][db][2] = S.o[nt][db][3] = 0.f;
    }
}

// q of the slab's columns as B fragments of the score product: for tile nt and k
// step kk (dims 16 kk .. 16 kk + 15), (column 8 nt + gid, dims 2t, 2t+1) and
// (column 8 nt + gid, dims 2t+8, 2t+9); zero past the last column.
template <int G, int NT>
__device__ __forceinline__ void load_q(const DecodeArgs& a, int b, int g, int NC, int lane, uint32_t (&qb)[NT][8][2])
{
    const int gid = lane >> 2, t = lane & 3;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const int col = 8 * nt + gid;
        const bool live = col < NC;
        const int qi = col / G, j = col - qi * G;
        const uint32_t* qr =
            reinterpret_cast<const uint32_t*>(a.q + (live ? ((int64_t)b * a.Q + qi) * a.H + g * G + j : 0) * kHeadDim);
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            qb[nt][kk][0] = live ? __ldg(qr + 8 * kk + t) : 0u;
            qb[nt][kk][1] = live ? __ldg(qr + 8 * kk + t + 4) : 0u;
        }
    }
}

// One tile: stage holds K (boxes 0, 1) and V (boxes 2, 3); rows >= cnt are not
// part of the segment (their V rows must already be zero when !FULL).
template <bool FULL, int NT>
__device__ __forceinline__ void mma_tile(MmaState<NT>& S, const uint32_t (&qb)[NT][8][2], uint32_t stage, int cnt,
                                         float cs, int lane)
{
    const int gid = lane >> 2;
    // Scores: ldmatrix lane -> (row, chunk) of the A fragment: rows 0-7 / 8-15 by
    // bit 3 of the lane, chunk +0 / +1 by bit 4. One K fragment serves all tiles.
    const int ar = (lane & 7) + (lane & 8), ac = lane >> 4;
    float c[NT][4];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) c[nt][0] = c[nt][1] = c[nt][2] = c[nt][3] = 0.f;
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
        uint32_t af[4];
        ldsm_x4(stage + (kk >> 2) * kBoxBytes + swz(ar, (kk & 3) * 2 + ac), af);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma16816(c[nt], af, qb[nt][kk][0], qb[nt][kk][1]);
    }
    uint32_t bh0[NT], bh1[NT], bl0[NT], bl1[NT];
    // c: (row gid, columns 2t, 2t+1), (row gid + 8, columns 2t, 2t+1). Lazy
    // rescaling as in the fp32 kernel: a column's running max only moves when a
    // score tops it by more than kSlack.
    float s[NT][4];
    bool over = false;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
        for (int i = 0; i < 4; ++i) s[nt][i] = c[nt][i] * cs;
        if (!FULL) {
            if (gid >= cnt) s[nt][0] = s[nt][1] = -INFINITY;
            if (gid + 8 >= cnt) s[nt][2] = s[nt][3] = -INFINITY;
        }
        over |= fmaxf(s[nt][0], s[nt][2]) > S.m[nt][0] + kSlack || fmaxf(s[nt][1], s[nt][3]) > S.m[nt][1] + kSlack;
    }
    if (__any_sync(kFull, over)) {
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            float y0 = fmaxf(s[nt][0], s[nt][2]), y1 = fmaxf(s[nt][1], s[nt][3]);
#pragma unroll
            for (int o = 4; o <= 16; o <<= 1) {
                y0 = fmaxf(y0, __shfl_xor_sync(kFull, y0, o));
                y1 = fmaxf(y1, __shfl_xor_sync(kFull, y1, o));
            }
            const float mn0 = fmaxf(S.m[nt][0], y0), mn1 = fmaxf(S.m[nt][1], y1);
            const float al0 = (mn0 == -INFINITY) ? 1.f : ex2(S.m[nt][0] - mn0);
            const float al1 = (mn1 == -INFINITY) ? 1.f : ex2(S.m[nt][1] - mn1);
            S.l[nt][0] *= al0;
            S.l[nt][1] *= al1;
#pragma unroll
            for (int db = 0; db < 8; ++db) {
                S.o[nt][db][0] *= al0;
                S.o[nt][db][1] *= al1;
                S.o[nt][db][2] *= al0;
                S.o[nt][db][3] *= al1;
            }
            S.m[nt][0] = mn0;
            S.m[nt][1] = mn1;
        }
    }
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        const float r0 = (S.m[nt][0] == -INFINITY) ? 0.f : S.m[nt][0];
        const float r1 = (S.m[nt][1] == -INFINITY) ? 0.f : S.m[nt][1];
        const float p0 = ex2(s[nt][0] - r0), p1 = ex2(s[nt][1] - r1);  // 2^-inf = 0
        const float p2 = ex2(s[nt][2] - r0), p3 = ex2(s[nt][3] - r1);
        S.l[nt][0] += p0 + p2;
        S.l[nt][1] += p1 + p3;
        // P^T as B fragments: bf16 high part and remainder, transposed by movmatrix
        // from (row, column pair) to (row pair, column).
        const uint32_t h01 = bf16x2(p0, p1), h23 = bf16x2(p2, p3);
        const uint32_t l01 = bf16x2(p0 - __uint_as_float(h01 << 16), p1 - __uint_as_float(h01 & 0xffff0000u));
        const uint32_t l23 = bf16x2(p2 - __uint_as_float(h23 << 16), p3 - __uint_as_float(h23 & 0xffff0000u));
        bh0[nt] = movm_t(h01);
        bh1[nt] = movm_t(h23);
        bl0[nt] = movm_t(l01);
        bl1[nt] = movm_t(l23);
    }
    // O^T += V^T P^T: ldmatrix.trans lane -> (row, chunk): rows 0-7 / 8-15 by
    // bit 4 of the lane, chunk +0 / +1 by bit 3. One V fragment serves all tiles.
    const int vr = (lane & 7) + ((lane >> 4) << 3), vc = (lane >> 3) & 1;
    const uint32_t vt = stage + 2 * kBoxBytes;
#pragma unroll
    for (int db = 0; db < 8; ++db) {
        uint32_t af[4];
        ldsm_x4_t(vt + (db >> 2) * kBoxBytes + swz(vr, (db & 3) * 2 + vc), af);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
            mma16816(S.o[nt][db], af, bh0[nt], bh1[nt]);
            mma16816(S.o[nt][db], af, bl0[nt], bl1[nt]);
        }
    }
}

// Softmax denominators of the lane's columns, summed over the gid lanes.
template <int NT>
__device__ __forceinline__ void finish_l(const MmaState<NT>& S, float (&l2)[NT][2])
{
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
        float a = S.l[nt][0], b = S.l[nt][1];
#pragma unroll
        for (int o = 4; o <= 16; o <<= 1) {
            a += __shfl_xor_sync(kFull, a, o);
            b += __shfl_xor_sync(kFull, b, o);
        }
        l2[nt][0] = a;
        l2[nt][1] = b;
    }
}

// The state as a record: o[NC][128] at o_dst, (m, l)[NC] at ml_dst.
template <int NT>
__device__ __forceinline__ void store_mma_state(const MmaState<NT>& S, const float (&l2)[NT][2], float* o_dst,
                                                float* ml_dst, int NC, int lane)
{
    const int gid = lane >> 2, t = lane & 3;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int j = 8 * nt + 2 * t + q;
            if (j < NC) {
#pragma unroll
                for (int db = 0; db < 8; ++db) {
                    o_dst[j * kHeadDim + 16 * db + gid] = S.o[nt][db][q];
                    o_dst[j * kHeadDim + 16 * db + gid + 8] = S.o[nt][db][2 + q];
                }
                if (gid == 0) *reinterpret_cast<float2*>(ml_dst + 2 * j) = make_float2(S.m[nt][q], l2[nt][q]);
            }
        }
}

// Final answer of a slab held by one warp: out = o / l for every column.
template <int G, int NT>
__device__ __forceinline__ void write_mma_out(const DecodeArgs& a, const MmaState<NT>& S, const float (&l2)[NT][2],
                                              int b, int g, int NC, int lane)
{
    const int gid = lane >> 2, t = lane & 3;
#pragma unroll
    for (int nt = 0; nt < NT; ++nt)
#pragma unroll
        for (int q = 0; q < 2; ++q) {
            const int j = 8 * nt + 2 * t + q;
            if (j < NC) {
                const float inv = l2[nt][q] > 0.f ? 1.f / l2[nt][q] : 0.f;
                float* dst = a.out + out_row<G>(a, b, g, j) * kHeadDim;
#pragma unroll
                for (int db = 0; db < 8; ++db) {
                    dst[16 * db + gid] = S.o[nt][db][q] * inv;
                    dst[16 * db + gid + 8] = S.o[nt][db][2 + q] * inv;
                }
            }
        }
}

// ------------------------------------------------------------ kernel
// MULTI: columns are Q x G with Q from the arguments (multi-query); otherwise
// the G heads of the decode step, fixed at compile time.
template <int G, int NT, bool FUSED, bool MULTI>
__global__ void __launch_bounds__(MKFor<G, NT, MULTI>::NW * 32, 1)
    decode_mma_kernel(const __grid_constant__ DecodeArgs a, const __grid_constant__ CacheMaps maps)
{
    using C = MKFor<G, NT, MULTI>;
    constexpr int NCC = MULTI ? 0 : G;
    const int NC = MULTI ? a.NC : G;
    constexpr int TR = C::TR, NS = C::NS, NW = C::NW;
    extern __shared__ __align__(128) unsigned char smem_raw[];
    // The ring starts on a 1024-byte boundary (the swizzle pattern's period).
    unsigned char* smem = smem_raw + ((C::kAlign - (smem_u32(smem_raw) & (C::kAlign - 1))) & (C::kAlign - 1));
    const SeqTable tab = seq_table_at(smem + C::kFixedBytes, a);
    int32_t* seg_first = reinterpret_cast<int32_t*>(smem + C::kRingBytes + C::kBarBytes);
    int32_t* seg_last = seg_first + NW;
    int32_t* seg_p0 = seg_first + 2 * NW;  // [2 NW] layer rows [p0, p1) of entry 2 w (first) / 2 w + 1 (last)
    int32_t* seg_p1 = seg_first + 4 * NW;

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int NHl = a.B * a.Hkv;
    const int c = blockIdx.x;
    uint64_t* my_bars = reinterpret_cast<uint64_t*>(smem + C::kRingBytes) + warp * NS;

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
                for (int j = 0; j < NC; ++j)
                    write_out<G>(a, h / a.Hkv, h % a.Hkv, j, make_float4(0.f, 0.f, 0.f, 0.f), 0.f, lane);
    }
    const int A = part_start(c, R, a.nctas), Bc = part_start(c + 1, R, a.nctas);
    if (A >= Bc) return;  // uniform: this CTA has no rows
    const int wA = A + (int)(((int64_t)(Bc - A) * warp) / NW);
    const int wB = A + (int)(((int64_t)(Bc - A) * (warp + 1)) / NW);
    unsigned char* my_ring = smem + warp * C::kWarpRing;
    MmaState<NT> S;
    float l2[NT][2];
    bool have_last = false;  // S holds the state of this warp's last slab

    if (wA < wB) {
        const int hfirst = slab_containing(a, tab, NHl, wA);
        const int hlast = slab_containing(a, tab, NHl, wB - 1);
        const int hend = hlast + 1;
        const uint64_t pol = evict_first_policy();

        Cursor ld;
        ld.h = hfirst;
        cursor_seek(ld, a, tab, hend, wA, wB);
        Cursor cp = ld;

        // Whole 16-row boxes from the tile's first cache row; the rows past the
        // segment are masked later. (The new token's row is read too and then
        // overwritten in shared memory from k_new / v_new.)
        auto issue = [&](const Cursor& cu, int stage) {
            const int row = (int)(cu.base + (cu.x - cu.p0));
            // Bounds-checked build: the tile's rows lie in the cache (a TMA box past
            // the end reads zeros, so the copy itself stays in bounds either way).
            in_bounds(row >= 0 && (a.rows_cap == 0 || row + min(C::TR, cu.s1 - cu.x) <= a.rows_cap), a.status);
            const uint32_t bar = smem_u32(&my_bars[stage]);
            const uint32_t dst = smem_u32(my_ring + stage * C::kStageBytes);
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(bar, C::kStageBytes);
            tma_load_2d(dst, &maps.k, 0, row, bar, pol);
            tma_load_2d(dst + kBoxBytes, &maps.k, 64, row, bar, pol);
            tma_load_2d(dst + 2 * kBoxBytes, &maps.v, 0, row, bar, pol);
            tma_load_2d(dst + 3 * kBoxBytes, &maps.v, 64, row, bar, pol);
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
        if (lane == 0 && wB - wA >= kL2MinRows) {
            // The next tiles' K and V rows into L2: exactly the segment's rows, all in the cache.
            Cursor it = ld;
            for (int s = 0; s < kL2Tiles && it.h < hend; ++s) {
                const int cnt = min(TR, it.s1 - it.x);
                const int64_t row = it.base + (it.x - it.p0);
                prefetch_l2_bulk(a.Kc + row * kHeadDim, (uint32_t)cnt * kRowBytes);
                prefetch_l2_bulk(a.Vc + row * kHeadDim, (uint32_t)cnt * kRowBytes);
                cursor_next<TR>(it, a, tab, hend, wA, wB);
            }
        }
        int stage = 0;
        uint32_t phase = 0;
        const float cs = a.qscale;  // softmax scale * log2(e)

        while (cp.h < hend && !dead) {
            const int h = cp.h;
            const int p0h = cp.p0, p1h = cp.p0 + cp.n_h;  // the slab's layer rows
            const int b = h / a.Hkv, g = h - b * a.Hkv;
            uint32_t qb[NT][8][2];
            load_q<G, NT>(a, b, g, NC, lane, qb);
            state_reset(S);

            while (cp.h == h) {
                const int cnt = min(TR, cp.s1 - cp.x);
                const int r0 = cp.x - cp.p0;
                unsigned char* st = my_ring + stage * C::kStageBytes;
                // Every lane observes the completed phase itself (acquire) before reading.
                if (!__all_sync(kFull, mbar_wait(smem_u32(&my_bars[stage]), phase))) {
                    dead = true;
                    if (lane == 0) atomicOr(a.status, 0x2 /* DKV_DEV_TMA_TIMEOUT */);
                    break;
                }
                --inflight;
                bool touched = false;
                if (cp.app && r0 + cnt == cp.n_h) {
                    // This step's token: into the tile from k_new/v_new, and into the
                    // slab's next free row for later steps.
                    const int kv = lane >> 4, sub = lane & 15;
                    const uint16_t* src = (kv ? a.v_new : a.k_new) + ((int64_t)b * a.Hkv + g) * kHeadDim;
                    const uint4 v = __ldg(reinterpret_cast<const uint4*>(src) + sub);
                    *reinterpret_cast<uint4*>(st + (2 * kv + (sub >> 3)) * kBoxBytes + swz(cnt - 1, sub & 7)) = v;
                    const int64_t nrow = cp.base + (cp.n_h - 1);
                    if (in_bounds(nrow >= 0 && (a.rows_cap == 0 || nrow < a.rows_cap), a.status)) {
                        uint16_t* dstg = (kv ? a.Vc : a.Kc) + nrow * kHeadDim;
                        *(reinterpret_cast<uint4*>(dstg) + sub) = v;
                    }
                    touched = true;
                }
                if (cnt < TR) {
                    // V rows past the segment: zeros (their p is 0, but 0 * inf or
                    // 0 * nan would not be).
                    for (int k = lane; k < (TR - cnt) * 16; k += 32) {
                        const int row = cnt + (k >> 4), sub = k & 15;
                        *reinterpret_cast<uint4*>(st + (2 + (sub >> 3)) * kBoxBytes + swz(row, sub & 7)) =
                            make_uint4(0u, 0u, 0u, 0u);
                    }
                    touched = true;
                }
                if (touched) {
                    fence_proxy_async_smem();  // order these generic writes before later bulk copies
                    __syncwarp();
                }
                if (cnt == TR)
                    mma_tile<true, NT>(S, qb, smem_u32(st), cnt, cs, lane);
                else
                    mma_tile<false, NT>(S, qb, smem_u32(st), cnt, cs, lane);
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
            finish_l(S, l2);
            if (h == hlast) {
                have_last = true;  // merged with the other warps at the end
                if (lane == 0) {
                    seg_last[warp] = h;
                    seg_p0[2 * warp + 1] = p0h;
                    seg_p1[2 * warp + 1] = p1h;
                }
            } else if (h == hfirst) {
                const int64_t rec = (int64_t)c * NW + warp;  // this slab continues in an earlier warp
                store_mma_state<NT>(S, l2, a.warp_o + rec * NC * kHeadDim, a.warp_ml + rec * NC * 2, NC, lane);
                if (lane == 0) {
                    seg_first[warp] = h;
                    seg_p0[2 * warp] = p0h;
                    seg_p1[2 * warp] = p1h;
                }
            } else if (FUSED) {
                write_mma_out<G, NT>(a, S, l2, b, g, NC, lane);  // the whole slab lies in this warp's range
            } else {
                const int64_t slot = (int64_t)c + h;  // the whole slab lies in this warp's range
                store_mma_state<NT>(S, l2, a.work_o + slot * NC * kHeadDim, a.work_ml + slot * NC * 2, NC, lane);
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
    // final state goes there. Then the CTA merges, all warps sharing the work.
    __syncwarp();
    if (have_last)
        store_mma_state<NT>(S, l2, reinterpret_cast<float*>(my_ring), reinterpret_cast<float*>(my_ring) + NC * kHeadDim,
                            NC, lane);
    __syncthreads();
    pdl_wait();  // the merges write the workspace and out: the previous kernel must be done with them
    cta_tail<G, NW, FUSED, NCC>(a, smem, C::kWarpRing, seg_first, c, R, warp, lane);
}

template <int G, int NT, bool FUSED, bool MULTI>
cudaError_t launch_mma_g(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg, cudaStream_t st)
{
    using C = MKFor<G, NT, MULTI>;
    // The configuration must be this kernel's: its warps and shared-memory layout;
    // the grid is the call's CTA count (at most the configuration's).
    if (cfg.nwarps != C::NW || cfg.smem_bytes < C::bytes(a.B) || a.nctas < 1 || a.nctas > cfg.nctas)
        return cudaErrorInvalidConfiguration;
    return launch_pdl(decode_mma_kernel<G, NT, FUSED, MULTI>, a.nctas, C::NW * 32, cfg.smem_bytes, st, a, maps);
}

// Launch configuration of the tensor-core kernels of one kind: the decode step
// (NT = 1, partial and fused), or multi-query with NT column tiles (fused only).
template <int G, int NT, bool MULTI>
cudaError_t config_mma_g(int B, DecodeConfig* cfg)
{
    using C = MKFor<G, NT, MULTI>;
    const int smem = C::bytes(B);
    cudaError_t e;
    if constexpr (!MULTI) {
        if ((e = cudaFuncSetAttribute(decode_mma_kernel<G, NT, false, false>,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, smem)) != cudaSuccess)
            return e;
    }
    if ((e = cudaFuncSetAttribute(decode_mma_kernel<G, NT, true, MULTI>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  smem)) != cudaSuccess)
        return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_mma_kernel<G, NT, true, MULTI>, C::NW * 32,
                                                           smem)) != cudaSuccess)
        return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    cfg->nctas = sms * per_sm;
    cfg->nwarps = C::NW;
    cfg->smem_bytes = smem;
    return cudaSuccess;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static std::once_flag once;
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

}  // namespace

cudaError_t make_cache_maps(const void* Kc, const void* Vc, int64_t rows, CacheMaps* maps, bool short_boxes,
                            int box_rows)
{
    if (box_rows < 8 || box_rows > 256 || (box_rows & 7)) return cudaErrorInvalidValue;
    if (rows < 1 || rows > kMaxMmaRows) return cudaErrorInvalidValue;
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    const cuuint64_t dim[2] = {(cuuint64_t)kHeadDim, (cuuint64_t)rows};
    const cuuint64_t stride[1] = {(cuuint64_t)kRowBytes};
    // short_boxes (fault injection): 8-row boxes deliver half the bytes each
    // stage's mbarrier expects, inside the stage, so every wait runs out.
    const cuuint32_t box[2] = {64, (cuuint32_t)(short_boxes ? box_rows / 2 : box_rows)};
    const cuuint32_t elem[2] = {1, 1};
    const void* base[2] = {Kc, Vc};
    CUtensorMap* out[2] = {&maps->k, &maps->v};
    for (int i = 0; i < 2; ++i)
        if (enc(out[i], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base[i]), dim, stride, box, elem,
                CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
            return cudaErrorInvalidValue;
    return cudaSuccess;
}

cudaError_t decode_config_mma(int G, int B, int kind, DecodeConfig* cfg)
{
    if (B < 1 || B > kMaxB || kind < 0 || kind > 2) return cudaErrorInvalidValue;
#define DKV_CFG_CASE(g)                                                               \
    case g:                                                                           \
        return kind == 0 ? config_mma_g<g, 1, false>(B, cfg)                          \
                         : (kind == 1 ? config_mma_g<g, 1, true>(B, cfg) : config_mma_g<g, 2, true>(B, cfg));
    switch (G) {
        DKV_CFG_CASE(1)
        DKV_CFG_CASE(2)
        DKV_CFG_CASE(3)
        DKV_CFG_CASE(4)
        DKV_CFG_CASE(5)
        DKV_CFG_CASE(6)
        DKV_CFG_CASE(7)
        DKV_CFG_CASE(8)
        default: return cudaErrorInvalidValue;
    }
#undef DKV_CFG_CASE
}

template <bool FUSED>
static cudaError_t launch_mma_any(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg, cudaStream_t st)
{
    // The decode step (Q = 1) takes the kernels with the G columns fixed at
    // compile time; multi-query calls the fused ones with one or two column tiles.
    const bool multi = a.Q > 1, two = a.NC > 8;
    if (multi && !FUSED) return cudaErrorInvalidValue;
#define DKV_LAUNCH_CASE(g)                                                                        \
    case g:                                                                                       \
        return !multi ? launch_mma_g<g, 1, FUSED, false>(a, maps, cfg, st)                        \
                      : (two ? launch_mma_g<g, 2, true, true>(a, maps, cfg, st)                   \
                             : launch_mma_g<g, 1, true, true>(a, maps, cfg, st));
    switch (a.G) {
        DKV_LAUNCH_CASE(1)
        DKV_LAUNCH_CASE(2)
        DKV_LAUNCH_CASE(3)
        DKV_LAUNCH_CASE(4)
        DKV_LAUNCH_CASE(5)
        DKV_LAUNCH_CASE(6)
        DKV_LAUNCH_CASE(7)
        DKV_LAUNCH_CASE(8)
        default: return cudaErrorInvalidValue;
    }
#undef DKV_LAUNCH_CASE
}

cudaError_t launch_decode_mma_partial(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg,
                                      cudaStream_t st)
{
    return launch_mma_any<false>(a, maps, cfg, st);
}

cudaError_t launch_decode_mma_fused(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg,
                                    cudaStream_t st)
{
    return launch_mma_any<true>(a, maps, cfg, st);
}

}  // namespace dkv
