// Multi-query decode over the packed cache (Sec. 3.4; shared-context reuse,
// Sec. 4.1) on the fifth-generation tensor cores: tcgen05.mma with operands in
// shared memory and accumulators in tensor memory (TMEM), for 17 to 64 columns
// (queries x heads of a KV head's group) per slab.
//
// Work split: the layer's rows (every slab end to end, plus the rows appended in
// earlier steps) are cut into contiguous CTA ranges (one CTA per SM, a
// cooperative launch, so every CTA is resident at once): whole numbers of CTAs
// per slab while the slabs are few (TcPart below), else equal ranges as in the
// other decode kernels. A CTA walks its range in tiles of 64 rows, slab segment
// by slab segment (a segment: the part of one slab inside the CTA's range).
//
//   warp 0 (one lane)   TMA: a tile's K rows and V rows, each as 16-row 2-D
//                       boxes (64 dims, 128-byte swizzle; measured faster than
//                       64- or 32-row boxes), into separate
//                       rings (4 K stages, 5 V stages): a K stage is released as
//                       soon as its score product is done, a V stage only after
//                       its output product, so V is the deeper ring.
//   warp 1 (one lane)   MMA: S^T = Q K^T  (M = 64 query-column rows of Q, zero
//                       past the last column, N = 64 cache rows, K = 128 dims;
//                       8 MMAs) into one of four TMEM score buffers, running up
//                       to four tiles ahead of O^T += V^T P  (M = 128 dims, N =
//                       the columns rounded up to 16, K = 64 rows; V^T read
//                       MN-major from its stage; P as a bf16 high part and
//                       remainder side by side, N = 2 x the columns, one MMA per
//                       k-step) into the TMEM output accumulator of the tile's
//                       softmax group, whose two halves are summed when read.
//                       Output products go first; a group announces its P only
//                       once the tile's V stage has landed, so that is the one
//                       barrier the lane tests for them.
//   warps 2-5, 6-9      two softmax groups; group g takes the tiles t with
//                       t % 2 == g, with its own running max and sum of every
//                       column and its own O accumulator (merged at a segment's
//                       end). With M = 64, row c of S^T (column c) sits in TMEM
//                       lane 32 (c / 16) + c % 16; a 16x32bx2 TMEM load gives
//                       lanes l and l + 16 of warp (group, quarter) column
//                       16 quarter + l, rows 0-31 and 32-63 of the tile: tile
//                       max (one shuffle joins the halves), lazily rescaled
//                       running max (a column's max moves only when a score
//                       tops it by kSlackTc; O is then rescaled in TMEM),
//                       P = 2^(s - m) written to shared memory
//                       as the B operand of the output product, V rows past a
//                       segment zeroed. For O, thread (quarter, lane) owns
//                       dimension 32 quarter + lane (TMEM lane).
//
// Segments alternate between two Q buffers, each loaded two segments ahead, so
// the score products run on across a slab boundary.
//
// A slab wholly inside one CTA is written out at its segment's end. Otherwise
// each CTA of the slab writes its partial (m, l, o of every column) and counts
// itself in; once the CTA's range is done it waits (bounded) until all the
// slab's CTAs have counted in, then merges its share of the slab's columns
// (CTA k of the slab's nct CTAs takes columns k NC / nct .. (k+1) NC / nct):
// the merge is spread over the slab's CTAs instead of falling on the last one.
//
// Every wait is bounded (polls and 2 s). A wait that runs out sets a
// DKV_DEV_* bit, the roles stop (the softmax groups keep walking the tiles,
// without work, so that they still meet at every named barrier), the copies and
// products in flight are drained with the same bound, and TMEM is freed before
// the CTA exits.
#include "dkv_decode_common.cuh"

#include <cuda.h>

#include <math.h>

namespace dkv {
namespace {

constexpr int kTcRows = 64;                    // cache rows per tile
constexpr int kKStages = 4;                    // K ring stages
constexpr int kVStages = 5;                    // V ring stages
constexpr int kTcBox = kTcRows * 128;          // one 64-dim half of a tile: 64 rows x 64 dims of bf16 (8 KB)
constexpr int kTcBoxRows = 16;                 // rows of one TMA box (measured: 16-row boxes beat 64- and 32-row ones)
constexpr int kTcHalfTile = 2 * kTcBox;        // K (or V) rows of one tile: dims 0-63, then 64-127
constexpr int kTcThreads = 320;                // warps: 0 TMA, 1 MMA, 2-5 and 6-9 the two softmax groups
constexpr int kTcSoft = 256;                   // threads of the softmax warps
constexpr int kTcGroup = 128;                  // threads of one softmax group
constexpr int kTcQRows = 64;                   // M of the score product: the most columns
constexpr int kTcQHalf = kTcQRows * 128;       // one 64-dim half of Q (8 KB)
constexpr int kTcQBytes = 2 * kTcQHalf;        // Q as the A operand: 64 rows x 128 dims (two buffers: segments alternate)
constexpr int kTcPBytes = 2 * kTcMaxCols * 128;  // one P buffer: high parts (rows 0..NCpad-1), then low parts, 64 rows each
constexpr int kSBufs = 4;                      // TMEM score buffers
static_assert((kKStages & (kKStages - 1)) == 0 && (kSBufs & (kSBufs - 1)) == 0, "indexed by masks");
constexpr int kTcTmemCols = 512;               // S buffers at columns 0, 64, 128, 192; O of group g at 256 + 128 g
constexpr int kTcOCols = 2 * kTcMaxCols;       // O of one group: the product with P's high parts, then with its low parts
constexpr int kTcOCol = kSBufs * kTcRows;
// Named barriers: 1 + g for softmax group g, kBarSoft for both groups, kBarTmem for warps 1-9.
constexpr int kBarSoft = 3, kBarTmem = 4;

// Shared-memory layout, from a 1024-byte aligned base.
constexpr int kOffK = 0;
constexpr int kOffV = kOffK + kKStages * kTcHalfTile;
constexpr int kOffQ = kOffV + kVStages * kTcHalfTile;
constexpr int kOffP = kOffQ + 2 * kTcQBytes;
constexpr int kOffStats = kOffP + 2 * kTcPBytes;           // per group: max [2][64], sum [2][64], alpha [2][64] (floats)
constexpr int kOffFlags = kOffStats + 6 * kTcMaxCols * 4;  // int[kNumFlags]
constexpr int kOffBars = kOffFlags + 24 * 4;               // uint64 barriers
// k_full[K], k_empty[K], v_full[V], v_empty[V], s_full[4], p_full[2], o_done[2], q_full[2], fin
constexpr int kNumBars = 2 * kKStages + 2 * kVStages + kSBufs + 7;
constexpr int kOffTmem = kOffBars + kNumBars * 8;
constexpr int kOffTable = (kOffTmem + 16 + 15) / 16 * 16;
constexpr int kTcAlign = 1024;
__host__ __device__ constexpr int tc_smem_bytes(int B) { return kTcAlign + kOffTable + seq_table_bytes(B); }
static_assert(tc_smem_bytes(kMaxB) <= 227 * 1024, "fits the opt-in shared memory of one CTA");

// Flag slots.
constexpr int kFlagVote = 0;      // [2][4] per-warp rescale votes of each softmax group
constexpr int kFlagAbort = 8;     // a bounded wait ran out
constexpr int kFlagOk = 9;        // [2] result of a group leader's wait, for its group (10: group 1)
constexpr int kFlagSegOk = 11;    // no wait ran out before a segment's end (for both groups)
constexpr int kFlagKIssued = 12;  // K tiles the TMA lane issued
constexpr int kFlagVIssued = 13;  // V tiles the TMA lane issued
constexpr int kFlagMmaLast = 14;  // the MMA lane issued products (fin must be awaited before freeing TMEM)
constexpr int kFlagOk2 = 16;      // [2] result of a group leader's second wait of a tile (17: group 1)
constexpr int kNumFlags = 24;

// Lazy-rescale threshold of the running max (log2 units): P stays below 2^32,
// far inside fp32 and bf16 range, and a rescale of O in TMEM (a load, multiply
// and store of every column) is rare even with outlier keys.
constexpr float kSlackTc = 32.f;

// Device status bits (include/dkv.h).
constexpr int kDevTmaTimeout = 0x2, kDevMergeTimeout = 0x4;

// ------------------------------------------------------------ tcgen05 wrappers
// Shared-memory matrix descriptor: start address, leading and stride byte
// offsets (16-byte units), descriptor version 1, 128-byte swizzle.
__device__ __forceinline__ uint64_t sdesc(uint32_t addr, uint32_t lbo, uint32_t sbo)
{
    return (uint64_t)((addr >> 4) & 0x3fff) | ((uint64_t)((lbo >> 4) & 0x3fff) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3fff) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// Instruction descriptor of kind::f16: fp32 accumulate, bf16 A and B, the
// operands' major-ness (0: K-major, 1: MN-major), N and M.
__device__ __forceinline__ uint32_t idesc(int M, int N, int a_mn, int b_mn)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)a_mn << 15) | ((uint32_t)b_mn << 16) |
           ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t id, uint32_t acc)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(id), "r"(acc)
        : "memory");
}

// The mbarrier arrives once every product issued so far by this thread is done.
__device__ __forceinline__ void umma_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive TMEM columns of this thread's lane (warp w reads lanes 32 (w % 4) ..).
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 TMEM lanes from taddr: lanes 0-15 of the warp read columns [col, col + 32),
// lanes 16-31 the same TMEM lanes at columns [col + 32, col + 64).
__device__ __forceinline__ void tmem_ld16x2(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.16x32bx2.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32], 32;"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// 16 consecutive TMEM columns of this thread's lane, without the wait: the
// registers are valid only after tmem_wait_ld, which takes them as operands so
// that no use of them can be scheduled before it.
__device__ __forceinline__ void tmem_ld16_async(uint32_t taddr, uint32_t (&r)[16])
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_fence_regs(uint32_t (&r)[16])
{
    asm volatile(""
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]), "+r"(r[6]), "+r"(r[7]),
                   "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]), "+r"(r[12]), "+r"(r[13]), "+r"(r[14]),
                   "+r"(r[15]));
}

__device__ __forceinline__ void tmem_wait_ld(uint32_t (&a)[16], uint32_t (&b)[16], uint32_t (&c)[16],
                                             uint32_t (&d)[16])
{
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
    tmem_fence_regs(a);
    tmem_fence_regs(b);
    tmem_fence_regs(c);
    tmem_fence_regs(d);
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32])
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]), "f"(v[8]),
        "f"(v[9]), "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]), "f"(v[15]), "f"(v[16]),
        "f"(v[17]), "f"(v[18]), "f"(v[19]), "f"(v[20]), "f"(v[21]), "f"(v[22]), "f"(v[23]), "f"(v[24]),
        "f"(v[25]), "f"(v[26]), "f"(v[27]), "f"(v[28]), "f"(v[29]), "f"(v[30]), "f"(v[31])
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void named_sync(int id, int n) { asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(n) : "memory"); }

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void tma_box(uint32_t dst, const CUtensorMap* map, int x, int y, uint32_t bar, uint64_t pol)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(dst),
        "l"(map), "r"(x), "r"(y), "r"(bar), "l"(pol)
        : "memory");
}

// Byte offset of 16-byte chunk ch (0..7) of 128-byte row r in a 128-byte-swizzled tile.
__device__ __forceinline__ int sw128(int r, int ch) { return r * 128 + ((ch ^ (r & 7)) << 4); }

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    return d;
}

// Bounded wait by one thread; true when the phase completed.
__device__ __forceinline__ bool wait_phase(uint64_t* bar, uint32_t parity) { return mbar_wait(smem_u32(bar), parity); }
// One poll that never suspends the thread (mbarrier.try_wait may suspend it for a
// system-defined time while the phase is incomplete, which would stall the
// schedulers below on one stage while another is ready).
__device__ __forceinline__ bool test_phase(uint64_t* bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    return ok != 0;
}

// ------------------------------------------------------------ tiles
// The CTA's tiles, slab segment by slab segment; tiles are 64 rows from the
// segment's start.
struct TileWalk {
    Cursor cu;
    int hend, A, B;
    __device__ void begin(const DecodeArgs& a, const SeqTable& t, int hfirst, int hend_, int A_, int B_)
    {
        hend = hend_;
        A = A_;
        B = B_;
        cu.h = hfirst;
        cursor_seek(cu, a, t, hend, A, B);
    }
    __device__ bool more() const { return cu.h < hend; }
    __device__ int cnt() const { return min(kTcRows, cu.s1 - cu.x); }
    __device__ bool first() const { return cu.x == cu.s0; }
    __device__ bool last() const { return cu.x + kTcRows >= cu.s1; }
    __device__ int cache_row() const { return (int)(cu.base + (cu.x - cu.p0)); }
    __device__ void next(const DecodeArgs& a, const SeqTable& t) { cursor_next<kTcRows>(cu, a, t, hend, A, B); }
};

// Slab of the segment `skip` segments after the one under `cu` (>= hend when
// there is none).
__device__ __forceinline__ int later_segment_slab(Cursor cu, const DecodeArgs& a, const SeqTable& t, int hend, int A,
                                                  int B, int skip)
{
    for (int k = 0; k < skip && cu.h < hend; ++k) {
        ++cu.h;
        cursor_seek(cu, a, t, hend, A, B);
    }
    return cu.h;
}

// Q of slab h as the A operand: row c (column c: query c / G, head g G + c % G)
// of 128 bf16 dims, two 64-dim halves, 128-byte swizzle; rows NC.. are zero.
template <int G>
__device__ void load_q_tc(const DecodeArgs& a, int h, unsigned char* sQ, int tid)
{
    const int b = h / a.Hkv, g = h - b * a.Hkv;
    for (int i = tid; i < kTcQRows * 16; i += kTcSoft) {
        const int c = i >> 4, ch = i & 15;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (c < a.NC) {
            const int qi = c / G, j = c - qi * G;
            const uint4* src = reinterpret_cast<const uint4*>(a.q + (((int64_t)b * a.Q + qi) * a.H + g * G + j) * kHeadDim);
            v = __ldg(src + ch);
        }
        *reinterpret_cast<uint4*>(sQ + (ch >> 3) * kTcQHalf + sw128(c, ch & 7)) = v;
    }
}

// Idle polling of the TMA and MMA lanes is bounded like every wait: kWaitSpins
// polls without progress or kWaitNs of globaltimer.
struct IdleBound {
    int spins = 0;
    unsigned long long t0 = 0;
    __device__ void progress() { spins = 0; }
    __device__ bool expired()
    {
        if (spins == 0) t0 = global_ns();
        ++spins;
        return spins >= kWaitSpins || ((spins & 63) == 0 && global_ns() - t0 > kWaitNs);
    }
};

// Row partition of a layer over the CTAs. A CTA whose range holds a slab
// boundary drains its pipeline at that segment's end (~5 us), and the slab's
// merge waits for it. So while the slabs are few (at most a quarter as many as
// the CTAs) and the rounding keeps every CTA within 1.15 shares of rows, each
// slab gets a whole number of CTAs, cb(h+1) - cb(h) with cb(h) = round(P S_h / R)
// (S_h: the slab's first row), and splits its rows evenly over them. An empty
// slab gets no CTA and lies inside the CTA that starts the next one. Otherwise
// the rows are cut into P equal ranges, as in the other decode kernels. Every
// CTA evaluates the same float expressions, so all agree on the partition.
struct TcPart {
    bool aligned;
    int R, P, NHl;
    float scale;  // P / R
    __device__ int cb(const DecodeArgs& a, const SeqTable& t, int h) const
    {
        if (h >= NHl) return P;
        return min(P, (int)floorf(fmaf((float)slab_start(a, t, h), scale, 0.5f)));
    }
    // First row of CTA c (c <= P).
    __device__ int start(const DecodeArgs& a, const SeqTable& t, int c) const
    {
        if (!aligned) return part_start(c, R, P);
        if (c >= P) return R;
        int lo = 0, hi = NHl - 1;  // home slab: the first h with cb(h + 1) > c
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (cb(a, t, mid + 1) > c)
                hi = mid;
            else
                lo = mid + 1;
        }
        const int f = lo, cf = cb(a, t, f);
        if (c == cf) {  // the first CTA of slab f also takes the slabs before it that got no CTA
            int l2 = 0, h2 = f;
            while (l2 < h2) {
                const int mid = (l2 + h2) >> 1;
                if (cb(a, t, mid) >= c)
                    h2 = mid;
                else
                    l2 = mid + 1;
            }
            return slab_start(a, t, l2);
        }
        const int s0 = slab_start(a, t, f);
        const unsigned nf = (unsigned)(slab_start(a, t, f + 1) - s0), n = (unsigned)(cb(a, t, f + 1) - cf);
        const unsigned w = (unsigned)(c - cf), q = nf / n, r = nf - q * n;  // floor(w nf / n), w r < n^2
        return s0 + (int)(w * q + (w * r) / n);
    }
    // CTAs whose ranges overlap slab h (with rows [p0, p1)): their count, first and last.
    __device__ int slab_ctas(const DecodeArgs& a, const SeqTable& t, int h, int p0, int p1, int* c0, int* c1) const
    {
        if (!aligned) return ctas_of_slab(p0, p1, R, P, c0, c1);
        const int b0 = cb(a, t, h), b1 = cb(a, t, h + 1);
        if (b1 > b0) {
            *c0 = b0;
            *c1 = b1 - 1;
            return b1 - b0;
        }
        *c0 = *c1 = min(b0, P - 1);
        return 1;
    }
};

template <int G>
__global__ void __launch_bounds__(kTcThreads, 1)
    decode_tc_kernel(const __grid_constant__ DecodeArgs a, const __grid_constant__ CacheMaps maps)
{
    extern __shared__ __align__(128) unsigned char smem_raw[];
    unsigned char* sm = smem_raw + ((kTcAlign - (smem_u32(smem_raw) & (kTcAlign - 1))) & (kTcAlign - 1));
    unsigned char* ringK = sm + kOffK;
    unsigned char* ringV = sm + kOffV;
    unsigned char* sQ = sm + kOffQ;
    unsigned char* sP = sm + kOffP;
    float* g_max = reinterpret_cast<float*>(sm + kOffStats);  // [2][64] running max of each group, at a segment's end
    float* g_sum = g_max + 2 * kTcMaxCols;                     // [2][64] its sum
    float* g_alpha = g_sum + 2 * kTcMaxCols;                   // [2][64] rescale factors of a tile
    volatile int* flags = reinterpret_cast<volatile int*>(sm + kOffFlags);
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + kOffBars);
    uint64_t* k_full = bars;                        // [K] the stage's K rows landed
    uint64_t* k_empty = k_full + kKStages;          // [K] its score product is done
    uint64_t* v_full = k_empty + kKStages;          // [V] the stage's V rows landed
    uint64_t* v_empty = v_full + kVStages;          // [V] its output product is done
    uint64_t* s_full = v_empty + kVStages;          // [4] S of tile t (buffer t % 4) is done
    uint64_t* p_full = s_full + kSBufs;             // [2] P of tile t (buffer t % 2) is written
    uint64_t* o_done = p_full + 2;                  // [2] the output product of tile t is done
    uint64_t* q_full = o_done + 2;                  // [2] Q buffer b holds the Q of its next segment
    uint64_t* fin = q_full + 2;                     // drain after a timeout
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + kOffTmem);
    const SeqTable tab = seq_table_at(sm + kOffTable, a);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int NHl = a.B * a.Hkv;
    const int c = blockIdx.x;

    if (warp == 0)
        build_seq_table(a, tab, false);
    else
        load_slab_cache(a, tab, 32, kTcThreads - 32);
    if (tid == 32) {
        for (int i = 0; i < kNumBars; ++i) mbar_init(smem_u32(&bars[i]), 1);
        for (int i = 0; i < kNumFlags; ++i) flags[i] = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_proxy_async_smem();
    }
    __syncthreads();
    pdl_launch_dependents();

    const int R = slab_start(a, tab, NHl);
    if (c == 0 && warp == 2) {
        // Slabs with no rows belong to no CTA: their outputs are zero (after the
        // wait, as every write of out).
        pdl_wait();
        for (int h = 0; h < NHl; ++h)
            if (slab_start(a, tab, h) == slab_start(a, tab, h + 1))
                for (int j = 0; j < a.NC; ++j)
                    write_out<G>(a, h / a.Hkv, h % a.Hkv, j, make_float4(0.f, 0.f, 0.f, 0.f), 0.f, lane);
    }
    TcPart part;
    part.R = R;
    part.P = a.nctas;
    part.NHl = NHl;
    part.scale = (float)a.nctas / (float)max(R, 1);
    part.aligned = NHl * 4 <= a.nctas && R >= 4 * a.nctas;
    // Only while no CTA would get more than 1.15 shares of rows (R / P), and every
    // slab with rows gets a CTA of its own.
    for (int h = 0; h < NHl && part.aligned; ++h) {
        const int rows = slab_start(a, tab, h + 1) - slab_start(a, tab, h);
        const int n = part.cb(a, tab, h + 1) - part.cb(a, tab, h);
        if (rows > 0 && (n < 1 || (float)rows * part.scale > 1.15f * (float)n)) part.aligned = false;
    }
    const int A = part.start(a, tab, c), Bc = part.start(a, tab, c + 1);
    if (A >= Bc) return;  // uniform: this CTA has no rows (no TMEM taken yet)
    const int hfirst = slab_containing(a, tab, NHl, A);
    const int hend = slab_containing(a, tab, NHl, Bc - 1) + 1;
    const int NC = a.NC;
    const int NCpad = (NC + 15) & ~15;
    const float cs = a.qscale;
    uint32_t tmem = 0;

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA
        // Starts at once (the copies need no TMEM); K and V of a tile go to their
        // own rings, each issued as soon as its stage is free.
        if (lane == 0) {
            const uint64_t pol = evict_first_policy();
            TileWalk wk, wv;
            wk.begin(a, tab, hfirst, hend, A, Bc);
            wv = wk;
            int tk = 0, tv = 0;
            bool waited = false;
            IdleBound idle;
            while ((wk.more() || wv.more()) && !flags[kFlagAbort]) {
                bool moved = false;
                if (wk.more() && (tk < kKStages || test_phase(&k_empty[tk % kKStages], ((tk / kKStages) - 1) & 1))) {
                    if (tk == PRE && !waited) {
                        pdl_wait();  // later copies after the previous kernel, as in the other kernels
                        waited = true;
                    }
                    const int s = tk % kKStages, row = wk.cache_row();
                    // Bounds-checked build: the tile's rows lie in the cache (TMA reads
                    // zeros past the end, so the copy stays in bounds either way).
                    in_bounds(row >= 0 && (a.rows_cap == 0 || row + wk.cnt() <= a.rows_cap), a.status);
                    const uint32_t bar = smem_u32(&k_full[s]), dst = smem_u32(ringK + s * kTcHalfTile);
                    mbar_arrive_expect_tx(bar, kTcHalfTile);
#pragma unroll
                    for (int j = 0; j < kTcRows / kTcBoxRows; ++j) {
                        tma_box(dst + j * kTcBoxRows * 128, &maps.k, 0, row + j * kTcBoxRows, bar, pol);
                        tma_box(dst + kTcBox + j * kTcBoxRows * 128, &maps.k, 64, row + j * kTcBoxRows, bar, pol);
                    }
                    ++tk;
                    wk.next(a, tab);
                    moved = true;
                }
                if (wv.more() && tv < tk && (tv < kVStages || test_phase(&v_empty[tv % kVStages], ((tv / kVStages) - 1) & 1))) {
                    const int s = tv % kVStages, row = wv.cache_row();
                    const uint32_t bar = smem_u32(&v_full[s]), dst = smem_u32(ringV + s * kTcHalfTile);
                    mbar_arrive_expect_tx(bar, kTcHalfTile);
#pragma unroll
                    for (int j = 0; j < kTcRows / kTcBoxRows; ++j) {
                        tma_box(dst + j * kTcBoxRows * 128, &maps.v, 0, row + j * kTcBoxRows, bar, pol);
                        tma_box(dst + kTcBox + j * kTcBoxRows * 128, &maps.v, 64, row + j * kTcBoxRows, bar, pol);
                    }
                    ++tv;
                    wv.next(a, tab);
                    moved = true;
                }
                if (moved) {
                    idle.progress();
                } else if (idle.expired()) {
                    atomicOr(a.status, kDevTmaTimeout);
                    flags[kFlagAbort] = 1;
                    break;
                } else {
                    __nanosleep(32);
                }
            }
            flags[kFlagKIssued] = tk;
            flags[kFlagVIssued] = tv;
        }
    } else {
        if (warp >= 2) {
            // The first two segments' Q (buffers 0 and 1), loaded while warp 1
            // allocates TMEM: the first score product waits for both.
            const int st = tid - 64;
            pdl_wait();  // q and the outputs belong to the previous kernel's epoch
            TileWalk w0;
            w0.begin(a, tab, hfirst, hend, A, Bc);
            const int h1 = later_segment_slab(w0.cu, a, tab, hend, A, Bc, 1);
            load_q_tc<G>(a, w0.cu.h, sQ, st);
            if (h1 < hend) load_q_tc<G>(a, h1, sQ + kTcQBytes, st);
            fence_proxy_async_smem();
            named_sync(kBarSoft, kTcSoft);
            if (st == 0) {
                mbar_arrive(smem_u32(&q_full[0]));
                if (h1 < hend) mbar_arrive(smem_u32(&q_full[1]));
            }
        }
        if (warp == 1) {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                         "r"(kTcTmemCols));
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
        }
        tc_fence_before();
        named_sync(kBarTmem, kTcThreads - 32);
        tc_fence_after();
        tmem = *tmem_slot;
    }

    if (warp == 1) {
        // ---------------------------------------------------------------- MMA
        // Score products run up to kSBufs tiles ahead of the output products; a
        // score product needs its K stage, its S buffer free (the output product
        // of tile t - 4 issued, so its softmax is done) and, first in a segment,
        // the segment's Q; an output product needs its P and its V stage.
        if (lane == 0) {
            const uint32_t id1 = idesc(kTcQRows, kTcRows, 0, 0);
            const uint32_t id2 = idesc(128, 2 * NCpad, 1, 0);  // high and low parts of P side by side
            // Operand descriptors: every operand here has a stride byte offset of 1 KB,
            // version 1 and the 128-byte swizzle, so the high word is one constant; a
            // stage or k-step further on adds to the address field of the low word (16-byte
            // units; every shared-memory address is below 2^18 bytes, so the 14-bit field
            // never carries). One thread issues every product and its per-product work is
            // the pipeline's pace, so the loop keeps to 32-bit adds and running counters.
            const uint32_t dhi = (uint32_t)(sdesc(0, 0, 1024) >> 32);
            const uint32_t dQ = (uint32_t)sdesc(smem_u32(sQ), 16, 1024);
            const uint32_t dK = (uint32_t)sdesc(smem_u32(ringK), 16, 1024);
            const uint32_t dV = (uint32_t)sdesc(smem_u32(ringV), kTcBox, 1024);
            const uint32_t dP = (uint32_t)sdesc(smem_u32(sP), 16, 1024);
            auto desc = [dhi](uint32_t lo) { return ((uint64_t)dhi << 32) | lo; };
            TileWalk w1;
            w1.begin(a, tab, hfirst, hend, A, Bc);
            int t1 = 0, t2 = 0, seg = 0, seg_start = 0;
            int vs = 0;  // V stage of tile t2 (t2 % kVStages)
            // Bit t % kSBufs: tile t (between the two products) is one of the first two
            // of its segment, so its group's output product starts the accumulator afresh.
            uint32_t fresh_bits = 0;
            int qbuf = 0;  // Q buffer of the segment of tile t1
            bool issued = false, ok = true, qseen = false;
            IdleBound idle;
            while (w1.more() || t2 < t1) {
                bool moved = false;
                // Output products first: the softmax group of tile t2 waits for it before
                // it can write its next P. P of a tile is announced only after its V stage
                // landed (the group's leader waits for it), so p_full is the one test.
                if (t2 < t1) {
                    const int b = t2 & 1;
                    if (test_phase(&p_full[b], (t2 >> 1) & 1)) {
                        tc_fence_after();
                        // O^T += V^T [P_hi P_lo] into the group's accumulator (the two
                        // halves are summed when O is read); a group's first tile of a
                        // segment starts it afresh.
                        const uint32_t va = dV + (uint32_t)vs * (kTcHalfTile >> 4);
                        const uint32_t pb = dP + (uint32_t)b * (kTcPBytes >> 4);
                        const uint32_t o = tmem + kTcOCol + b * kTcOCols;
                        const uint32_t fresh = (fresh_bits >> (t2 & (kSBufs - 1))) & 1u;
                        umma(o, desc(va), desc(pb), id2, fresh ^ 1u);
#pragma unroll
                        for (int k = 1; k < kTcRows / 16; ++k)
                            umma(o, desc(va + k * (2048 >> 4)), desc(pb + k * (32 >> 4)), id2, 1u);
                        umma_commit(smem_u32(&o_done[b]));
                        umma_commit(smem_u32(&v_empty[vs]));
                        ++t2;
                        if (++vs == kVStages) vs = 0;
                        moved = true;
                    }
                }
                if (w1.more() && t1 < t2 + kSBufs) {
                    const int s = t1 & (kKStages - 1);
                    const bool first = w1.first();
                    if (first && !qseen && test_phase(&q_full[seg & 1], (seg >> 1) & 1)) {
                        qbuf = seg & 1;
                        ++seg;
                        seg_start = t1;
                        qseen = true;  // this segment's Q is in place
                    }
                    if ((!first || qseen) && test_phase(&k_full[s], (t1 / kKStages) & 1)) {
                        tc_fence_after();
                        // S^T[64 x 64] = Q[64 x 128] K^T: k-steps of 16 dims (+32 B inside a
                        // 64-dim half, +kTcBox or +kTcQHalf to the next half).
                        const uint32_t qa = dQ + (uint32_t)qbuf * (kTcQBytes >> 4);
                        const uint32_t kb = dK + (uint32_t)s * (kTcHalfTile >> 4);
                        const uint32_t d = tmem + (t1 & (kSBufs - 1)) * kTcRows;
#pragma unroll
                        for (int k = 0; k < 8; ++k)
                            umma(d, desc(qa + (k >> 2) * (kTcQHalf >> 4) + (k & 3) * 2),
                                 desc(kb + (k >> 2) * (kTcBox >> 4) + (k & 3) * 2), id1, k > 0 ? 1u : 0u);
                        umma_commit(smem_u32(&s_full[t1 & (kSBufs - 1)]));
                        umma_commit(smem_u32(&k_empty[s]));
                        const uint32_t bit = 1u << (t1 & (kSBufs - 1));
                        fresh_bits = (t1 - seg_start < 2) ? (fresh_bits | bit) : (fresh_bits & ~bit);
                        issued = true;
                        qseen = false;
                        ++t1;
                        w1.next(a, tab);
                        moved = true;
                    }
                }
                if (moved) {
                    idle.progress();
                } else if (flags[kFlagAbort] || idle.expired()) {
                    // Another role gave up, or nothing moved within the bound.
                    ok = false;
                    break;
                } else {
                    __nanosleep(20);
                }
            }
            if (!ok) {
                atomicOr(a.status, kDevTmaTimeout);
                flags[kFlagAbort] = 1;
            }
            flags[kFlagMmaLast] = issued ? 1 : 0;
        }
    } else if (warp >= 2) {
        // ---------------------------------------------------------------- softmax groups and epilogue
        const int gi = (warp - 2) >> 2;
        const int quarter = warp & 3;
        const int gt = tid - 64 - kTcGroup * gi;   // 0..127 within the group
        const int st = tid - 64;                    // 0..255 within both groups
        const bool gleader = gt == 0, leader = st == 0;
        const int gbar = 1 + gi;
        const uint32_t lane_addr = (uint32_t)(32 * quarter) << 16;
        const int half = lane >> 4;                 // rows 32 half .. 32 half + 31 of a tile
        const int col = 16 * quarter + (lane & 15);
        const bool live = col < NC;
        const int dim = 32 * quarter + lane;
        const uint32_t my_o = tmem + lane_addr + kTcOCol + gi * kTcOCols;
        TileWalk w;
        w.begin(a, tab, hfirst, hend, A, Bc);
        int seg_idx = -1;              // index of the current segment
        float m = -INFINITY, l = 0.f;  // this group's running max (log2 units) and sum of column col
        int t = 0, seg_start = 0;
        int last_mine = -1;            // this group's last tile of the current segment
        bool stop = false;             // set at a segment's end, the same in both groups
        // After a wait runs out a group keeps walking the tiles (without work) so that
        // both groups meet at every segment's end: a named barrier has no bound.
        for (; w.more() && !stop; ++t, w.next(a, tab)) {
            if (w.first()) {
                seg_start = t;
                ++seg_idx;
                last_mine = -1;
                m = -INFINITY;
                l = 0.f;
            }
            const bool last = w.last();
            if ((t & 1) == gi) {
                const int b = gi;
                const int cnt = w.cnt();
                const bool gfirst = t - seg_start < 2;  // the group's first tile of the segment
                last_mine = t;
                // The tile's scores (and, for a partial tile, its V rows, zeroed below).
                // The end of the group's previous output product, which read P buffer b
                // and wrote the group's O, is awaited once the scores are loaded (below),
                // or here for the group's first tile of a segment, which has no vote.
                if (gleader) {
                    bool ok = !flags[kFlagAbort] && wait_phase(&s_full[t % kSBufs], (t / kSBufs) & 1);
                    if (ok && gfirst && t >= 2) ok = wait_phase(&o_done[b], ((t - 2) >> 1) & 1);
                    // The tile's V stage (zeroed below past a partial tile's rows; and P is
                    // announced to the MMA lane only once V has landed).
                    if (ok) ok = wait_phase(&v_full[t % kVStages], (t / kVStages) & 1);
                    if (!ok && !flags[kFlagAbort]) {
                        atomicOr(a.status, kDevTmaTimeout);
                        flags[kFlagAbort] = 1;
                    }
                    flags[kFlagOk + gi] = ok;
                    tc_fence_before();
                }
                named_sync(gbar, kTcGroup);
                if (!flags[kFlagOk + gi]) {
                    named_sync(gbar, kTcGroup);  // the flag is rewritten at the group's next tile
                } else {
                    tc_fence_after();
                    float sc[32];  // rows 32 half + i of the tile, column col
                    tmem_ld16x2(tmem + lane_addr + (t % kSBufs) * kTcRows, sc);
                    if (cnt < kTcRows) {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (32 * half + i >= cnt) sc[i] = -INFINITY;  // rows past the segment
                    }
                    float mx[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) mx[i] = fmaxf(fmaxf(sc[4 * i], sc[4 * i + 1]), fmaxf(sc[4 * i + 2], sc[4 * i + 3]));
                    float mt = fmaxf(fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3])),
                                     fmaxf(fmaxf(mx[4], mx[5]), fmaxf(mx[6], mx[7])));
                    mt = fmaxf(mt, __shfl_xor_sync(kFull, mt, 16));  // the column's other half
                    mt = live ? mt * cs : -INFINITY;  // scale > 0: the max of the scaled scores
                    bool go = true;
                    if (gfirst) {
                        m = mt;
                        l = 0.f;
                    } else {
                        // Lazy rescale: only when a column's tile max tops its running max by kSlackTc.
                        const bool vote = live && mt > m + kSlackTc;
                        const unsigned any = __ballot_sync(kFull, vote);
                        if (lane == 0) flags[kFlagVote + 4 * gi + quarter] = any != 0;
                        if (gleader) {
                            bool ok = t < 2 || wait_phase(&o_done[b], ((t - 2) >> 1) & 1);
                            if (!ok && !flags[kFlagAbort]) {
                                atomicOr(a.status, kDevTmaTimeout);
                                flags[kFlagAbort] = 1;
                            }
                            flags[kFlagOk2 + gi] = ok;
                            tc_fence_before();
                        }
                        named_sync(gbar, kTcGroup);
                        go = flags[kFlagOk2 + gi];
                        tc_fence_after();
                        const bool rescale = flags[kFlagVote + 4 * gi] | flags[kFlagVote + 4 * gi + 1] |
                                             flags[kFlagVote + 4 * gi + 2] | flags[kFlagVote + 4 * gi + 3];
                        if (go && rescale) {
                            float alpha = 1.f;
                            if (vote) {
                                alpha = ex2(m - mt);
                                m = mt;
                                l *= alpha;
                            }
                            if (half == 0) g_alpha[gi * kTcMaxCols + col] = alpha;
                            named_sync(gbar, kTcGroup);
                            // The group's O, both halves (its previous product is done: waited above).
                            for (int c0 = 0; c0 < 2 * NCpad; c0 += 32) {
                                float v[32];
                                tmem_ld32(my_o + c0, v);
#pragma unroll
                                for (int i = 0; i < 32; ++i) {
                                    const int cc = c0 + i < NCpad ? c0 + i : c0 + i - NCpad;
                                    v[i] *= cc < NC ? g_alpha[gi * kTcMaxCols + cc] : 1.f;
                                }
                                tmem_st32(my_o + c0, v);
                            }
                        }
                    }
                    if (go) {
                        // P = 2^(s - m): a bf16 high part (the top 16 bits) and the bf16 of
                        // the remainder, row col of the B operand (64 rows, 128 bytes, swizzled).
                        if (col < NCpad) {
                            // Columns past NC get p = 0: 2^(s - inf) = 0 for finite or -inf s.
                            const float nm = live ? -m : -INFINITY;
                            unsigned char* ph = sP + b * kTcPBytes + col * 128;
                            unsigned char* pl = ph + NCpad * 128;  // row NCpad + col: same swizzle phase
                            float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                            for (int ch = 0; ch < 4; ++ch) {
                                uint32_t hi[4], lo[4];
#pragma unroll
                                for (int i = 0; i < 4; ++i) {
                                    const float p0 = ex2(fmaf(sc[8 * ch + 2 * i], cs, nm));  // 2^-inf = 0
                                    const float p1 = ex2(fmaf(sc[8 * ch + 2 * i + 1], cs, nm));
                                    ls[i] += p0 + p1;
                                    const uint32_t h0 = __float_as_uint(p0) & 0xffff0000u;
                                    const uint32_t h1 = __float_as_uint(p1) & 0xffff0000u;
                                    hi[i] = __byte_perm(h0, h1, 0x7632);
                                    lo[i] = pack_bf16(p0 - __uint_as_float(h0), p1 - __uint_as_float(h1));
                                }
                                const int off = ((4 * half + ch) ^ (col & 7)) << 4;
                                *reinterpret_cast<uint4*>(ph + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                                *reinterpret_cast<uint4*>(pl + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
                            }
                            l += (ls[0] + ls[1]) + (ls[2] + ls[3]);
                        }
                        if (cnt < kTcRows) {
                            // V rows past the segment: zeros (their p is 0, but 0 * inf or 0 * nan would not be).
                            unsigned char* v0 = ringV + (t % kVStages) * kTcHalfTile;
                            for (int i = gt; i < (kTcRows - cnt) * 16; i += kTcGroup) {
                                const int r = cnt + (i >> 4), k = i & 15;
                                *reinterpret_cast<uint4*>(v0 + (k >> 3) * kTcBox + r * 128 + ((k & 7) << 4)) =
                                    make_uint4(0u, 0u, 0u, 0u);
                            }
                        }
                        fence_proxy_async_smem();
                        tc_fence_before();
                        named_sync(gbar, kTcGroup);
                        if (gleader) mbar_arrive(smem_u32(&p_full[b]));
                    }
                }
            }
            if (!last) continue;

            // ---- end of a segment, both groups: the next segment's Q, then the merge of
            // the two groups' states, and this segment's output or partial.
            if (leader) flags[kFlagSegOk] = !flags[kFlagAbort];
            named_sync(kBarSoft, kTcSoft);  // every S product of the segment was seen done by its group
            const bool seg_ok = flags[kFlagSegOk];
            const int h = w.cu.h, p0h = w.cu.p0, p1h = w.cu.p0 + w.cu.n_h;
            const bool whole = w.cu.s0 == p0h && w.cu.s1 == p1h;
            // Q of the segment after next into this segment's buffer (its score
            // products are all done: each group saw its tiles' S).
            const int h2 = later_segment_slab(w.cu, a, tab, hend, A, Bc, 2);
            if (h2 < hend) {
                load_q_tc<G>(a, h2, sQ + (seg_idx & 1) * kTcQBytes, st);
                fence_proxy_async_smem();
            }
            const bool has0 = (t - seg_start >= 1) || ((seg_start & 1) == 0);  // group 0 had a tile here
            const bool has1 = (t - seg_start >= 1) || ((seg_start & 1) == 1);
            const float lsum = l + __shfl_xor_sync(kFull, l, 16);  // the column's two halves
            if (half == 0) {
                g_max[gi * kTcMaxCols + col] = m;
                g_sum[gi * kTcMaxCols + col] = lsum;
            }
            named_sync(kBarSoft, kTcSoft);
            if (leader && h2 < hend) mbar_arrive(smem_u32(&q_full[seg_idx & 1]));
            if (gleader) {
                bool ok = seg_ok;
                if (ok && last_mine >= 0) ok = wait_phase(&o_done[gi], (last_mine >> 1) & 1);
                if (seg_ok && !ok) {
                    atomicOr(a.status, kDevTmaTimeout);
                    flags[kFlagAbort] = 1;
                }
                flags[kFlagOk + gi] = ok;
                tc_fence_before();
            }
            named_sync(kBarSoft, kTcSoft);
            const bool merge_ok = flags[kFlagOk] && flags[kFlagOk + 1];
            stop = !merge_ok;
            tc_fence_after();
            // Merge of the groups: group gi writes the columns 32 gi .. 32 gi + 31 of every dimension.
            const int oc0 = 32 * gi;
            const int bq = h / a.Hkv, g = h - bq * a.Hkv;
            const int64_t slot = (int64_t)c + h;
            if (merge_ok && oc0 < NCpad) {
                // O of each group = its product with P_hi + its product with P_lo, 16
                // columns at a time (whole 32-column blocks spilled registers to local
                // memory, which misses the small L1 left beside this kernel's shared
                // memory and cost microseconds per segment end).
                const uint32_t o0 = tmem + lane_addr + kTcOCol, o1 = o0 + kTcOCols;
#pragma unroll 1
                for (int c16 = oc0; c16 < oc0 + 32 && c16 < NC; c16 += 16) {
                    uint32_t r0[16], w0[16], r1[16], w1[16];
                    tmem_ld16_async(o0 + c16, r0);
                    tmem_ld16_async(o0 + NCpad + c16, w0);
                    tmem_ld16_async(o1 + c16, r1);
                    tmem_ld16_async(o1 + NCpad + c16, w1);
                    tmem_wait_ld(r0, w0, r1, w1);
                    // Columns up to c16 + 15 are read even past NC (the statistics arrays
                    // hold kTcMaxCols columns), so that every shared-memory load of the
                    // chunk is independent of the stores: a load-use chain per column
                    // cost ~250 cycles a column under the kernel's shared-memory traffic.
                    float ov[16], Mv[16], Lv[16];
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int cc = c16 + i;
                        const float m0 = has0 ? g_max[cc] : -INFINITY, m1 = has1 ? g_max[kTcMaxCols + cc] : -INFINITY;
                        const float M = fmaxf(m0, m1);
                        const float f0 = has0 ? ex2(m0 - M) : 0.f, f1 = has1 ? ex2(m1 - M) : 0.f;
                        const float v0 = __uint_as_float(r0[i]) + __uint_as_float(w0[i]);
                        const float v1 = __uint_as_float(r1[i]) + __uint_as_float(w1[i]);
                        ov[i] = (has0 ? f0 * v0 : 0.f) + (has1 ? f1 * v1 : 0.f);
                        Mv[i] = M;
                        Lv[i] = (has0 ? f0 * g_sum[cc] : 0.f) + (has1 ? f1 * g_sum[kTcMaxCols + cc] : 0.f);
                    }
                    // Stores that skip L1 (st.global.cg): the L1 path is busy with the
                    // tiles' shared-memory traffic, and plain stores made a segment's
                    // end ~2.4 % of the whole launch slower (Q = 8 and 16). Every reader
                    // of these partials loads them from L2 (ld.global.cg).
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const int cc = c16 + i;
                        if (cc < NC) {
                            if (whole) {
                                __stcg(a.out + out_row<G>(a, bq, g, cc) * kHeadDim + dim, Lv[i] > 0.f ? ov[i] / Lv[i] : 0.f);
                            } else {
                                __stcg(a.work_o + (slot * NC + cc) * kHeadDim + dim, ov[i]);
                                if (dim == 0)
                                    __stcg(reinterpret_cast<float2*>(a.work_ml + (slot * NC + cc) * 2), make_float2(Mv[i], Lv[i]));
                            }
                        }
                    }
                }
            }
            // g_max / g_sum are rewritten at the next segment's end, after these reads.
            named_sync(kBarSoft, kTcSoft);
            if (merge_ok && !whole && leader) {
                // This CTA's partial of slab h is written (the barrier above orders the
                // other threads' stores before this thread's fence): count it in.
                __threadfence();
                atomicAdd(a.slab_count + (int64_t)h * kMaxCols * 2, 1);
            }
        }

        // ---- the CTA's share of the merges of its slabs that span several CTAs
        // (its first and its last segment; the slabs in between were whole).
        const int P = a.nctas;
        for (int e = 0; e < 2; ++e) {
            const int h = e == 0 ? hfirst : hend - 1;
            if (e == 1 && h == hfirst) break;
            const int p0 = slab_start(a, tab, h), p1 = slab_start(a, tab, h + 1);
            int c0 = 0, c1 = 0;
            const int nct = part.slab_ctas(a, tab, h, p0, p1, &c0, &c1);
            if (nct <= 1) continue;  // uniform: written at its segment's end
            int32_t* ctr = a.slab_count + (int64_t)h * kMaxCols * 2;
            if (leader) {
                // Every CTA of the slab counts in once its partial is written; the CTAs
                // are all resident (cooperative launch), so the count completes.
                bool ok = !flags[kFlagAbort];
                if (ok) {
                    ok = false;
                    const unsigned long long t0 = global_ns();
                    for (int i = 1; i < kWaitSpins; ++i) {
                        int n;
                        asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(n) : "l"(ctr) : "memory");
                        if (n >= nct + a.merge_extra) {
                            ok = true;
                            break;
                        }
                        if ((i & 63) == 0 && global_ns() - t0 > kWaitNs) break;
                    }
                    if (!ok) atomicOr(a.status, kDevMergeTimeout);
                }
                flags[kFlagSegOk] = ok;
            }
            named_sync(kBarSoft, kTcSoft);
            if (flags[kFlagSegOk]) {
                // Rank of this CTA among the slab's CTAs (every CTA of the range is live
                // when the layer has at least one row per CTA).
                const bool all_live = R >= P;
                int k = 0;
                if (all_live) {
                    k = c - c0;
                } else {
                    for (int cc = c0; cc < c; ++cc) k += part.start(a, tab, cc) < part.start(a, tab, cc + 1) ? 1 : 0;
                }
                const int j0 = (int)((int64_t)k * NC / nct), j1 = (int)((int64_t)(k + 1) * NC / nct);
                const int hb = h / a.Hkv, hg = h - hb * a.Hkv;
                // Columns j0 .. j1-1: warp (gi, quarter) takes j0 + 4 gi + quarter, then
                // every 8th. Per round of 32 partials, lane k loads the k-th partial's
                // (m, l) once (the weights of the round, with a running rescale when a
                // slab has more than 32 CTAs); then each lane covers 4 dims and keeps 16
                // partials' o in flight, so a round costs two or three L2 round trips.
                const int ncta = c1 - c0 + 1;
                for (int j = j0 + 4 * gi + quarter; j < j1; j += 8) {
                    float M = -INFINITY, L = 0.f;  // L: this lane's share of the sum
                    float4 O = make_float4(0.f, 0.f, 0.f, 0.f);
                    for (int k0 = 0; k0 < ncta; k0 += 32) {
                        const int cc = c0 + k0 + lane;
                        const bool okp = cc <= c1 && (all_live || part.start(a, tab, cc) < part.start(a, tab, cc + 1));
                        const float2 ml = okp ? __ldcg(reinterpret_cast<const float2*>(a.work_ml + (((int64_t)cc + h) * NC + j) * 2))
                                              : make_float2(-INFINITY, 0.f);
                        float rm = ml.x;
#pragma unroll
                        for (int o = 16; o >= 1; o >>= 1) rm = fmaxf(rm, __shfl_xor_sync(kFull, rm, o));
                        const float Mn = fmaxf(M, rm);
                        const float sc = M == -INFINITY ? 0.f : ex2(M - Mn);  // rescale of the earlier rounds
                        const float f = ml.x == -INFINITY ? 0.f : ex2(ml.x - Mn);
                        M = Mn;
                        L = fmaf(ml.y, f, L * sc);
                        O.x *= sc;
                        O.y *= sc;
                        O.z *= sc;
                        O.w *= sc;
                        const int n = min(32, ncta - k0);
                        for (int u0 = 0; u0 < n; u0 += 16) {
                            float4 v[16];
                            float fk[16];
#pragma unroll
                            for (int u = 0; u < 16; ++u) {
                                const int k = u0 + u;
                                fk[u] = __shfl_sync(kFull, f, k & 31);
                                const bool okk = __shfl_sync(kFull, okp ? 1 : 0, k & 31) != 0 && k < n;
                                v[u] = okk ? __ldcg(reinterpret_cast<const float4*>(
                                                        a.work_o + (((int64_t)c0 + k0 + k + h) * NC + j) * kHeadDim) +
                                                    lane)
                                           : make_float4(0.f, 0.f, 0.f, 0.f);
                                if (!okk) fk[u] = 0.f;
                            }
#pragma unroll
                            for (int u = 0; u < 16; ++u) {
                                O.x = fmaf(v[u].x, fk[u], O.x);
                                O.y = fmaf(v[u].y, fk[u], O.y);
                                O.z = fmaf(v[u].z, fk[u], O.z);
                                O.w = fmaf(v[u].w, fk[u], O.w);
                            }
                        }
                    }
#pragma unroll
                    for (int o = 16; o >= 1; o >>= 1) L += __shfl_xor_sync(kFull, L, o);
                    write_out<G>(a, hb, hg, j, O, L, lane);
                }
            }
            named_sync(kBarSoft, kTcSoft);
            if (leader) {
                // The last CTA of the slab to finish its share resets the counters for
                // the next call (every wait on the arrival count is over by then).
                const int done = atomicAdd(ctr + 1, 1);
                if (done == nct - 1) {
                    ctr[0] = 0;
                    ctr[1] = 0;
                    __threadfence();
                }
            }
        }
    }

    // ---------------------------------------------------------------- teardown
    tc_fence_before();
    __syncthreads();
    if (flags[kFlagAbort]) {
        // Drain what is still in flight, with the same bound, before the CTA exits:
        // the copies of every stage issued (a landed stage's wait returns at once),
        // and the products (a final commit).
        if (tid == 0) {
            const int nk = flags[kFlagKIssued], nv = flags[kFlagVIssued];
            for (int u = max(0, nk - kKStages); u < nk; ++u) wait_phase(&k_full[u % kKStages], (u / kKStages) & 1);
            for (int u = max(0, nv - kVStages); u < nv; ++u) wait_phase(&v_full[u % kVStages], (u / kVStages) & 1);
        }
        if (tid == 32 && flags[kFlagMmaLast]) {
            umma_commit(smem_u32(fin));
            wait_phase(fin, 0);
        }
        tc_fence_before();
        __syncthreads();
    }
    tc_fence_after();
    if (warp == 1)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTcTmemCols));
}

template <int G>
cudaError_t config_tc_g(int B, DecodeConfig* cfg)
{
    const int smem = tc_smem_bytes(B);
    cudaError_t e = cudaFuncSetAttribute(decode_tc_kernel<G>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0, per_sm = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_tc_kernel<G>, kTcThreads, smem)) !=
        cudaSuccess)
        return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    cfg->nctas = sms;  // one CTA per SM: co-resident (cooperative), and the TMEM allocation never waits
    cfg->nwarps = kTcThreads / 32;
    cfg->smem_bytes = smem;
    return cudaSuccess;
}

template <int G>
cudaError_t launch_tc_g(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg, cudaStream_t st)
{
    if (cfg.nwarps != kTcThreads / 32 || cfg.smem_bytes < tc_smem_bytes(a.B) || a.nctas < 1 || a.nctas > cfg.nctas ||
        a.NC < 1 || a.NC > kTcMaxCols || !a.slab_count)
        return cudaErrorInvalidConfiguration;
    // Cooperative (every CTA resident: a CTA waits for the other CTAs of its slabs)
    // and programmatic stream serialization, as the other decode kernels.
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3(a.nctas);
    lc.blockDim = dim3(kTcThreads);
    lc.dynamicSmemBytes = cfg.smem_bytes;
    lc.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeCooperative;
    attr[1].val.cooperative = 1;
    lc.attrs = attr;
    lc.numAttrs = 2;
    return cudaLaunchKernelEx(&lc, decode_tc_kernel<G>, a, maps);
}

}  // namespace

cudaError_t decode_config_tc(int G, int B, DecodeConfig* cfg)
{
    if (B < 1 || B > kMaxB) return cudaErrorInvalidValue;
    switch (G) {
        case 1: return config_tc_g<1>(B, cfg);
        case 2: return config_tc_g<2>(B, cfg);
        case 3: return config_tc_g<3>(B, cfg);
        case 4: return config_tc_g<4>(B, cfg);
        case 5: return config_tc_g<5>(B, cfg);
        case 6: return config_tc_g<6>(B, cfg);
        case 7: return config_tc_g<7>(B, cfg);
        case 8: return config_tc_g<8>(B, cfg);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_decode_tc(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg, cudaStream_t st)
{
    switch (a.G) {
        case 1: return launch_tc_g<1>(a, maps, cfg, st);
        case 2: return launch_tc_g<2>(a, maps, cfg, st);
        case 3: return launch_tc_g<3>(a, maps, cfg, st);
        case 4: return launch_tc_g<4>(a, maps, cfg, st);
        case 5: return launch_tc_g<5>(a, maps, cfg, st);
        case 6: return launch_tc_g<6>(a, maps, cfg, st);
        case 7: return launch_tc_g<7>(a, maps, cfg, st);
        case 8: return launch_tc_g<8>(a, maps, cfg, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace dkv
