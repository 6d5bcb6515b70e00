// Internal declarations shared by the translation units of libdkv.so.
// Nothing here is part of the public ABI (include/dkv.h is).
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace dkv {

constexpr int kHeadDim = 128;   // elements per row
constexpr int kRowBytes = 256;  // bytes per bf16 row

// Bounds-checked build (-DDKV_DEBUG, build.build_library(debug=True)): the
// kernels check the indices and offsets they read against the ranges the plan
// gives them, skip an access that falls outside, and set DKV_DEV_BOUNDS in the
// plan's status word. No trap and no assert, so the context stays usable and
// the host reads the word. In the normal build the checks compile to nothing.
#ifdef DKV_DEBUG
__device__ __forceinline__ bool in_bounds(bool ok, int32_t* status)
{
    if (!ok && status) atomicOr(status, 0x8 /* DKV_DEV_BOUNDS */);
    return ok;
}
#else
__device__ __forceinline__ constexpr bool in_bounds(bool, int32_t*) { return true; }
#endif

// ---------------------------------------------------------------- pattern map
struct MapArgs {
    const uint8_t* M;       // [L][H][D]
    const int32_t* Tc;      // [B]
    int2* runs;             // [NH][D+2]: kept runs of each slab in token order, (first output row, first position)
    int32_t* nruns;         // [NH]
    int32_t* len;           // [NH]
    int64_t* off;           // [NH+1]
    int64_t* ioff;          // [NH+1]
    int32_t* idx;           // [kept]
    int64_t* tail;          // [3 + L]: total rows, kept rows, longest slab, kept rows of each layer
    unsigned* done;         // CTAs of the runs pass that have finished (zero before the launch)
    int32_t* order;         // in place: [NH] slabs by length, longest first; else null
    int L, H, Hkv, D, B, sink, recent, bin_width, reserve;
    int NH;                 // L*B*Hkv
    int64_t stride;         // 0: slabs packed end to end; > 0: slab h starts at row h * stride (in place)
    int32_t* status;        // the plan's device status word (bounds-checked build)
};
constexpr int kMapChunk = 8192;  // output rows per CTA of the index-list write

// The runs of every slab, their lengths, the offset scans and the totals (and,
// in place, the slab order); then, once idx is allocated, the index-list write
// (max_len: the longest slab, from the totals).
cudaError_t launch_map(const MapArgs& a, cudaStream_t st);
cudaError_t launch_map_write(const MapArgs& a, int max_len, cudaStream_t st);

// ---------------------------------------------------------------- compaction
struct CompactArgs {
    const int32_t* len;
    const int64_t* off;
    const int64_t* ioff;
    const int32_t* idx;
    const uint16_t* K;
    const uint16_t* V;
    uint16_t* Kc;
    uint16_t* Vc;
    int64_t T_stride;
    int64_t kept;
    int NH;
    int32_t* status;        // the plan's device status word (bounds-checked build)
    int64_t rows_cap;       // rows of the packed cache (out of place) or of each buffer (in place)
};
cudaError_t launch_compact(const CompactArgs& a, cudaStream_t st);
// In place: K and V are both source and destination, slab h at rows h * T_stride
// (Kc/Vc unused); every slab's kept rows move to its first len rows, in order.
// order: the NH slabs, longest first; claim: a counter the launch zeroes.
cudaError_t launch_compact_inplace(const CompactArgs& a, const int32_t* order, int32_t* claim, cudaStream_t st);

// ---------------------------------------------------------------- decode
struct DecodeArgs {
    const uint16_t* q;      // [B][H][128] bf16 bits
    const uint16_t* k_new;  // [B][Hkv][128] or null
    const uint16_t* v_new;
    const int32_t* n_app;   // [B] or null
    uint16_t* Kc;
    uint16_t* Vc;
    const int32_t* len;     // layer slice [NHl]
    const int64_t* off;     // layer slice [NHl]
    const int64_t* ioff;    // layer slice [NHl+1] (absolute; the layer prefix is ioff[h]-ioff[0])
    float* work_o;          // [slots][G][128], one slot per (CTA, slab) partial
    float* work_ml;         // [slots][G][2]
    float* warp_o;          // [nparts][G][128]: a warp's state for a slab it left mid-range
    float* warp_ml;         // [nparts][G][2]
    float* out;             // [B][H][128]
    int32_t* slab_count;    // [B*Hkv][cols][2] arrivals, partials written (zero between calls)
    int32_t* status;
    int64_t rows_cap;       // rows of Kc/Vc, for the bounds-checked build; 0 when the caller does not give it
    int B, H, Hkv, G;
    int reserve;
    int append;             // 1 when k_new/v_new are given
    float qscale;           // softmax scale * log2(e)
    int nctas;              // CTAs of the split-K grid: the row partition's part count
    int Q;                  // queries per sequence (1 for the decode step); q and out are [B][Q][H][128]
    int NC;                 // columns per slab: Q * G; partial records hold NC rows of 128 + 2 floats
    int merge_extra;        // partials a fused merge waits for beyond the other CTAs' (0; 1 injects a wait that runs out)
};

// Most columns (queries x group heads) one decode call handles; the plan's
// split-K workspace and arrival counters are sized for this many.
constexpr int kMaxCols = 16;
// Most columns of one tcgen05 multi-query call (its CTA partials are sized for this many).
constexpr int kTcMaxCols = 64;

struct DecodeConfig {
    int nctas;        // the kernel's full grid (one CTA per SM); a call may use fewer (DecodeArgs::nctas)
    int nwarps;       // warps per CTA of the kernel
    int smem_bytes;   // dynamic shared memory of the kernel
};

// Carve-up of the split-K workspace, in floats from its base: the (CTA, slab)
// partials o [slots][slot_cols][128] and (m, l) [slots][slot_cols][2], the warp
// records o [warp_records][warp_cols][128] and (m, l) [warp_records][warp_cols][2].
// Each region starts on a 256-byte boundary: the kernels move o with 16-byte vector
// accesses and (m, l) with 8-byte ones, whatever slots x columns is (an odd
// product would otherwise leave the warp records 8-byte aligned).
struct WorkspaceLayout {
    int64_t work_o, work_ml, warp_o, warp_ml;  // region offsets (floats)
    int64_t total;                                     // floats of the whole workspace
};
constexpr int64_t kWorkAlignFloats = 64;  // 256 bytes
inline int64_t round_up_work(int64_t n) { return (n + kWorkAlignFloats - 1) / kWorkAlignFloats * kWorkAlignFloats; }
inline WorkspaceLayout workspace_layout(int64_t slots, int slot_cols, int64_t warp_records, int warp_cols)
{
    WorkspaceLayout w;
    w.work_o = 0;
    w.work_ml = w.work_o + round_up_work(slots * slot_cols * kHeadDim);
    w.warp_o = w.work_ml + round_up_work(slots * slot_cols * 2);
    w.warp_ml = w.warp_o + round_up_work(warp_records * warp_cols * kHeadDim);
    w.total = w.warp_ml + round_up_work(warp_records * warp_cols * 2);
    return w;
}
// The workspace of kernels of up to `nctas` CTAs of up to `nwarps` warps
// handling up to `cols` columns over a layer of `heads_per_layer` slabs: one
// record per column for every (CTA, slab) slot (nctas + slabs) and for every
// warp of the grid.
inline WorkspaceLayout decode_workspace(int nctas, int nwarps, int cols, int heads_per_layer)
{
    return workspace_layout((int64_t)nctas + heads_per_layer, cols, (int64_t)nctas * nwarps, cols);
}
// Grid and shared memory of the partial kernel for group size G on this device.
cudaError_t decode_config(int G, int B, DecodeConfig* cfg);
// Split-K partials of one layer into the workspace, then the per-(b, q-head) merge.
cudaError_t launch_decode_partial(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st);
// The partial pass with the combine fused in: the last CTA to finish a slab merges
// the slab's partials and writes out (uses a.slab_count).
cudaError_t launch_decode_fused(const DecodeArgs& a, const DecodeConfig& cfg, cudaStream_t st);
cudaError_t launch_decode_combine(const DecodeArgs& a, cudaStream_t st);

// Tensor-core decode kernel (dkv_decode_mma.cu): the same passes with K/V tiles
// fetched as 2-D TMA boxes through tensor maps of the packed K and V caches
// (rows x 128 bf16, 256-byte rows). Usable while the cache has at most
// kMaxMmaRows rows (TMA row coordinates are 32-bit).
struct CacheMaps {
    CUtensorMap k, v;
};
constexpr int64_t kMaxMmaRows = ((int64_t)1 << 31) - 16;
// Boxes of box_rows rows x 64 dims (16 for the mma.sync kernels, 64 for the tcgen05 one).
cudaError_t make_cache_maps(const void* Kc, const void* Vc, int64_t rows, CacheMaps* maps, bool short_boxes = false,
                            int box_rows = 16);
// Launch configuration of the tensor-core kernels of one kind: 0 = the decode
// step (G columns), 1 = multi-query with one tile of 8 columns, 2 = multi-query
// with two tiles (up to 16 columns).
cudaError_t decode_config_mma(int G, int B, int kind, DecodeConfig* cfg);
cudaError_t launch_decode_mma_partial(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg,
                                      cudaStream_t st);
cudaError_t launch_decode_mma_fused(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg,
                                    cudaStream_t st);
cudaError_t launch_advance(int32_t* n_app, int B, int reserve, int32_t* status, cudaStream_t st);

// tcgen05 multi-query kernel (dkv_decode_tc.cu): 1 to kTcMaxCols columns, one CTA
// per SM (a cooperative launch), the merge of slabs over several CTAs fused in
// (uses a.slab_count: entry [h][0][0..1] of each slab).
cudaError_t decode_config_tc(int G, int B, DecodeConfig* cfg);
cudaError_t launch_decode_tc(const DecodeArgs& a, const CacheMaps& maps, const DecodeConfig& cfg, cudaStream_t st);

// Exact-budget Top-K pattern export (dkv_topk.cu): device workspace bytes, and
// the launches (4 histogram passes, tie count, mark) on `st`.
int64_t topk_workspace_bytes();

// Page-backed buffers (dkv_vmm.cu): which pages a slab layout still needs, and
// the release of the others (synchronises the device first).
void vmm_pages_to_keep(const int32_t* len, int64_t nslabs, int64_t T_stride, int64_t reserve, int64_t guard,
                       int64_t row_bytes, int64_t page, int64_t npages, uint8_t* keep);
// phantom_cta (fault injection): the grid barriers wait for one CTA more than
// the grid has, so the first wait runs out at its bound.
cudaError_t launch_topk(const float* P, int64_t n, int64_t K, uint8_t* M, void* workspace, cudaStream_t st,
                        bool phantom_cta = false);

}  // namespace dkv
