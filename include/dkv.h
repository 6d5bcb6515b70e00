/*
 * dkv.h -- C ABI of the GB300 (sm_103a) Distance-KV inference hot path.
 *
 * Distance-KV (Sec. 3.2) keeps a static binary pattern M in {0,1}^{L x H x D}
 * over (layer, query head, relative-distance bin). At inference (Sec. 3.4) the
 * pattern is mapped once onto the context positions, the KV cache is pruned and
 * packed in token order, and every decode step attends over the packed cache
 * plus the tokens appended since. This library does those three steps on one
 * GPU:
 *
 *   dkv_map_pattern   pattern -> per-slab kept positions, lengths, offsets
 *   dkv_compact       one-time prune-and-pack of the dense K/V
 *   dkv_decode_attn   split-K decode attention over the packed cache
 *   dkv_free          release a plan
 *
 * and the step before them, the export of the pattern from learned retention
 * probabilities with an exact budget (dkv_budget, dkv_topk_mask; Eq. 3).
 *
 * Conventions used by every entry point
 *  - A "slab" is one (layer l, sequence b, KV head g); slabs are flattened as
 *    h = (l*B + b)*H_kv + g. A "row" is one token's key (or value) vector for
 *    one KV head: head_dim = 128 bf16 values = 256 bytes.
 *  - Positions are zero-indexed, p = i - 1 for the paper's one-indexed i.
 *    With sink S, recent R and bin width W, position p of a context of Tc
 *    tokens is kept by query head h of layer l when p < S, or p >= Tc - R, or
 *    M[l][h][floor((Tc - R - 1 - p) / W)] = 1 (Eqs. 4 and 5; the paper uses
 *    S = 128, R = 1024, W = 128).
 *  - GQA: query head h reads KV head h / G, G = H / H_kv (contiguous groups).
 *    A KV head keeps p when any query head of its group keeps p (Sec. 3.4,
 *    last paragraph); every query head then attends over that union.
 *  - Device pointers are plain CUDA device addresses on the current device.
 *    The caller owns every buffer it passes; the library owns the plan.
 *  - All calls are asynchronous on `stream`, except where stated. They never
 *    throw and never exit the process: they return a dkv_status, and
 *    dkv_last_error() holds a message for the calling thread.
 *  - Kernels never spin without a bound. A device-side problem (an append past
 *    the reserve, a copy that never lands) sets bits of the plan's device
 *    status word, which dkv_plan_status() reads.
 */
#ifndef DKV_H
#define DKV_H

#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    DKV_OK = 0,
    DKV_ERR_INVALID_ARG = 1, /* bad pointer, size, alignment or shape */
    DKV_ERR_CUDA = 2,        /* a CUDA runtime call or kernel launch failed */
    DKV_ERR_OOM = 3,         /* device or host allocation failed */
    DKV_ERR_RANGE = 4,       /* a context needs bins the pattern does not have */
    DKV_ERR_TIMEOUT = 5      /* reserved: bounded device waits report through dkv_plan_status */
} dkv_status;

/* Device status word bits (dkv_plan_status). */
#define DKV_DEV_APPEND_OVERFLOW 0x1 /* n_appended reached the slab's reserve: token not appended */
#define DKV_DEV_TMA_TIMEOUT 0x2     /* a bulk copy did not complete within the wait bound */
#define DKV_DEV_MERGE_TIMEOUT 0x4   /* a fused merge's partials were not all written within the wait bound */
#define DKV_DEV_BOUNDS 0x8          /* bounds-checked build only: an index or offset a kernel read was out of its range; the access was skipped */

/* Pattern and model geometry (Sec. 3.2, Sec. 3.4). */
typedef struct {
    int32_t L;         /* layers */
    int32_t H;         /* query heads per layer */
    int32_t H_kv;      /* KV heads per layer; H % H_kv == 0 */
    int32_t D;         /* distance bins of the pattern */
    int32_t head_dim;  /* must be 128 */
    int32_t sink;      /* S: leading positions always kept (paper: 128) */
    int32_t recent;    /* R: trailing positions always kept (paper: 1024) */
    int32_t bin_width; /* W: positions per distance bin (paper: 128) */
} dkv_shape;

typedef struct dkv_plan dkv_plan; /* opaque, library-owned */

/* Message of the last failing call on this thread ("" if none). */
const char* dkv_last_error(void);

/*
 * Map the pattern onto the context positions of every slab (Eqs. 4-5, GQA
 * union, Sec. 3.4) and build a packing plan.
 *
 * M_host        host uint8 [L][H][D], entries 0 or 1. Copied; caller keeps it.
 * ctx_len_host  host int32 [B], context length Tc[b] >= 0 of each sequence.
 * B             number of sequences, 1 <= B <= 512.
 * s             geometry; head_dim must be 128.
 * reserve_rows  free rows after every slab for appended tokens (>= 0).
 * stream        stream for the copies and kernels.
 * out           receives the plan.
 *
 * Packed layout decided here: slab h occupies rows [off[h], off[h+1]) of the
 * packed caches, its first len[h] rows are the kept context positions in
 * ascending order, and the next reserve_rows rows take appended tokens. The
 * kept positions themselves are listed in idx[ioff[h] .. ioff[h+1]).
 *
 * Errors: DKV_ERR_INVALID_ARG for a NULL pointer, an M entry other than 0/1,
 * H % H_kv != 0, head_dim != 128, a negative length or reserve, B out of range,
 * or a layer whose rows (with reserve) exceed 2^31 - 1; DKV_ERR_RANGE when some
 * Tc[b] - S - R > D * W (positions with no bin); DKV_ERR_OOM / DKV_ERR_CUDA.
 * Synchronises `stream` once, to learn the row counts (which size the index
 * list and the caller's packed caches). The index list is then written by a
 * kernel that the call leaves running on `stream`: work queued on `stream`
 * afterwards is ordered after it; other streams must wait for `stream`.
 * Device memory: one allocation for the plan's metadata and counters, and one,
 * sized after the sync, for the index list and the split-K workspace.
 */
dkv_status dkv_map_pattern(const uint8_t* M_host, const int32_t* ctx_len_host, int32_t B,
                           const dkv_shape* s, int32_t reserve_rows, cudaStream_t stream,
                           dkv_plan** out);

/*
 * Plan for the uncompressed ("Dense", Sec. 4.3) cache laid out as
 * [L][B][H_kv][T_stride][head_dim]: slab h starts at row h * T_stride and holds
 * Tc[b] context rows; the remaining T_stride - max(Tc) rows take appended
 * tokens. Used for the dense decode baseline; dkv_compact rejects it.
 * Errors: DKV_ERR_INVALID_ARG (as above, or T_stride < max Tc), OOM, CUDA.
 * Synchronous (small host-to-device copies).
 */
dkv_status dkv_plan_dense(const int32_t* ctx_len_host, int32_t B, const dkv_shape* s,
                          int64_t T_stride, cudaStream_t stream, dkv_plan** out);

/*
 * Read-only views of a plan. Any output pointer may be NULL. Besides the total
 * row count and the len/off/idx views, it returns kept_rows (the size of d_idx)
 * and d_ioff (where each slab's positions start in d_idx): a caller cannot
 * walk d_idx without them, and dkv_decode_attn_noalloc takes d_ioff.
 * total_rows  rows the packed caches need (sum of len + reserve).
 * kept_rows   number of kept context positions (sum of len).
 * d_len       device int32 [L*B*H_kv]
 * d_off       device int64 [L*B*H_kv + 1], slab start rows
 * d_ioff      device int64 [L*B*H_kv + 1], slab starts in d_idx (NULL for dense plans)
 * d_idx       device int32 [kept_rows], kept positions (NULL for dense plans)
 */
dkv_status dkv_plan_query(const dkv_plan* plan, int64_t* total_rows, int64_t* kept_rows,
                          const int32_t** d_len, const int64_t** d_off, const int64_t** d_ioff,
                          const int32_t** d_idx);

/*
 * Copy a plan's metadata to host buffers (any may be NULL to skip it):
 * len_host int32 [L*B*H_kv], off_host and ioff_host int64 [L*B*H_kv + 1],
 * idx_host int32 [kept_rows] (ioff/idx are skipped for dense plans).
 * Synchronises `stream`. Errors: DKV_ERR_INVALID_ARG (NULL plan), DKV_ERR_CUDA.
 */
dkv_status dkv_plan_read(const dkv_plan* plan, int32_t* len_host, int64_t* off_host, int64_t* ioff_host,
                         int32_t* idx_host, cudaStream_t stream);

/*
 * One-time prune-and-pack (Sec. 3.4: evicted states are physically removed and
 * the rest packed in token order, positions and RoPE unchanged).
 *
 * K, V      device bf16 [L][B][H_kv][T_stride][128], post-RoPE dense caches.
 * T_stride  row stride of one slab of K/V; >= max Tc.
 * Kc, Vc    device bf16 [total_rows][128], caller-allocated; rows
 *           [off[h], off[h] + len[h]) are written, reserve rows are not.
 * All four pointers must be 16-byte aligned. Bytes are copied exactly.
 * Errors: DKV_ERR_INVALID_ARG (NULL/unaligned pointer, dense plan, bad stride),
 * DKV_ERR_CUDA.
 */
dkv_status dkv_compact(const dkv_plan* plan, const void* K, const void* V, int64_t T_stride,
                       void* Kc, void* Vc, cudaStream_t stream);

/*
 * In-place variant of the two calls above (Sec. 3.4: evicted states are
 * physically removed): the packed cache lives inside the dense one, so no
 * second cache is allocated at compaction time.
 *
 * dkv_map_pattern_inplace   as dkv_map_pattern, but slab h starts at row
 *                           h * T_stride, the first row of its own region of the
 *                           dense K/V [L][B][H_kv][T_stride][128]: off[h] =
 *                           h * T_stride, total_rows = L*B*H_kv * T_stride, and
 *                           rows [len[h], len[h] + reserve_rows) of the region
 *                           take appended tokens. Needs T_stride >= max ctx_len
 *                           + reserve_rows.
 * dkv_compact_inplace       moves each slab's kept rows, in token order, to the
 *                           start of its region of K and of V (rows [0, len)).
 *                           Rows past len are left as they were. Afterwards pass
 *                           K and V as Kc and Vc to the decode calls. K and V:
 *                           device, 16-byte aligned, distinct.
 * Errors: DKV_ERR_INVALID_ARG (as above; a plan not made by
 * dkv_map_pattern_inplace), DKV_ERR_RANGE, DKV_ERR_OOM, DKV_ERR_CUDA.
 */
dkv_status dkv_map_pattern_inplace(const uint8_t* M, const int32_t* ctx_len, int32_t B, const dkv_shape* shape,
                                   int32_t reserve_rows, int64_t T_stride, cudaStream_t stream, dkv_plan** plan);
dkv_status dkv_compact_inplace(const dkv_plan* plan, void* K, void* V, cudaStream_t stream);

/*
 * Page-backed cache buffers, so that the memory of evicted states can be given
 * back after an in-place compaction (Sec. 3.4: evicted states are physically
 * removed; App. C reports the memory this saves).
 *
 * dkv_vmm_alloc      a device buffer of at least `bytes` bytes, one reserved
 *                    address range backed by separate physical pages of the
 *                    device's allocation granularity (*dptr: its address).
 *                    Allocate the dense K and the dense V each this way, then
 *                    fill them, map and compact in place.
 * dkv_vmm_trim       unmap and release every page of the buffer that holds no
 *                    row in [0, min(T_stride, len[h] + reserve + guard_rows)) of
 *                    any slab h of the in-place plan (rows of 256 bytes, slab h
 *                    at row h * T_stride). Accessing a released page faults:
 *                    afterwards use the buffer only through that plan (decode,
 *                    multi-query decode, appends within the reserve).
 *                    guard_rows >= 16: the decode kernels read whole 16-row
 *                    tiles, up to 15 rows past a slab's last row. Synchronises
 *                    the device. *freed_bytes: the memory released by this call.
 * dkv_vmm_pages_to_keep  the page rule of dkv_vmm_trim on host arrays: keep[i]
 *                    = 1 for page i of npages (page_bytes each) that must stay
 *                    mapped for slabs of len[h] rows (host only).
 * dkv_vmm_mapped_bytes / dkv_vmm_page_bytes  mapped bytes now; page size.
 * dkv_vmm_free       synchronise the device and release the buffer (NULL-safe).
 * Errors: DKV_ERR_INVALID_ARG, DKV_ERR_OOM, DKV_ERR_CUDA.
 */
typedef struct dkv_vmm dkv_vmm;
dkv_status dkv_vmm_alloc(int64_t bytes, dkv_vmm** buffer, void** dptr);
dkv_status dkv_vmm_trim(dkv_vmm* buffer, const dkv_plan* plan, int32_t guard_rows, int64_t* freed_bytes);
void dkv_vmm_pages_to_keep(const int32_t* len, int64_t nslabs, int64_t T_stride, int32_t reserve, int32_t guard_rows,
                           int64_t row_bytes, int64_t page_bytes, int64_t npages, uint8_t* keep);
int64_t dkv_vmm_mapped_bytes(const dkv_vmm* buffer);
int64_t dkv_vmm_page_bytes(const dkv_vmm* buffer);
void dkv_vmm_free(dkv_vmm* buffer);

/*
 * Decode-step attention of one layer over the packed cache (Sec. 3.4), split-K
 * over the kept rows with an online-softmax merge.
 *
 * layer         0 <= layer < L.
 * q             device bf16 [B][H][128], the decode query of this layer.
 * k_new, v_new  device bf16 [B][H_kv][128], this step's key/value, or both NULL.
 *               When given they are first appended at row
 *               off[h] + len[h] + n_appended[b] of each slab (generated tokens
 *               are kept in full, Sec. 3.4) and attended to in this call.
 * n_appended    device int32 [B]: tokens already appended to sequence b in
 *               earlier steps, or NULL for none. Not modified (see dkv_advance).
 * Kc, Vc        device bf16 packed caches from dkv_compact (or the dense K/V for
 *               a dense plan). 16-byte aligned.
 * scale         softmax scale; <= 0 selects 1/sqrt(128).
 * out           device fp32 [B][H][128]: softmax(scale q.k) v over the len[h] +
 *               n_appended[b] (+1 with k_new) rows of slab (layer, b, h / G);
 *               all zeros for a slab with no rows.
 * The plan holds the split-K workspace, so calls with the same plan must be
 * ordered (same stream, or synchronised). An append past the reserve is skipped
 * and sets DKV_DEV_APPEND_OVERFLOW.
 * The kernels use programmatic dependent launch: they may start while the
 * previous kernel in the stream is still running, and read q, k_new, v_new only
 * after it has completed. n_appended and the packed cache rows of earlier steps
 * are read before that point, so they must not be written by the kernel that
 * immediately precedes this call if that kernel signals early completion
 * (griddepcontrol.launch_dependents); an ordinary kernel never does.
 * Errors: DKV_ERR_INVALID_ARG (NULL/unaligned pointer, layer out of range,
 * only one of k_new/v_new), DKV_ERR_CUDA.
 */
dkv_status dkv_decode_attn(const dkv_plan* plan, int32_t layer, const void* q,
                           const void* k_new, const void* v_new, const int32_t* n_appended,
                           void* Kc, void* Vc, float scale, float* out, cudaStream_t stream);

/*
 * Several queries per sequence over one compressed cache (shared-context reuse,
 * Sec. 4.1: the compressed context cache serves the queries that follow it).
 * Each of the num_queries queries of sequence b attends, per query head, over
 * the same rows as dkv_decode_attn without k_new: the len[h] packed rows plus
 * the n_appended[b] rows appended so far. Nothing is appended and the queries
 * do not see each other.
 *
 * q    device bf16 [B][num_queries][H][128].
 * out  device fp32 [B][num_queries][H][128].
 * Needs 1 <= num_queries and num_queries * G <= 64 (G = H / H_kv), and a plan
 * whose cache has fewer than 2^31 rows. The query x head columns of a KV head
 * (num_queries * G of them) share every K/V row, so the rows are read once for
 * all queries:
 *   <= 16 columns  a split-K kernel whose warps multiply 16-row tiles on the
 *                  warp-level tensor-core path, then a combine kernel;
 *   17..64         one tcgen05 kernel: 64-row tiles staged by TMA, scores and
 *                  outputs accumulated in tensor memory, and the CTAs that
 *                  share a slab merge their partials inside the same launch.
 *                  It is a cooperative launch (all CTAs resident at once), so
 *                  it fails with DKV_ERR_CUDA where the device cannot grant
 *                  one (for example under a partitioned device).
 * Other arguments, ordering and errors are those of dkv_decode_attn; a
 * num_queries * G above 64 is DKV_ERR_INVALID_ARG.
 */
dkv_status dkv_decode_multi(const dkv_plan* plan, int32_t layer, const void* q, int32_t num_queries,
                            const int32_t* n_appended, void* Kc, void* Vc, float scale, float* out,
                            cudaStream_t stream);

/*
 * The two halves of dkv_decode_attn, for callers that schedule them apart
 * (or time them apart). dkv_decode_partial runs the split-K pass: every CTA of
 * a persistent grid takes an equal share of the layer's rows (slabs laid end to
 * end) and writes one (max, sum, unnormalised output) partial per slab it
 * touches into the plan's workspace, appending k_new/v_new as described above.
 * dkv_decode_combine merges those partials into `out`. The combine must follow
 * the partial of the same layer, with the same n_appended contents and
 * with_new_token = (k_new != NULL), before the plan's next partial call.
 * Arguments and errors are those of dkv_decode_attn.
 */
dkv_status dkv_decode_partial(const dkv_plan* plan, int32_t layer, const void* q, const void* k_new,
                              const void* v_new, const int32_t* n_appended, void* Kc, void* Vc,
                              float scale, cudaStream_t stream);
dkv_status dkv_decode_combine(const dkv_plan* plan, int32_t layer, const int32_t* n_appended,
                              int32_t with_new_token, float* out, cudaStream_t stream);

/*
 * End of a decode step: n_appended[b] += 1 for every sequence, on the device,
 * so a CUDA graph of one step can be replayed. Stops at the plan's reserve and
 * sets DKV_DEV_APPEND_OVERFLOW instead of passing it.
 * Errors: DKV_ERR_INVALID_ARG (NULL), DKV_ERR_CUDA.
 */
dkv_status dkv_advance(const dkv_plan* plan, int32_t* n_appended, cudaStream_t stream);

/*
 * Read (and optionally clear) the plan's device status word (DKV_DEV_* bits).
 * Synchronises `stream`. Returns DKV_OK even when bits are set.
 */
dkv_status dkv_plan_status(const dkv_plan* plan, int32_t* word, int32_t clear, cudaStream_t stream);

/*
 * dkv_decode_attn without any device allocation. The paper has no counterpart:
 * this is for callers that must not allocate device memory -- code hosted by a
 * serving engine or plugin framework that owns the whole device pool and
 * forbids cudaMalloc/cudaFree (both synchronise the device and fragment the
 * pool). Such callers cannot build a dkv_plan, so they pass the plan's metadata
 * themselves, laid out as dkv_plan_query describes:
 *   d_len  int32 [L*B*H_kv], d_off and d_ioff int64 [L*B*H_kv + 1] (device),
 * with reserve_rows the free rows after every slab. All other arguments are
 * those of dkv_decode_attn. status is a device int32 that receives the
 * DKV_DEV_* bits, or NULL to discard them.
 *
 * The split-K partials live in a fixed 8 MiB array inside the library image,
 * held on every GPU that loads the library until the process exits; a call
 * whose split-K records ((9 x SM count + B*H_kv) x G x 130 floats) do not fit gets
 * DKV_ERR_INVALID_ARG. The first call in a CUDA context (on each device, and
 * again after that context is destroyed and re-created, e.g. by
 * cudaDeviceReset) looks up the array's device address, and the first call for
 * each (G, B) in a context sets up the kernel's launch configuration; make
 * those first calls before any stream capture. Every call reuses the same
 * array, so calls whose kernels overlap on the GPU (other streams, other
 * threads) race with each other.
 * Errors: DKV_ERR_INVALID_ARG, DKV_ERR_CUDA.
 */
dkv_status dkv_decode_attn_noalloc(const dkv_shape* s, int32_t B, int32_t layer, int32_t reserve_rows,
                                   const int32_t* d_len, const int64_t* d_off, const int64_t* d_ioff,
                                   const void* q, const void* k_new, const void* v_new,
                                   const int32_t* n_appended, void* Kc, void* Vc, float scale,
                                   float* out, int32_t* status, cudaStream_t stream);

/* Release a plan (NULL-safe). Synchronises the device before freeing. */
void dkv_free(dkv_plan* plan);

/*
 * Exact-budget pattern export (Sec. 3.3, Eq. 3; App. A.3): learned retention
 * probabilities P in [0,1]^{L x H x D} become the binary pattern
 * M = TopKMask(P, K_rho) that dkv_map_pattern takes.
 *
 * dkv_budget     K_rho = round(rho * L * H * D) with round(x) = floor(x + 1/2)
 *                (host only). Returns -1 when rho is outside [0, 1] or a size is
 *                negative.
 * dkv_topk_workspace_bytes
 *                device workspace bytes dkv_topk_mask needs (about 29 KB, the
 *                same for every n).
 * dkv_topk_mask  P: device float [n], any layout, read in flat order.
 *                M: device uint8 [n], written in full. M[i] = 1 for the K first
 *                entries in this order: larger value first; equal values (+0
 *                and -0 are equal) by lower flat index; NaN after every number.
 *                workspace: device scratch of at least dkv_topk_workspace_bytes()
 *                bytes, 4-byte aligned; calls that share it must be ordered.
 *                Its first 32-bit word is a status word: nonzero after a call
 *                whose grid barrier wait ran out (M is then incomplete).
 *                One cooperative launch (all its CTAs resident at once).
 *                Asynchronous on stream; allocates nothing.
 * Errors: DKV_ERR_INVALID_ARG (n < 0 or n >= 2^31, K outside [0, n], a NULL
 * pointer with n > 0, a small or unaligned workspace), DKV_ERR_CUDA.
 */
int64_t dkv_budget(double rho, int32_t L, int32_t H, int32_t D);
int64_t dkv_topk_workspace_bytes(void);
dkv_status dkv_topk_mask(const float* P, int64_t n, int64_t K, uint8_t* M, void* workspace,
                         int64_t workspace_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* DKV_H */
