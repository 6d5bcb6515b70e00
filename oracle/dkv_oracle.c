/*
 * Distance-KV CPU oracle: a plain, slow, scalar statement of the inference-side
 * path of "Distance-KV: Exploiting Relative Distance for Efficient Long-Context
 * Inference" (Sec. 3.4, Static-Pattern Inference), in fp64 where it does
 * arithmetic.
 *
 * THIS IS TEST INFRASTRUCTURE. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it. The product path never calls it,
 * and it shares no code, header, table or helper with the CUDA library.
 *
 * Conventions (the readings of the paper this oracle follows):
 *  - Positions are zero-indexed, p = i - 1 for the paper's one-indexed i. The
 *    sink is p < S, the recent window is p >= Tc - R, and a compressible
 *    position p lies in bin d = floor((Tc - R - 1 - p) / W) (Eq. 4 with S=128,
 *    R=1024, W=128 in the paper; S, R, W are parameters here).
 *  - A logical query head h of layer l keeps p when p is sink or recent, or
 *    when M[l][h][d(p)] = 1 (Eq. 5).
 *  - Under GQA a KV head keeps p when ANY query head of its group keeps p
 *    (Sec. 3.4, last paragraph). Group g holds query heads g*G .. g*G+G-1.
 *  - Kept positions are packed in ascending token order (Sec. 3.4); each
 *    (layer, sequence, KV head) slab is followed by `reserve` free rows for
 *    appended tokens, which are kept in full (Sec. 3.4).
 *  - Attention of the decode query over a slab is softmax(scale * q.k) v with
 *    scale = 1/sqrt(head_dim) unless given, all in fp64 from exactly widened
 *    bf16 inputs.
 *
 * Parity pins live in tests/test_oracle_pins.py; every function below is
 * pinned there (none is "parity unpinned").
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum {
    ORACLE_OK = 0,
    ORACLE_ERR_INVALID_ARG = 1,
    ORACLE_ERR_RANGE = 4,
};

/* Model/pattern geometry. L layers, H query heads, Hkv KV heads, D distance
 * bins, head_dim, sink S, recent R, bin width W. */
typedef struct {
    int32_t L, H, Hkv, D, head_dim, sink, recent, bin_width;
} oracle_shape;

/* bf16 -> double, exact: a bf16 is the top half of an IEEE float. */
static double bf16_to_double(uint16_t b)
{
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Eq. 4, zero-indexed: the relative-distance bin of compressible position p. */
long oracle_distance_bin(long p, long Tc, const oracle_shape *s)
{
    return (Tc - (long)s->recent - 1 - p) / (long)s->bin_width;
}

/* Eq. 5: the logical retention decision m_{l,h,p} of query head h in layer l. */
int oracle_keep_logical(const uint8_t *M, const oracle_shape *s, int layer, int h, long p, long Tc)
{
    if (p < (long)s->sink) return 1;               /* sink set S(Tc)   */
    if (p >= Tc - (long)s->recent) return 1;       /* recent set R(Tc) */
    long d = oracle_distance_bin(p, Tc, s);
    return M[((size_t)layer * s->H + h) * s->D + (size_t)d] != 0;
}

/* Sec. 3.4: the physical decision of KV head g is the union over its group. */
int oracle_keep_physical(const uint8_t *M, const oracle_shape *s, int layer, int g, long p, long Tc)
{
    int G = s->H / s->Hkv;
    for (int j = 0; j < G; ++j)
        if (oracle_keep_logical(M, s, layer, g * G + j, p, Tc)) return 1;
    return 0;
}

/* Argument checks shared by the map functions. Returns an ORACLE_* code. */
int oracle_validate(const uint8_t *M, const int32_t *Tc, int B, const oracle_shape *s, int reserve)
{
    if (!M || !Tc || !s || B < 1 || reserve < 0) return ORACLE_ERR_INVALID_ARG;
    if (s->L < 1 || s->H < 1 || s->Hkv < 1 || s->D < 0 || s->sink < 0 || s->recent < 0 ||
        s->bin_width < 1 || s->head_dim < 1)
        return ORACLE_ERR_INVALID_ARG;
    if (s->H % s->Hkv != 0) return ORACLE_ERR_INVALID_ARG;
    for (size_t i = 0; i < (size_t)s->L * s->H * s->D; ++i)
        if (M[i] > 1) return ORACLE_ERR_INVALID_ARG;
    for (int b = 0; b < B; ++b) {
        if (Tc[b] < 0) return ORACLE_ERR_INVALID_ARG;
        long compressible = (long)Tc[b] - s->sink - s->recent;
        /* The pattern has D bins of W positions: a longer compressible span
         * has positions with no bin. */
        if (compressible > (long)s->D * s->bin_width) return ORACLE_ERR_RANGE;
    }
    return ORACLE_OK;
}

/*
 * Pattern -> positions (Eqs. 4-5, GQA union of Sec. 3.4) for every
 * (layer l, sequence b, KV head g), heads flattened as h = (l*B + b)*Hkv + g.
 *   len[h]   number of kept context positions
 *   off[h]   first row of slab h in the packed cache; slabs are len+reserve long
 *   ioff[h]  first entry of slab h in idx (prefix sum of len alone)
 *   idx      kept positions of each slab, ascending (may be NULL: counts only)
 * off and ioff have NH+1 entries. Walks every position of every head.
 */
int oracle_map(const uint8_t *M, const int32_t *Tc, int B, const oracle_shape *s, int reserve,
               int32_t *len, int64_t *off, int64_t *ioff, int32_t *idx)
{
    int rc = oracle_validate(M, Tc, B, s, reserve);
    if (rc != ORACLE_OK) return rc;
    if (!len || !off || !ioff) return ORACLE_ERR_INVALID_ARG;
    int64_t row = 0, entry = 0;
    size_t h = 0;
    for (int l = 0; l < s->L; ++l)
        for (int b = 0; b < B; ++b)
            for (int g = 0; g < s->Hkv; ++g, ++h) {
                off[h] = row;
                ioff[h] = entry;
                int32_t n = 0;
                for (long p = 0; p < Tc[b]; ++p)
                    if (oracle_keep_physical(M, s, l, g, p, Tc[b])) {
                        if (idx) idx[entry + n] = (int32_t)p;
                        ++n;
                    }
                len[h] = n;
                entry += n;
                row += (int64_t)n + reserve;
            }
    off[h] = row;
    ioff[h] = entry;
    return ORACLE_OK;
}

/*
 * One-time prune-and-pack (Sec. 3.4): copy the kept rows of every slab, in
 * order, from the dense cache K[L][B][Hkv][T_stride][head_dim] into the packed
 * cache Kc[total_rows][head_dim] at off[h]; same for V. Rows are copied as raw
 * bf16 bytes. Reserve rows of Kc/Vc are left untouched.
 */
int oracle_compact(const int32_t *len, const int64_t *off, const int64_t *ioff, const int32_t *idx,
                   int L, int B, int Hkv, int head_dim, int64_t T_stride,
                   const uint16_t *K, const uint16_t *V, uint16_t *Kc, uint16_t *Vc)
{
    if (!len || !off || !ioff || !idx || !K || !V || !Kc || !Vc) return ORACLE_ERR_INVALID_ARG;
    size_t row_bytes = (size_t)head_dim * sizeof(uint16_t);
    size_t h = 0;
    for (int l = 0; l < L; ++l)
        for (int b = 0; b < B; ++b)
            for (int g = 0; g < Hkv; ++g, ++h) {
                size_t slab = (((size_t)l * B + b) * Hkv + g) * (size_t)T_stride;
                for (int32_t r = 0; r < len[h]; ++r) {
                    int32_t p = idx[ioff[h] + r];
                    if (p < 0 || p >= T_stride) return ORACLE_ERR_RANGE;
                    memcpy(Kc + (size_t)(off[h] + r) * head_dim, K + (slab + p) * head_dim, row_bytes);
                    memcpy(Vc + (size_t)(off[h] + r) * head_dim, V + (slab + p) * head_dim, row_bytes);
                }
            }
    return ORACLE_OK;
}

/*
 * Softmax attention of G query rows over n cached rows, fp64:
 *   s_r = scale * sum_k q[k] K[r][k];  w_r = exp(s_r - max s) / sum exp(.);
 *   out = sum_r w_r V[r].
 * q is bf16 [G][hd], Krows/Vrows bf16 [n][hd] (row stride hd). n == 0 gives
 * out = 0. weights, when not NULL, receives w as [G][n].
 */
void oracle_attend(const uint16_t *q, const uint16_t *Krows, const uint16_t *Vrows, long n,
                   int G, int hd, double scale, double *out, double *weights)
{
    double *sc = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    for (int j = 0; j < G; ++j) {
        double *o = out + (size_t)j * hd;
        for (int k = 0; k < hd; ++k) o[k] = 0.0;
        if (n == 0) continue;
        const uint16_t *qj = q + (size_t)j * hd;
        double mx = -INFINITY;
        for (long r = 0; r < n; ++r) {
            double dot = 0.0;
            for (int k = 0; k < hd; ++k)
                dot += bf16_to_double(qj[k]) * bf16_to_double(Krows[(size_t)r * hd + k]);
            sc[r] = scale * dot;
            if (sc[r] > mx) mx = sc[r];
        }
        double den = 0.0;
        for (long r = 0; r < n; ++r) {
            sc[r] = exp(sc[r] - mx);
            den += sc[r];
        }
        for (long r = 0; r < n; ++r) {
            double w = sc[r] / den;
            if (weights) weights[(size_t)j * n + r] = w;
            for (int k = 0; k < hd; ++k) o[k] += w * bf16_to_double(Vrows[(size_t)r * hd + k]);
        }
    }
    free(sc);
}

/*
 * Append the new token's key/value of every (sequence b, KV head g) of layer
 * `layer` at row off[h] + len[h] + n_app[b] of the packed cache (Sec. 3.4:
 * generated tokens are appended and kept in full). k_new/v_new are bf16
 * [B][Hkv][hd]. Fails with ORACLE_ERR_RANGE when a slab's reserve is used up.
 */
int oracle_append(const int32_t *len, const int64_t *off, int layer, int B, int Hkv, int hd,
                  int reserve, const int32_t *n_app, const uint16_t *k_new, const uint16_t *v_new,
                  uint16_t *Kc, uint16_t *Vc)
{
    for (int b = 0; b < B; ++b) {
        int na = n_app ? n_app[b] : 0;
        if (na < 0 || na >= reserve) return ORACLE_ERR_RANGE;
        for (int g = 0; g < Hkv; ++g) {
            size_t h = ((size_t)layer * B + b) * Hkv + g;
            if (off[h] + len[h] + na >= off[h + 1]) return ORACLE_ERR_RANGE; /* slab full */
            size_t dst = (size_t)(off[h] + len[h] + na) * hd;
            size_t src = ((size_t)b * Hkv + g) * hd;
            memcpy(Kc + dst, k_new + src, (size_t)hd * sizeof(uint16_t));
            memcpy(Vc + dst, v_new + src, (size_t)hd * sizeof(uint16_t));
        }
    }
    return ORACLE_OK;
}

/*
 * Decode-step attention of layer `layer` (Sec. 3.4: the query attends to the
 * compressed context cache plus the appended tokens). For every sequence b and
 * query head h, with KV head g = h / G, attend over the n = len + rows rows
 * starting at off of slab (layer, b, g), where rows = n_rows_app[b] appended
 * rows follow the packed context. q is bf16 [B][H][hd]; out is fp64 [B][H][hd].
 */
void oracle_decode(const int32_t *len, const int64_t *off, int layer, int B, int H, int Hkv, int hd,
                   const int32_t *n_rows_app, const uint16_t *q, const uint16_t *Kc, const uint16_t *Vc,
                   double scale, double *out)
{
    int G = H / Hkv;
    for (int b = 0; b < B; ++b)
        for (int g = 0; g < Hkv; ++g) {
            size_t h = ((size_t)layer * B + b) * Hkv + g;
            long n = (long)len[h] + (n_rows_app ? n_rows_app[b] : 0);
            const uint16_t *Kr = Kc + (size_t)off[h] * hd;
            const uint16_t *Vr = Vc + (size_t)off[h] * hd;
            oracle_attend(q + ((size_t)b * H + (size_t)g * G) * hd, Kr, Vr, n, G, hd, scale,
                          out + ((size_t)b * H + (size_t)g * G) * hd, NULL);
        }
}

/*
 * Exact retention budget (App. A.3): K_rho = round(rho * L * H * D), with round
 * read as floor(x + 1/2). Returns -1 for rho outside [0, 1] or a negative size.
 */
long oracle_budget(double rho, long L, long H, long D)
{
    if (!(rho >= 0.0 && rho <= 1.0) || L < 0 || H < 0 || D < 0) return -1;
    return (long)floor(rho * (double)L * (double)H * (double)D + 0.5);
}

/* The total order of the global Top-K: larger value first; equal values (and
 * +0 / -0) by lower flat index; NaN after every number, NaNs by index. */
static const float *g_topk_values;

static int topk_before(long i, long j)
{
    const float a = g_topk_values[i], b = g_topk_values[j];
    const int na = isnan(a), nb = isnan(b);
    if (na != nb) return nb; /* the number comes first */
    if (!na && a != b) return a > b;
    return i < j;
}

static int topk_cmp(const void *x, const void *y)
{
    const long i = *(const long *)x, j = *(const long *)y;
    if (i == j) return 0;
    return topk_before(i, j) ? -1 : 1;
}

/*
 * Global Top-K selection (Eq. 3, App. A.3): M[i] = 1 for the K first entries of
 * P (n entries, flat order) in the order above, 0 for the rest. Sorts the index
 * list with that order and marks its first K. K must lie in [0, n].
 */
int oracle_topk_mask(const float *P, long n, long K, uint8_t *M)
{
    if (n < 0 || K < 0 || K > n || (n > 0 && (!P || !M))) return ORACLE_ERR_INVALID_ARG;
    long *order = (long *)malloc((size_t)(n > 0 ? n : 1) * sizeof(long));
    if (!order) return ORACLE_ERR_INVALID_ARG;
    for (long i = 0; i < n; ++i) order[i] = i;
    g_topk_values = P;
    qsort(order, (size_t)n, sizeof(long), topk_cmp);
    memset(M, 0, (size_t)n);
    for (long r = 0; r < K; ++r) M[order[r]] = 1;
    free(order);
    return ORACLE_OK;
}
