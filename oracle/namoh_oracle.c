/*
 * namoh_oracle.c -- plain fp64 CPU oracle for the NAMOH routed-attention path.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the correctness authority that the
 * CUDA path is compared against.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it; the product path never does.  It
 * shares no code, header, table or helper with the CUDA library.
 *
 * Everything here follows the paper's definitions literally, in fp64:
 *   - routing:   Sec. 3.1, Eq. (namoh-gates)  a_t = softmax(x_t W_r), S_K(t) = TopK(a_t),
 *                m_{t,i} = 1{i in S_K(t)}, g_{t,i} = m_{t,i} a_{t,i}  (no renormalisation,
 *                App. A.3, Eq. (namoh-biased-routing) and the sentence after it).
 *   - dispatch:  Sec. 3.1, ordered index sets I_i = {t : m_{t,i} = 1}, n_i = |I_i|;
 *                Sec. 3.2 "Efficient execution": each (batch, head) subsequence is packed
 *                as an independent sequence.
 *   - rank:      Sec. 3.2, Eq. (namoh-head-rope)  rho_i(t) = sum_{s<=t} m_{s,i} - 1.
 *   - RoPE:      Sec. 3.2, Eq. (namoh-head-rope)  q~ = q R(rho), k~ = k R(rho).
 *   - attention: Sec. 3.1, Eq. (namoh-attention)  h_{t,i} = Attn(q~_{t,i}, [k~_{s,i}], [v_{s,i}]),
 *                s in I_i, s <= t, standard scaled dot-product attention.
 *   - combine:   Sec. 3.1, Eq. (namoh-attention)  the per-slot term g_{t,i} h_{t,i}.
 *   - layer:     Sec. 3.1, Eq. (namoh-qkv)  q, k, v = x_t W^(i) for active pairs only, in the
 *                packed layout; Eq. (namoh-attention)  o_t = sum_i g_{t,i} h_{t,i} W_O^(i).
 *   - decode:    Sec. 3.1 (last paragraph) and Sec. 3.2: a new token appends to and attends
 *                within only its selected heads' histories; its rank is the current length.
 *   - GQA:       App. B.7, "Adopted KV-group routing": K/g of H/g groups are selected, the g
 *                query heads of a group share its gate, key/value history and rank.
 *   - shared:    the shared-head variant (Sec. 4.4): always-active heads over the full causal
 *                prefix or a sliding window of the last w tokens, at global RoPE positions.
 *   - SA+NAMOH:  App. B.8 with the selection model of App. B.3, Eqs. (app-block-budget) and
 *                (app-selected-entries): blocks of Bk entries in each routed history's local
 *                order; the current block plus the ceil(alpha N_B(r)) - 1 completed blocks
 *                scoring highest against their mean-pooled keys.
 *
 * Readings where the paper is silent (each listed in the design notes):
 *   - TopK compares the raw fp32 router logits (softmax is monotone, so the selected
 *     set equals TopK of a_t); ties go to the lower head index; slots are ordered by
 *     descending score.
 *   - RoPE is the half-split form: pairs (j, j + d/2), theta_j = base^(-2j/d),
 *     x'_j = x_j cos - x_{j+d/2} sin,  x'_{j+d/2} = x_{j+d/2} cos + x_j sin.
 *     Variants: interleaved pairs (2j, 2j+1), and the token's global index t as the
 *     position instead of its rank (the global-RoPE reading of Sec. 3.2).
 *   - Attention scale 1/sqrt(d_head).
 *   - Packed rows: segments in (batch, head) order, rows ascending in t inside a segment.
 *
 * Inputs in bf16 are passed as raw uint16 bit patterns and widened exactly.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG (-1)
#define ORACLE_ERR_NONFINITE (-2)
#define ORACLE_ERR_NOMEM (-3)
#define ORACLE_ERR_CAPACITY (-4)

/* ------------------------------------------------------------------------- */
/* small helpers                                                             */
/* ------------------------------------------------------------------------- */

static double bf16_to_double(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* A tiny parallel-for over [0, n) with a shared atomic counter. */
typedef void (*item_fn)(long item, void *ctx);
struct pool_job {
    long n;
    long next;
    item_fn fn;
    void *ctx;
};

static void *pool_worker(void *arg)
{
    struct pool_job *job = (struct pool_job *)arg;
    for (;;) {
        long i = __atomic_fetch_add(&job->next, 1, __ATOMIC_RELAXED);
        if (i >= job->n) break;
        job->fn(i, job->ctx);
    }
    return NULL;
}

static void parallel_for(long n, int nthreads, item_fn fn, void *ctx)
{
    struct pool_job job = {n, 0, fn, ctx};
    if (nthreads <= 1 || n <= 1) {
        pool_worker(&job);
        return;
    }
    if (nthreads > 256) nthreads = 256;
    pthread_t tid[256];
    int started = 0;
    for (int i = 0; i < nthreads - 1; ++i) {
        if (pthread_create(&tid[i], NULL, pool_worker, &job) == 0) ++started;
    }
    pool_worker(&job);
    for (int i = 0; i < started; ++i) pthread_join(tid[i], NULL);
}

/* ------------------------------------------------------------------------- */
/* Routing and dispatch (Sec. 3.1 Eq. namoh-gates; Sec. 3.2 Eq. namoh-head-rope) */
/* ------------------------------------------------------------------------- */

/* Head a precedes head b in the TopK order: larger score first, ties to the
 * lower index.  Scores are compared exactly as fp32 values (+0 == -0). */
static int head_precedes(const float *s, int a, int b)
{
    if (s[a] > s[b]) return 1;
    if (s[a] < s[b]) return 0;
    return a < b;
}

/*
 * oracle_route_topk: per token, S_K(t) and g_{t,i}.
 *   scores    [N, H] fp32 router logits x_t W_r (N = B*T tokens)
 *   topk_head [N, K] selected heads in descending score order (ties -> lower index)
 *   gate      [N, K] fp64 softmax over all H heads, taken at the selected heads
 * Returns ORACLE_ERR_NONFINITE if any score is NaN or infinite (outside the contract).
 */
int oracle_route_topk(const float *scores, long N, int H, int K, int32_t *topk_head, double *gate)
{
    if (!scores || !topk_head || !gate || N < 0 || H < 1 || K < 1 || K > H || H > 1024) return ORACLE_ERR_ARG;
    int order[1024];
    for (long t = 0; t < N; ++t) {
        const float *s = scores + t * (long)H;
        for (int i = 0; i < H; ++i)
            if (!isfinite(s[i])) return ORACLE_ERR_NONFINITE;
        /* insertion sort of head indices by (score desc, index asc) */
        for (int i = 0; i < H; ++i) {
            int j = i;
            while (j > 0 && head_precedes(s, i, order[j - 1])) {
                order[j] = order[j - 1];
                --j;
            }
            order[j] = i;
        }
        /* affinities a_t = softmax over all H heads, in fp64 */
        double mx = (double)s[order[0]];
        double z = 0.0;
        for (int i = 0; i < H; ++i) z += exp((double)s[i] - mx);
        for (int k = 0; k < K; ++k) {
            topk_head[t * K + k] = order[k];
            gate[t * K + k] = exp((double)s[order[k]] - mx) / z;
        }
    }
    return ORACLE_OK;
}

/*
 * oracle_route_biased: App. A.3, Eq. (namoh-biased-routing).  In fp64, per token:
 *   a_t = softmax(x_t W_r) over all H heads,
 *   S_K(t) = TopK_i(a_{t,i} + b_i)  (larger first, ties to the lower index),
 *   g_{t,i} = a_{t,i} at the selected heads (the bias stays out of the gates).
 *   bias      [H] fp32 per-head biases
 *   topk_head [N, K], gate [N, K] as oracle_route_topk
 *   key       [N, H] out: a_{t,i} + b_i, the quantity the selection ranks
 */
int oracle_route_biased(const float *scores, const float *bias, long N, int H, int K, int32_t *topk_head,
                        double *gate, double *key)
{
    if (!scores || !bias || !topk_head || !gate || !key || N < 0 || H < 1 || K < 1 || K > H || H > 1024)
        return ORACLE_ERR_ARG;
    int order[1024];
    double a[1024];
    for (int i = 0; i < H; ++i)
        if (!isfinite(bias[i])) return ORACLE_ERR_NONFINITE;
    for (long t = 0; t < N; ++t) {
        const float *s = scores + t * (long)H;
        double *kt = key + t * (long)H;
        double mx = -INFINITY;
        for (int i = 0; i < H; ++i) {
            if (!isfinite(s[i])) return ORACLE_ERR_NONFINITE;
            if ((double)s[i] > mx) mx = (double)s[i];
        }
        double z = 0.0;
        for (int i = 0; i < H; ++i) {
            a[i] = exp((double)s[i] - mx);
            z += a[i];
        }
        for (int i = 0; i < H; ++i) {
            a[i] /= z;
            kt[i] = a[i] + (double)bias[i];
        }
        /* insertion sort of head indices by (key desc, index asc) */
        for (int i = 0; i < H; ++i) {
            int j = i;
            while (j > 0 && kt[i] > kt[order[j - 1]]) {
                order[j] = order[j - 1];
                --j;
            }
            order[j] = i;
        }
        for (int k = 0; k < K; ++k) {
            topk_head[t * K + k] = order[k];
            gate[t * K + k] = a[order[k]];
        }
    }
    return ORACLE_OK;
}

/*
 * oracle_dispatch: ordered index sets I_i per (batch, head), walking t = 0..T-1
 * and appending each token to the heads it selected.
 *   topk_head   [B, T, K]
 *   n           [B*H]      n_{b,h} = |I_h| within sequence b
 *   seg_offsets [B*H + 1]  exclusive prefix sum of n in (b, h) order
 *   rank        [B, T, K]  rho_h(t), zero-based rank within the head's subsequence
 *   row         [B, T, K]  packed row = seg_offsets[b*H + h] + rho
 *   row_src     [B*T*K]    inverse map: row_src[row] = (b*T + t)*K + k
 */
int oracle_dispatch(const int32_t *topk_head, int B, int T, int H, int K,
                    int32_t *n, int32_t *seg_offsets, int32_t *rank, int32_t *row, int32_t *row_src)
{
    if (!topk_head || !n || !seg_offsets || !rank || !row || !row_src) return ORACLE_ERR_ARG;
    if (B < 0 || T < 0 || H < 1 || K < 1 || K > H) return ORACLE_ERR_ARG;
    for (long i = 0; i < (long)B * H; ++i) n[i] = 0;
    /* ranks: append in token order */
    for (int b = 0; b < B; ++b) {
        for (int t = 0; t < T; ++t) {
            for (int k = 0; k < K; ++k) {
                long idx = ((long)b * T + t) * K + k;
                int h = topk_head[idx];
                if (h < 0 || h >= H) return ORACLE_ERR_ARG;
                rank[idx] = n[(long)b * H + h];
                n[(long)b * H + h] += 1;
            }
        }
    }
    seg_offsets[0] = 0;
    for (long i = 0; i < (long)B * H; ++i) seg_offsets[i + 1] = seg_offsets[i] + n[i];
    for (int b = 0; b < B; ++b) {
        for (int t = 0; t < T; ++t) {
            for (int k = 0; k < K; ++k) {
                long idx = ((long)b * T + t) * K + k;
                int h = topk_head[idx];
                int r = seg_offsets[(long)b * H + h] + rank[idx];
                row[idx] = r;
                row_src[r] = (int32_t)idx;
            }
        }
    }
    return ORACLE_OK;
}

/*
 * oracle_dispatch_varlen: the same append over a ragged batch.  Sequence b holds
 * the tokens cu_seqlens[b] .. cu_seqlens[b+1]-1 of the flat token axis (N tokens in
 * all); each sequence has its own index sets and ranks (Sec. 3.1, Sec. 3.2).
 *   topk_head   [N, K]
 *   n           [B*H], seg_offsets [B*H + 1] as oracle_dispatch
 *   rank, row   [N, K]
 *   row_src     [N*K]      inverse map: row_src[row] = tok*K + k (tok on the flat axis)
 * cu_seqlens must start at 0, not decrease, and end at N.
 */
int oracle_dispatch_varlen(const int32_t *topk_head, const int32_t *cu_seqlens, int B, int H, int K,
                           int32_t *n, int32_t *seg_offsets, int32_t *rank, int32_t *row, int32_t *row_src)
{
    if (!topk_head || !cu_seqlens || !n || !seg_offsets || !rank || !row || !row_src) return ORACLE_ERR_ARG;
    if (B < 0 || H < 1 || K < 1 || K > H || cu_seqlens[0] != 0) return ORACLE_ERR_ARG;
    for (int b = 0; b < B; ++b)
        if (cu_seqlens[b + 1] < cu_seqlens[b]) return ORACLE_ERR_ARG;
    for (long i = 0; i < (long)B * H; ++i) n[i] = 0;
    for (int b = 0; b < B; ++b) {
        for (long tok = cu_seqlens[b]; tok < cu_seqlens[b + 1]; ++tok) {
            for (int k = 0; k < K; ++k) {
                long idx = tok * K + k;
                int h = topk_head[idx];
                if (h < 0 || h >= H) return ORACLE_ERR_ARG;
                rank[idx] = n[(long)b * H + h];
                n[(long)b * H + h] += 1;
            }
        }
    }
    seg_offsets[0] = 0;
    for (long i = 0; i < (long)B * H; ++i) seg_offsets[i + 1] = seg_offsets[i] + n[i];
    for (int b = 0; b < B; ++b) {
        for (long tok = cu_seqlens[b]; tok < cu_seqlens[b + 1]; ++tok) {
            for (int k = 0; k < K; ++k) {
                long idx = tok * K + k;
                int r = seg_offsets[(long)b * H + topk_head[idx]] + rank[idx];
                row[idx] = r;
                row_src[r] = (int32_t)idx;
            }
        }
    }
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------- */
/* RoPE (Sec. 3.2, Eq. namoh-head-rope)                                       */
/* ------------------------------------------------------------------------- */

/* x [d] (widened bf16) rotated to position p: out [d].  Pair j (frequency theta_j) is
 * (x_j, x_{j+d/2}) in the half-split form, (x_{2j}, x_{2j+1}) in the interleaved one. */
static void rope_rotate(const double *x, int d, double p, double base, int interleaved, double *out)
{
    int half = d / 2;
    for (int j = 0; j < half; ++j) {
        double theta = pow(base, -2.0 * (double)j / (double)d);
        double ang = p * theta;
        double c = cos(ang), s = sin(ang);
        int i0 = interleaved ? 2 * j : j, i1 = interleaved ? 2 * j + 1 : j + half;
        double x0 = x[i0], x1 = x[i1];
        out[i0] = x0 * c - x1 * s;
        out[i1] = x1 * c + x0 * s;
    }
}

/*
 * oracle_rope: rotate each bf16 row x[i, :] (row stride ld elements) to
 * position pos[i] and write fp64 rows out[i, :].
 */
int oracle_rope(const uint16_t *x, long rows, int d, long ld, const int64_t *pos, double base, int interleaved,
                double *out)
{
    if (!x || !pos || !out || rows < 0 || d < 2 || (d & 1) || ld < d) return ORACLE_ERR_ARG;
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    if (!tmp) return ORACLE_ERR_NOMEM;
    for (long i = 0; i < rows; ++i) {
        for (int c = 0; c < d; ++c) tmp[c] = bf16_to_double(x[i * ld + c]);
        rope_rotate(tmp, d, (double)pos[i], base, interleaved, out + i * (long)d);
    }
    free(tmp);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------- */
/* Scaled dot-product attention of one query over a history (Eq. namoh-attention) */
/* ------------------------------------------------------------------------- */

/* q [d], keys [len, d], values [len, d] -> h [d]; weights scratch [len] */
static void attend(const double *q, const double *keys, const double *values, long len, int d,
                   double *weights, double *h)
{
    double scale = 1.0 / sqrt((double)d);
    double mx = -INFINITY;
    for (long s = 0; s < len; ++s) {
        double acc = 0.0;
        for (int c = 0; c < d; ++c) acc += q[c] * keys[s * d + c];
        weights[s] = acc * scale;
        if (weights[s] > mx) mx = weights[s];
    }
    double z = 0.0;
    for (long s = 0; s < len; ++s) {
        weights[s] = exp(weights[s] - mx);
        z += weights[s];
    }
    for (int c = 0; c < d; ++c) h[c] = 0.0;
    for (long s = 0; s < len; ++s) {
        double w = weights[s] / z;
        for (int c = 0; c < d; ++c) h[c] += w * values[s * d + c];
    }
}

/* ------------------------------------------------------------------------- */
/* Prefill: RoPE at rank, routed causal attention, gate-weighted combine      */
/* ------------------------------------------------------------------------- */

struct prefill_ctx {
    const uint16_t *q, *v;
    const double *krot;        /* [R, d] rotated keys */
    const int32_t *seg_offsets;
    const int32_t *row_src;
    const double *gate;
    double *y;
    int nseg, d, g;
    double base;
    int interleaved;
    const int64_t *pos;       /* [R] position of each packed row, or NULL for its rank */
    long *item_seg, *item_r0; /* work items: (segment, first local query) */
    int chunk;
    int status;
};

static void prefill_item(long it, void *vctx)
{
    struct prefill_ctx *c = (struct prefill_ctx *)vctx;
    int d = c->d, g = c->g;
    long s = c->item_seg[it];
    long r0 = c->item_r0[it];
    long off = c->seg_offsets[s];
    long n = c->seg_offsets[s + 1] - off;
    long r1 = r0 + c->chunk < n ? r0 + c->chunk : n;
    double *vals = (double *)malloc(sizeof(double) * (size_t)(r1 > 0 ? r1 : 1) * d);
    double *w = (double *)malloc(sizeof(double) * (size_t)(r1 > 0 ? r1 : 1));
    double *qin = (double *)malloc(sizeof(double) * (size_t)d);
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    if (!vals || !w || !qin || !qr || !h) {
        c->status = ORACLE_ERR_NOMEM;
        free(vals); free(w); free(qin); free(qr); free(h);
        return;
    }
    for (long sidx = 0; sidx < r1; ++sidx)
        for (int cc = 0; cc < d; ++cc) vals[sidx * d + cc] = bf16_to_double(c->v[(off + sidx) * d + cc]);
    for (long r = r0; r < r1; ++r) {
        long row = off + r;
        long dst = c->row_src[row];
        for (int j = 0; j < g; ++j) {
            for (int cc = 0; cc < d; ++cc) qin[cc] = bf16_to_double(c->q[(row * g + j) * d + cc]);
            rope_rotate(qin, d, c->pos ? (double)c->pos[row] : (double)r, c->base, c->interleaved, qr);
            /* causal history: local ranks 0..r of this head (s in I_i, s <= t) */
            attend(qr, c->krot + off * d, vals, r + 1, d, w, h);
            double gt = c->gate[dst];
            for (int cc = 0; cc < d; ++cc) c->y[(dst * g + j) * d + cc] = gt * h[cc];
        }
    }
    free(vals); free(w); free(qin); free(qr); free(h);
}

struct rotk_ctx {
    const uint16_t *k;
    const int32_t *seg_offsets;
    double *krot;
    int d;
    double base;
    int interleaved;
    const int64_t *pos;
};

static void rotate_k_segment(long s, void *vctx)
{
    struct rotk_ctx *c = (struct rotk_ctx *)vctx;
    int d = c->d;
    long off = c->seg_offsets[s], end = c->seg_offsets[s + 1];
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    if (!tmp) return;
    for (long row = off; row < end; ++row) {
        for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(c->k[row * d + cc]);
        rope_rotate(tmp, d, c->pos ? (double)c->pos[row] : (double)(row - off), c->base, c->interleaved,
                    c->krot + row * d);
    }
    free(tmp);
}

/*
 * oracle_prefill: full prefill over packed rows.
 *   q        [R*g, d] bf16, query row of packed row r and group head j at r*g + j
 *   k, v     [R, d]   bf16 packed rows (segments in (b, h) order)
 *   nseg     number of segments (B * H, or B * H/g under KV-group routing)
 *   seg_offsets [nseg+1], row_src [R], gate [R] (indexed by row_src value)
 *   y        [R*g, d] fp64 output indexed by (row_src*g + j): the per-slot combine g*h
 *   k_rot    [R, d]   fp64 rotated keys, or NULL
 */
int oracle_prefill(const uint16_t *q, const uint16_t *k, const uint16_t *v, int nseg, int d, int g,
                   double base, const int32_t *seg_offsets, const int32_t *row_src, const double *gate,
                   double *y, double *k_rot, int nthreads, int interleaved, const int64_t *pos)
{
    if (!q || !k || !v || !seg_offsets || !row_src || !gate || !y) return ORACLE_ERR_ARG;
    if (nseg < 0 || d < 2 || (d & 1) || g < 1) return ORACLE_ERR_ARG;
    long R = seg_offsets[nseg];
    double *krot = k_rot;
    if (!krot) {
        krot = (double *)malloc(sizeof(double) * (size_t)(R > 0 ? R : 1) * d);
        if (!krot) return ORACLE_ERR_NOMEM;
    }
    struct rotk_ctx rk = {k, seg_offsets, krot, d, base, interleaved, pos};
    parallel_for(nseg, nthreads, rotate_k_segment, &rk);

    const int chunk = 64;
    long nitems = 0;
    for (int s = 0; s < nseg; ++s) {
        long n = seg_offsets[s + 1] - seg_offsets[s];
        nitems += (n + chunk - 1) / chunk;
    }
    long *item_seg = (long *)malloc(sizeof(long) * (size_t)(nitems > 0 ? nitems : 1));
    long *item_r0 = (long *)malloc(sizeof(long) * (size_t)(nitems > 0 ? nitems : 1));
    if (!item_seg || !item_r0) {
        free(item_seg); free(item_r0);
        if (!k_rot) free(krot);
        return ORACLE_ERR_NOMEM;
    }
    long it = 0;
    for (int s = 0; s < nseg; ++s) {
        long n = seg_offsets[s + 1] - seg_offsets[s];
        for (long r0 = 0; r0 < n; r0 += chunk) {
            item_seg[it] = s;
            item_r0[it] = r0;
            ++it;
        }
    }
    struct prefill_ctx ctx = {q, v, krot, seg_offsets, row_src, gate, y, nseg, d, g, base, interleaved, pos,
                              item_seg, item_r0, chunk, ORACLE_OK};
    parallel_for(nitems, nthreads, prefill_item, &ctx);
    free(item_seg); free(item_r0);
    if (!k_rot) free(krot);
    return ctx.status;
}

/*
 * oracle_prefill_rows: the same computation for a chosen list of query rows only
 * (used for sampled checks at sizes where the full oracle would be slow).
 *   rows [nrows] packed row indices, heads [nrows] group head j of each query
 *   out  [nrows, d] fp64 g*h for those queries
 */
int oracle_prefill_rows(const uint16_t *q, const uint16_t *k, const uint16_t *v, int nseg, int d, int g,
                        double base, const int32_t *seg_offsets, const int32_t *row_src, const double *gate,
                        const int64_t *rows, const int32_t *heads, long nrows, double *out, int interleaved,
                        const int64_t *pos)
{
    if (!q || !k || !v || !seg_offsets || !row_src || !gate || !rows || !heads || !out) return ORACLE_ERR_ARG;
    long R = seg_offsets[nseg];
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    /* rotated keys / widened values of the current segment, extended as needed
     * (rows listed in segment order reuse them) */
    double *keys = NULL, *vals = NULL, *w = NULL;
    long cached_seg = -1, cached_len = 0, cap_rows = 0;
    int st = (tmp && qr && h) ? ORACLE_OK : ORACLE_ERR_NOMEM;
    for (long i = 0; i < nrows && st == ORACLE_OK; ++i) {
        long row = rows[i];
        int j = heads[i];
        if (row < 0 || row >= R || j < 0 || j >= g) { st = ORACLE_ERR_ARG; break; }
        /* the segment containing this row */
        int lo = 0, hi = nseg;
        while (hi - lo > 1) {
            int mid = (lo + hi) / 2;
            if (seg_offsets[mid] <= row) lo = mid; else hi = mid;
        }
        long off = seg_offsets[lo];
        long n = seg_offsets[lo + 1] - off;
        long r = row - off;
        if (lo != cached_seg) {
            cached_seg = lo;
            cached_len = 0;
        }
        if (cap_rows < n) {
            free(keys); free(vals); free(w);
            keys = (double *)malloc(sizeof(double) * (size_t)n * d);
            vals = (double *)malloc(sizeof(double) * (size_t)n * d);
            w = (double *)malloc(sizeof(double) * (size_t)n);
            cap_rows = n;
            cached_len = 0;
            if (!keys || !vals || !w) { st = ORACLE_ERR_NOMEM; break; }
        }
        for (long s = cached_len; s <= r; ++s) {
            for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(k[(off + s) * d + cc]);
            rope_rotate(tmp, d, pos ? (double)pos[off + s] : (double)s, base, interleaved, keys + s * d);
            for (int cc = 0; cc < d; ++cc) vals[s * d + cc] = bf16_to_double(v[(off + s) * d + cc]);
        }
        if (r + 1 > cached_len) cached_len = r + 1;
        for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(q[(row * g + j) * d + cc]);
        rope_rotate(tmp, d, pos ? (double)pos[row] : (double)r, base, interleaved, qr);
        attend(qr, keys, vals, r + 1, d, w, h);
        double gt = gate[row_src[row]];
        for (int cc = 0; cc < d; ++cc) out[i * d + cc] = gt * h[cc];
    }
    free(keys); free(vals); free(w);
    free(tmp); free(qr); free(h);
    return st;
}

/* ------------------------------------------------------------------------- */
/* Decode step (Sec. 3.1 last paragraph; Sec. 3.2 "Efficient execution")     */
/* ------------------------------------------------------------------------- */

/*
 * oracle_decode_step: one new token per sequence.
 *   topk_head [B, Kr] selected heads (groups), gate [B, Kr] their gates
 *   q [B, Kr*g, d] bf16; k, v [B, Kr, d] bf16
 *   k_cache, v_cache [cap_total, d] fp64 histories (k_cache holds rotated keys);
 *   seg_base [B*Hr], seg_len [B*Hr] (updated in place), seg_cap [B*Hr]
 *   y [B, Kr*g, d] fp64: g * h for each selected (group) head
 * For each (b, slot): rho = seg_len; k~ = k R(p) and v are appended at rho;
 * q~ = q R(p) attends over the rho + 1 entries; seg_len += 1.  The rotation position
 * p is rho, or token_pos[b] (the new token's index in its sequence) when token_pos is
 * given; interleaved selects the pairing of rope_rotate.
 */
int oracle_decode_step(const int32_t *topk_head, const double *gate, const uint16_t *q, const uint16_t *k,
                       const uint16_t *v, int B, int Hr, int Kr, int d, int g, double base,
                       double *k_cache, double *v_cache, const int64_t *seg_base, int32_t *seg_len,
                       const int32_t *seg_cap, double *y, int interleaved, const int64_t *token_pos, int window)
{
    if (!topk_head || !gate || !q || !k || !v || !k_cache || !v_cache || !seg_base || !seg_len || !seg_cap || !y)
        return ORACLE_ERR_ARG;
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    if (!tmp || !qr || !h) { free(tmp); free(qr); free(h); return ORACLE_ERR_NOMEM; }
    int st = ORACLE_OK;
    for (int b = 0; b < B && st == ORACLE_OK; ++b) {
        for (int kk = 0; kk < Kr; ++kk) {
            int head = topk_head[b * Kr + kk];
            if (head < 0 || head >= Hr) { st = ORACLE_ERR_ARG; break; }
            long s = (long)b * Hr + head;
            long rho = seg_len[s];
            if (rho >= seg_cap[s]) { st = ORACLE_ERR_CAPACITY; break; }
            long base_row = seg_base[s];
            for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(k[((long)b * Kr + kk) * d + cc]);
            const double p = token_pos ? (double)token_pos[b] : (double)rho;
            rope_rotate(tmp, d, p, base, interleaved, k_cache + (base_row + rho) * d);
            for (int cc = 0; cc < d; ++cc)
                v_cache[(base_row + rho) * d + cc] = bf16_to_double(v[((long)b * Kr + kk) * d + cc]);
            double *w = (double *)malloc(sizeof(double) * (size_t)(rho + 1));
            if (!w) { st = ORACLE_ERR_NOMEM; break; }
            /* a sliding window keeps the last `window` rows, the new one included */
            const long first = (window > 0 && rho + 1 > window) ? rho + 1 - window : 0;
            for (int j = 0; j < g; ++j) {
                long qi = ((long)b * Kr + kk) * g + j;
                for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(q[qi * d + cc]);
                rope_rotate(tmp, d, p, base, interleaved, qr);
                attend(qr, k_cache + (base_row + first) * d, v_cache + (base_row + first) * d, rho + 1 - first, d, w,
                       h);
                for (int cc = 0; cc < d; ++cc) y[qi * d + cc] = gate[b * Kr + kk] * h[cc];
            }
            free(w);
            seg_len[s] = (int32_t)(rho + 1);
        }
    }
    free(tmp); free(qr); free(h);
    return st;
}

/* ------------------------------------------------------------------------- */
/* Projections around the path (Sec. 3.1, Eq. namoh-qkv and Eq. namoh-attention) */
/* ------------------------------------------------------------------------- */

struct proj_qkv_ctx {
    const uint16_t *x, *w;
    const int32_t *seg_offsets, *row_src;
    int nseg, Hr, Kr, g, d, d_model;
    double *q, *k, *v;
};

/* One packed row r: the token is row_src[r] / Kr, the group head that of r's segment. */
static void proj_qkv_row(long r, void *arg)
{
    const struct proj_qkv_ctx *c = (const struct proj_qkv_ctx *)arg;
    int lo = 0, hi = c->nseg;
    while (hi - lo > 1) {
        int mid = (lo + hi) / 2;
        if (c->seg_offsets[mid] <= r) lo = mid; else hi = mid;
    }
    const int hr = lo % c->Hr;
    const long tok = c->row_src[r] / c->Kr;
    const int ncols = (c->g + 2) * c->d;
    const uint16_t *xr = c->x + tok * (long)c->d_model;
    for (int n = 0; n < ncols; ++n) {
        const uint16_t *wr = c->w + ((long)hr * ncols + n) * c->d_model;
        double acc = 0.0;
        for (int m = 0; m < c->d_model; ++m) acc += bf16_to_double(xr[m]) * bf16_to_double(wr[m]);
        if (n < c->g * c->d) c->q[(r * c->g + n / c->d) * c->d + n % c->d] = acc;
        else if (n < (c->g + 1) * c->d) c->k[r * c->d + (n - c->g * c->d)] = acc;
        else c->v[r * c->d + (n - (c->g + 1) * c->d)] = acc;
    }
}

/*
 * oracle_proj_qkv: Sec. 3.1, Eq. (namoh-qkv): only active token-head pairs project,
 *   q_{t,i} = x_t W_Q^(i), k_{t,i} = x_t W_K^(i), v_{t,i} = x_t W_V^(i), t in I_i,
 * in the packed-row layout of the routing (App. B.7: a KV group projects one key and one
 * value and g queries, one per query head of the group).
 *   x           [N, d_model] bf16 token representations (N tokens on the flat axis)
 *   w           [Hr, (g+2) d, d_model] bf16: for group i, rows j d .. j d + d - 1 hold
 *               W_Q of query head i g + j transposed (row c = column c of W_Q), then
 *               d rows of W_K^(i) transposed, then d rows of W_V^(i) transposed
 *   seg_offsets [nseg + 1], row_src [R]: the routing's packed layout (nseg = B Hr)
 *   q [R g, d], k [R, d], v [R, d] fp64 out, q of row r and query head j at row r g + j
 */
int oracle_proj_qkv(const uint16_t *x, int d_model, const uint16_t *w, int Hr, int Kr, int g, int d,
                    const int32_t *seg_offsets, int nseg, const int32_t *row_src, double *q, double *k, double *v,
                    int nthreads)
{
    if (!x || !w || !seg_offsets || !row_src || !q || !k || !v) return ORACLE_ERR_ARG;
    if (d_model < 1 || Hr < 1 || Kr < 1 || g < 1 || d < 1 || nseg < 1) return ORACLE_ERR_ARG;
    struct proj_qkv_ctx c = {x, w, seg_offsets, row_src, nseg, Hr, Kr, g, d, d_model, q, k, v};
    parallel_for(seg_offsets[nseg], nthreads, proj_qkv_row, &c);
    return ORACLE_OK;
}

struct proj_out_ctx {
    const double *y;
    const uint16_t *w;
    const int32_t *topk_head;
    int Kr, g, d, d_model;
    double *o;
};

/* One token t: o_t = sum over its slots k and the g query heads j of the slot's group. */
static void proj_out_token(long t, void *arg)
{
    const struct proj_out_ctx *c = (const struct proj_out_ctx *)arg;
    const int gd = c->g * c->d;
    for (int m = 0; m < c->d_model; ++m) {
        double acc = 0.0;
        for (int k = 0; k < c->Kr; ++k) {
            const int hr = c->topk_head[t * c->Kr + k];
            const double *yk = c->y + (t * c->Kr + k) * (long)gd;
            const uint16_t *wr = c->w + ((long)hr * c->d_model + m) * gd;
            for (int e = 0; e < gd; ++e) acc += yk[e] * bf16_to_double(wr[e]);
        }
        c->o[t * c->d_model + m] = acc;
    }
}

/*
 * oracle_proj_out: Sec. 3.1, Eq. (namoh-attention): o_t = sum_{i in S_K(t)} g_{t,i} h_{t,i} W_O^(i),
 * from the combine's per-slot terms y = g h.
 *   y          [N, Kr, g, d] fp64 per-slot terms (slot k of token t, query head j of its group)
 *   topk_head  [N, Kr]: the group of each slot
 *   w          [Hr, d_model, g d] bf16: for group i, row m holds column m of W_O of query
 *              heads i g .. i g + g - 1, one after the other (W_O^(i g + j) row c at j d + c)
 *   o          [N, d_model] fp64 out
 */
int oracle_proj_out(const double *y, const int32_t *topk_head, long N, int Kr, int g, int d, const uint16_t *w,
                    int Hr, int d_model, double *o, int nthreads)
{
    if (!y || !topk_head || !w || !o || N < 0 || Kr < 1 || g < 1 || d < 1 || Hr < 1 || d_model < 1)
        return ORACLE_ERR_ARG;
    for (long i = 0; i < N * Kr; ++i)
        if (topk_head[i] < 0 || topk_head[i] >= Hr) return ORACLE_ERR_ARG;
    struct proj_out_ctx c = {y, w, topk_head, Kr, g, d, d_model, o};
    parallel_for(N, nthreads, proj_out_token, &c);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------- */
/* Shared heads (the always-active heads of the paper's shared-head variant)  */
/* ------------------------------------------------------------------------- */

struct shared_ctx {
    const uint16_t *q, *k, *v;
    int Hs, T, d, window, interleaved;
    double base;
    double *y;
};

/* One (sequence, shared head): every token, keys at global positions. */
static void shared_head(long bj, void *arg)
{
    const struct shared_ctx *c = (const struct shared_ctx *)arg;
    const int T = c->T, d = c->d;
    const long b = bj / c->Hs, j = bj % c->Hs;
    const long row0 = bj * (long)T;  /* q, k, v are [B, Hs, T, d] */
    double *keys = (double *)malloc(sizeof(double) * (size_t)T * d);
    double *vals = (double *)malloc(sizeof(double) * (size_t)T * d);
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    double *w = (double *)malloc(sizeof(double) * (size_t)T);
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    if (!keys || !vals || !tmp || !qr || !w || !h) goto done;
    for (long t = 0; t < T; ++t) {
        for (int cc = 0; cc < d; ++cc) {
            tmp[cc] = bf16_to_double(c->k[(row0 + t) * d + cc]);
            vals[t * d + cc] = bf16_to_double(c->v[(row0 + t) * d + cc]);
        }
        rope_rotate(tmp, d, (double)t, c->base, c->interleaved, keys + t * d);
    }
    for (long t = 0; t < T; ++t) {
        /* the full causal prefix, or the most recent `window` tokens including t */
        const long lo = (c->window > 0 && t + 1 > c->window) ? t + 1 - c->window : 0;
        for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(c->q[(row0 + t) * d + cc]);
        rope_rotate(tmp, d, (double)t, c->base, c->interleaved, qr);
        attend(qr, keys + lo * d, vals + lo * d, t + 1 - lo, d, w, h);
        for (int cc = 0; cc < d; ++cc) c->y[((b * T + t) * c->Hs + j) * d + cc] = h[cc];
    }
done:
    free(keys); free(vals); free(tmp); free(qr); free(w); free(h);
}

/*
 * oracle_shared_prefill: the always-active shared heads of the paper's shared-head variant
 * (Sec. 4.4, "Shared heads for local context"): every token, causal attention over the full
 * prefix (window = 0) or over the most recent `window` tokens including itself, RoPE at the
 * global position t, no gate.
 *   q, k, v  [B, Hs, T, d] bf16 bits (each head's sequence contiguous)
 *   y        [B, T, Hs, d] fp64 out
 */
int oracle_shared_prefill(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int Hs, int T, int d,
                          int window, double base, int interleaved, double *y, int nthreads)
{
    if (!q || !k || !v || !y || B < 1 || Hs < 1 || T < 1 || d < 2 || d % 2 || window < 0) return ORACLE_ERR_ARG;
    struct shared_ctx c = {q, k, v, Hs, T, d, window, interleaved, base, y};
    parallel_for((long)B * Hs, nthreads, shared_head, &c);
    return ORACLE_OK;
}

/* ------------------------------------------------------------------------- */
/* SA + NAMOH: block selection inside each routed history (App. B.3 "Block-   */
/* Selected Sparse Attention", App. B.8 "SA+NAMOH")                           */
/* ------------------------------------------------------------------------- */

/*
 * Within one routed head history (local order, keys k~ after head-relative RoPE), a query at
 * one-based local rank r sees N_B(r) = ceil(r / Bk) blocks of Bk entries (Eq. app-block-budget)
 * and keeps R(r) = ceil(alpha N_B(r)) of them: its current block, causally, and the R(r) - 1
 * completed historical blocks with the highest scores.  A block's score is the query's dot
 * product with the block's mean-pooled key (the MoBA selector named in App. B.3).  The query
 * then attends with scaled dot-product attention over the entries of those blocks, and the
 * gate-weighted combine is that of the plain path.
 * Readings: alpha = a_num / a_den exactly; ties between block scores go to the lower block
 * index; the pooled keys are the rotated keys k~ the attention itself uses.
 */
static long sa_blocks_kept(long r1, int Bk, long a_num, long a_den)
{
    long nb = (r1 + Bk - 1) / Bk;               /* N_B(r) */
    return (nb * a_num + a_den - 1) / a_den;    /* R(r) = ceil(alpha N_B(r)) */
}

struct sa_ctx {
    const uint16_t *q, *v;
    const double *krot, *kbar;   /* [R, d] rotated keys; [R, d] block means at off + b */
    const int32_t *seg_offsets, *row_src;
    const double *gate;
    double *y;
    const uint32_t *mask_in;
    uint32_t *mask_out;
    int mask_words;
    int nseg, d, g, Bk;
    long a_num, a_den;
    double base;
    int interleaved;
    const int64_t *pos;
    long *item_seg, *item_r0;
    int chunk;
    int status;
};

static void sa_item(long it, void *vctx)
{
    struct sa_ctx *c = (struct sa_ctx *)vctx;
    int d = c->d, g = c->g, Bk = c->Bk;
    long s = c->item_seg[it], r0 = c->item_r0[it];
    long off = c->seg_offsets[s], n = c->seg_offsets[s + 1] - off;
    long r1 = r0 + c->chunk < n ? r0 + c->chunk : n;
    long nblk = (n + Bk - 1) / Bk;
    double *keys = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1) * d);
    double *vals = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1) * d);
    double *vraw = (double *)malloc(sizeof(double) * (size_t)(r1 > 0 ? r1 : 1) * d);
    double *w = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    double *score = (double *)malloc(sizeof(double) * (size_t)(nblk > 0 ? nblk : 1));
    char *take = (char *)malloc((size_t)(nblk > 0 ? nblk : 1));
    double *qin = (double *)malloc(sizeof(double) * (size_t)d);
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    double *h = (double *)malloc(sizeof(double) * (size_t)d);
    if (!keys || !vals || !vraw || !w || !score || !take || !qin || !qr || !h) {
        c->status = ORACLE_ERR_NOMEM;
        goto done;
    }
    for (long t = 0; t < r1; ++t)
        for (int cc = 0; cc < d; ++cc) vraw[t * d + cc] = bf16_to_double(c->v[(off + t) * d + cc]);
    for (long r = r0; r < r1; ++r) {
        long row = off + r;
        long rank1 = r + 1;                       /* one-based local rank */
        long cur = r / Bk;                        /* current block: N_B(r) - 1 */
        long keep = sa_blocks_kept(rank1, Bk, c->a_num, c->a_den) - 1;  /* historical blocks kept */
        long dst = c->row_src[row];
        for (int j = 0; j < g; ++j) {
            long qi = row * g + j;
            const double qpos = c->pos ? (double)c->pos[row] : (double)r;
            for (int cc = 0; cc < d; ++cc) qin[cc] = bf16_to_double(c->q[qi * d + cc]);
            rope_rotate(qin, d, qpos, c->base, c->interleaved, qr);
            for (long b = 0; b < cur; ++b) take[b] = 0;
            if (c->mask_in) {
                for (long b = 0; b < cur; ++b)
                    take[b] = (char)((c->mask_in[qi * c->mask_words + b / 32] >> (b % 32)) & 1u);
            } else {
                /* scores of the completed blocks against their mean-pooled keys */
                for (long b = 0; b < cur; ++b) {
                    double acc = 0.0;
                    for (int cc = 0; cc < d; ++cc) acc += qr[cc] * c->kbar[(off + b) * d + cc];
                    score[b] = acc;
                }
                /* the `keep` highest, ties to the lower block index */
                for (long m = 0; m < keep; ++m) {
                    long best = -1;
                    for (long b = 0; b < cur; ++b)
                        if (!take[b] && (best < 0 || score[b] > score[best])) best = b;
                    if (best < 0) break;  /* keep <= cur always (alpha <= 1) */
                    take[best] = 1;
                }
            }
            if (c->mask_out) {
                for (int wd = 0; wd < c->mask_words; ++wd) c->mask_out[qi * c->mask_words + wd] = 0u;
                for (long b = 0; b < cur; ++b)
                    if (take[b]) c->mask_out[qi * c->mask_words + b / 32] |= 1u << (b % 32);
            }
            /* the attended entries: kept historical blocks, then the current block up to r */
            long len = 0;
            for (long b = 0; b <= cur; ++b) {
                if (b < cur && !take[b]) continue;
                long e1 = b < cur ? (b + 1) * Bk : r + 1;
                for (long t = b * Bk; t < e1; ++t, ++len) {
                    memcpy(keys + len * d, c->krot + (off + t) * d, sizeof(double) * (size_t)d);
                    memcpy(vals + len * d, vraw + t * d, sizeof(double) * (size_t)d);
                }
            }
            attend(qr, keys, vals, len, d, w, h);
            double gt = c->gate[dst];
            for (int cc = 0; cc < d; ++cc) c->y[(dst * g + j) * d + cc] = gt * h[cc];
        }
    }
done:
    free(keys); free(vals); free(vraw); free(w); free(score); free(take); free(qin); free(qr); free(h);
}

/* mean-pooled rotated keys of the complete blocks of segment s, at rows off + b */
struct sa_pool_ctx {
    const double *krot;
    const int32_t *seg_offsets;
    double *kbar;
    int d, Bk;
};

static void sa_pool_segment(long s, void *vctx)
{
    struct sa_pool_ctx *c = (struct sa_pool_ctx *)vctx;
    int d = c->d, Bk = c->Bk;
    long off = c->seg_offsets[s], n = c->seg_offsets[s + 1] - off;
    for (long b = 0; b < n / Bk; ++b)
        for (int cc = 0; cc < d; ++cc) {
            double acc = 0.0;
            for (long t = b * Bk; t < (b + 1) * Bk; ++t) acc += c->krot[(off + t) * d + cc];
            c->kbar[(off + b) * d + cc] = acc / (double)Bk;
        }
}

/*
 * oracle_sa_prefill: SA + NAMOH prefill over packed rows (layout as oracle_prefill).
 *   Bk          block size (>= 1); alpha = a_num / a_den in (0, 1]
 *   mask_in     [R*g, mask_words] kept historical blocks per query (bit b of word b/32), or NULL
 *               to select them here; only blocks before the query's current block are read
 *   mask_out    [R*g, mask_words] the blocks kept, or NULL
 *   y           [R*g, d] fp64 per-slot combine g*h at (row_src*g + j)
 */
int oracle_sa_prefill(const uint16_t *q, const uint16_t *k, const uint16_t *v, int nseg, int d, int g,
                      double base, const int32_t *seg_offsets, const int32_t *row_src, const double *gate,
                      int Bk, long a_num, long a_den, const uint32_t *mask_in, uint32_t *mask_out, int mask_words,
                      double *y, int nthreads, int interleaved, const int64_t *pos)
{
    if (!q || !k || !v || !seg_offsets || !row_src || !gate || !y) return ORACLE_ERR_ARG;
    if (nseg < 0 || d < 2 || (d & 1) || g < 1 || Bk < 1 || a_num < 1 || a_den < a_num) return ORACLE_ERR_ARG;
    long R = seg_offsets[nseg];
    long nmax = 0;
    for (int s = 0; s < nseg; ++s)
        if (seg_offsets[s + 1] - seg_offsets[s] > nmax) nmax = seg_offsets[s + 1] - seg_offsets[s];
    if ((mask_in || mask_out) && (long)mask_words * 32 < (nmax + Bk - 1) / Bk) return ORACLE_ERR_ARG;
    double *krot = (double *)malloc(sizeof(double) * (size_t)(R > 0 ? R : 1) * d);
    double *kbar = (double *)malloc(sizeof(double) * (size_t)(R > 0 ? R : 1) * d);
    if (!krot || !kbar) {
        free(krot); free(kbar);
        return ORACLE_ERR_NOMEM;
    }
    struct rotk_ctx rk = {k, seg_offsets, krot, d, base, interleaved, pos};
    parallel_for(nseg, nthreads, rotate_k_segment, &rk);
    struct sa_pool_ctx pc = {krot, seg_offsets, kbar, d, Bk};
    parallel_for(nseg, nthreads, sa_pool_segment, &pc);

    const int chunk = 64;
    long nitems = 0;
    for (int s = 0; s < nseg; ++s) nitems += (seg_offsets[s + 1] - seg_offsets[s] + chunk - 1) / chunk;
    long *item_seg = (long *)malloc(sizeof(long) * (size_t)(nitems > 0 ? nitems : 1));
    long *item_r0 = (long *)malloc(sizeof(long) * (size_t)(nitems > 0 ? nitems : 1));
    if (!item_seg || !item_r0) {
        free(item_seg); free(item_r0); free(krot); free(kbar);
        return ORACLE_ERR_NOMEM;
    }
    long it = 0;
    for (int s = 0; s < nseg; ++s)
        for (long r0 = 0; r0 < seg_offsets[s + 1] - seg_offsets[s]; r0 += chunk) {
            item_seg[it] = s;
            item_r0[it] = r0;
            ++it;
        }
    struct sa_ctx ctx = {q, v, krot, kbar, seg_offsets, row_src, gate, y, mask_in, mask_out, mask_words,
                         nseg, d, g, Bk, a_num, a_den, base, interleaved, pos, item_seg, item_r0, chunk,
                         ORACLE_OK};
    parallel_for(nitems, nthreads, sa_item, &ctx);
    free(item_seg); free(item_r0); free(krot); free(kbar);
    return ctx.status;
}

/*
 * oracle_sa_scores_rows: the fp64 block scores q~ . mean(k~ of block b), b < current block,
 * for chosen queries (the checks of a selection made elsewhere).
 *   rows [nrows] packed rows, heads [nrows] group heads; out [nrows, nblk_out], unused entries NaN
 */
int oracle_sa_scores_rows(const uint16_t *q, const uint16_t *k, int nseg, int d, int g, double base,
                          const int32_t *seg_offsets, int Bk, const int64_t *rows, const int32_t *heads, long nrows,
                          int nblk_out, double *out, int interleaved, const int64_t *pos)
{
    if (!q || !k || !seg_offsets || !rows || !heads || !out || Bk < 1 || nblk_out < 0) return ORACLE_ERR_ARG;
    long R = seg_offsets[nseg];
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    double *qr = (double *)malloc(sizeof(double) * (size_t)d);
    double *kr = (double *)malloc(sizeof(double) * (size_t)d);
    double *mean = (double *)malloc(sizeof(double) * (size_t)d);
    int st = (tmp && qr && kr && mean) ? ORACLE_OK : ORACLE_ERR_NOMEM;
    for (long i = 0; i < nrows && st == ORACLE_OK; ++i) {
        long row = rows[i];
        int j = heads[i];
        if (row < 0 || row >= R || j < 0 || j >= g) { st = ORACLE_ERR_ARG; break; }
        int lo = 0, hi = nseg;
        while (hi - lo > 1) {
            int mid = (lo + hi) / 2;
            if (seg_offsets[mid] <= row) lo = mid; else hi = mid;
        }
        long off = seg_offsets[lo], r = row - off, cur = r / Bk;
        for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(q[(row * g + j) * d + cc]);
        rope_rotate(tmp, d, pos ? (double)pos[row] : (double)r, base, interleaved, qr);
        for (long b = 0; b < nblk_out; ++b) out[i * nblk_out + b] = NAN;
        for (long b = 0; b < cur && b < nblk_out; ++b) {
            for (int cc = 0; cc < d; ++cc) mean[cc] = 0.0;
            for (long t = b * Bk; t < (b + 1) * Bk; ++t) {
                for (int cc = 0; cc < d; ++cc) tmp[cc] = bf16_to_double(k[(off + t) * d + cc]);
                rope_rotate(tmp, d, pos ? (double)pos[off + t] : (double)t, base, interleaved, kr);
                for (int cc = 0; cc < d; ++cc) mean[cc] += kr[cc];
            }
            double acc = 0.0;
            for (int cc = 0; cc < d; ++cc) acc += qr[cc] * (mean[cc] / (double)Bk);
            out[i * nblk_out + b] = acc;
        }
    }
    free(tmp); free(qr); free(kr); free(mean);
    return st;
}

/* Number of worker threads the oracle would use by default. */
int oracle_default_threads(void)
{
    long n = 1;
#ifdef _SC_NPROCESSORS_ONLN
    n = sysconf(_SC_NPROCESSORS_ONLN);
#endif
    return n > 0 ? (int)n : 1;
}
