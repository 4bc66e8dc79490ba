/*
 * namoh.h -- C ABI of the NAMOH routed-attention path on GB300 (sm_103a).
 *
 * NAMOH (mixture-of-head native sparse attention): each token activates K of H
 * heads; each head runs causal attention only over the subsequence of tokens
 * routed to it, with RoPE applied at the token's rank inside that subsequence.
 *
 * Conventions shared by every entry point
 *   - All array arguments are DEVICE pointers to caller-owned memory, unless a
 *     comment says otherwise.  The library never allocates, frees or keeps
 *     device memory in these calls; scratch space is the caller's `workspace`
 *     (size from the matching *_workspace_size query, 256-byte aligned).
 *   - bf16 tensors are passed as `uint16_t*` (raw bf16 bit patterns), row-major,
 *     rows 16-byte aligned.
 *   - `stream` is a cudaStream_t passed as `void*` (NULL = legacy default
 *     stream).  Calls only enqueue work on it and return; they never
 *     synchronise the host.
 *   - Argument errors are detected on the host before any launch and return a
 *     negative namoh_status with nothing enqueued.  A launch failure returns
 *     NAMOH_ERR_CUDA.
 *   - Data-dependent conditions found on the device (non-finite router logits,
 *     a full KV segment, a wait that timed out) are OR-ed as NAMOH_DEV_* bits
 *     into the caller's device word `*dev_status`; read it after synchronising.
 *     Kernels never trap: the affected outputs are left unspecified.
 *   - Global state: only a lazily filled per-device cache of properties and the
 *     driver's tensor-map encoder; calls are thread-safe.
 *
 * Notation (the paper's): B sequences of T tokens; H routed query heads, K
 * active per token; d_head the head width; g query heads per KV group
 * (App. B.7 "Adopted KV-group routing"; g = 1 without grouping).  With grouping
 * the router selects Kr = K/g of Hr = H/g groups, and everything keyed by
 * "head" below is keyed by group.  R = B*T*Kr packed key/value rows.
 */
#ifndef NAMOH_H
#define NAMOH_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define NAMOH_API __attribute__((visibility("default")))
#else
#define NAMOH_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Host return codes. */
typedef enum namoh_status {
    NAMOH_OK = 0,
    NAMOH_ERR_INVALID_ARG = -1, /* a pointer, size or alignment violates the contract */
    NAMOH_ERR_UNSUPPORTED = -2, /* valid but not built: d_head, group, or the device */
    NAMOH_ERR_WORKSPACE = -3,   /* workspace NULL, misaligned or smaller than required */
    NAMOH_ERR_CUDA = -4         /* a CUDA runtime/driver call or a launch failed */
} namoh_status;

/* Bits OR-ed into *dev_status by the kernels. */
#define NAMOH_DEV_NONFINITE_SCORE 0x1u /* a router logit was NaN or infinite */
#define NAMOH_DEV_CAPACITY 0x2u        /* a KV segment had no room for its rows */
#define NAMOH_DEV_TIMEOUT 0x4u         /* a pipeline wait exceeded its limit; bits 16-23 then
                                          hold the barrier's index in its kernel's barrier block
                                          and bits 24-31 the warp that gave up */
#define NAMOH_DEV_BAD_SEQLENS 0x8u     /* cu_seqlens of a ragged batch was malformed */

/* RoPE variants (the rope_flags argument of the *_ex entry points; 0 = the defaults).
 * NAMOH_ROPE_INTERLEAVED  rotate pairs (2j, 2j+1) instead of the half-split (j, j + d/2);
 *                         theta_j = rope_base^(-2j/d) in both.
 * NAMOH_ROPE_GLOBAL       encode each token at its index t in its sequence instead of
 *                         its rank rho_i(t) (Sec. 3.2: global-position RoPE replaces
 *                         rho_i(t) by t).  Cache rows still follow the rank.
 * Prefill and decode over one cache must use the same flags. */
#define NAMOH_ROPE_INTERLEAVED 0x1u
#define NAMOH_ROPE_GLOBAL 0x2u

/* Limits of this build. */
#define NAMOH_MAX_HEADS 64 /* H (or Hr) routed units */

/* Human-readable text for a namoh_status value.  Host function. */
NAMOH_API const char *namoh_status_string(int status);

/* ABI version: (major << 16) | minor. */
NAMOH_API int namoh_version(void);

/* Detail of the last NAMOH_ERR_CUDA returned on the calling thread: which launch
 * or CUDA call failed and the CUDA error name and text.  Thread-local, valid
 * until the thread's next failing call.  Host function. */
NAMOH_API const char *namoh_last_error_string(void);

/* ------------------------------------------------------------------------- *
 * Routing and dispatch.
 * Sec. 3.1, Eq. (namoh-gates): a_t = softmax(x_t W_r), S_K(t) = TopK(a_t),
 *   g_{t,i} = m_{t,i} a_{t,i} (not renormalised over the selected heads).
 * Sec. 3.1: ordered index sets I_i = {t : m_{t,i} = 1}, lengths n_i.
 * Sec. 3.2, Eq. (namoh-head-rope): rho_i(t) = sum_{s<=t} m_{s,i} - 1.
 * Sec. 3.2 "Efficient execution": each (batch, head) subsequence is packed as
 *   one independent sequence.
 *
 * scores      [B, T, H] fp32 router logits x_t W_r.  Selection compares these
 *             exactly (softmax is monotone); ties go to the lower head index.
 * topk_head   [B, T, K] int32 out: selected heads in descending score order
 *             ("slots"); every per-slot array below follows this order.
 * gate        [B, T, K] fp32 out: softmax over all H logits at the selected heads.
 * The remaining outputs form the packed layout; pass all four, or all four
 * NULL to skip it (e.g. when routing one decode token):
 * rank        [B, T, K] int32 out: rho of (t, slot) inside its (b, head) segment.
 * row         [B, T, K] int32 out: packed row = seg_offsets[b*H + head] + rank.
 * seg_offsets [B*H + 1] int32 out: exclusive prefix sum of n over (b, head)
 *             order; seg_offsets[B*H] = B*T*K.  Rows ascend in t in a segment.
 * row_src     [B*T*K]   int32 out: inverse of row: row_src[row] = (b*T + t)*K + slot.
 * Requires 1 <= K <= H <= NAMOH_MAX_HEADS, B >= 1, T >= 1, B*T*K < 2^31.
 * Non-finite logits set NAMOH_DEV_NONFINITE_SCORE (that token's outputs are
 * unspecified but in range).  Integer outputs are deterministic.
 * The packed layout takes two kernel launches (three when ceil(T/256)*H exceeds
 * 4096), chained by programmatic dependent launch: the first touches no global
 * memory before the work ahead of it in the stream has completed.  Every path
 * gives identical results.
 * ------------------------------------------------------------------------- */
NAMOH_API size_t namoh_route_workspace_size(int B, int T, int H, int K);
NAMOH_API int namoh_route(const float *scores, int B, int T, int H, int K, int32_t *topk_head, float *gate,
                int32_t *rank, int32_t *row, int32_t *seg_offsets, int32_t *row_src, void *workspace,
                size_t workspace_bytes, uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * namoh_route_biased: routing with loss-free balancing biases (App. A,
 *   Eq. namoh-biased-routing): S_K(t) = TopK_i(a_{t,i} + b_i) on the softmax
 *   affinities plus a per-head bias, ties to the lower head index; the gates stay
 *   g_{t,i} = a_{t,i} (the bias does not enter them, no renormalisation).
 * bias  [H] fp32 device array, finite, caller-owned, read-only; NULL gives
 *       exactly namoh_route.
 * Everything else (arguments, outputs, layout, errors) is as namoh_route.  The
 * affinities are fp32 (exp2 of pre-scaled logit differences), so where two
 * biased affinities lie within a few fp32 ulps of each other the order between
 * them is the fp32 one.
 * ------------------------------------------------------------------------- */
NAMOH_API int namoh_route_biased(const float *scores, const float *bias, int B, int T, int H, int K,
                                 int32_t *topk_head, float *gate, int32_t *rank, int32_t *row, int32_t *seg_offsets,
                                 int32_t *row_src, void *workspace, size_t workspace_bytes, uint32_t *dev_status,
                                 void *stream);

/* ------------------------------------------------------------------------- *
 * namoh_route_varlen: routing of a ragged batch (sequences of different lengths
 *   packed back to back, no padding).  Sequence b holds the tokens
 *   cu_seqlens[b] .. cu_seqlens[b+1]-1 of the flat token axis; ranks, index sets
 *   and segments are per sequence exactly as in namoh_route (Sec. 3.1, Sec. 3.2).
 * scores      [total_tokens, H] fp32.
 * cu_seqlens  [B + 1] int32 device array: 0 = cu_seqlens[0] <= ... <=
 *             cu_seqlens[B] = total_tokens, every length <= max_seqlen (empty
 *             sequences are allowed).  A violation found on the device sets
 *             NAMOH_DEV_BAD_SEQLENS; the outputs are then unspecified but stay a
 *             layout of rows below total_tokens*K, so later stages stay in bounds.
 * bias        [H] or NULL: as namoh_route_biased.
 * topk_head, gate, rank, row [total_tokens, K]; seg_offsets [B*H + 1] with
 *             seg_offsets[B*H] = total_tokens*K; row_src [total_tokens*K] with
 *             row_src[row] = tok*K + slot, tok on the flat axis.  The packed layout
 *             is optional as in namoh_route (without it cu_seqlens is not read).
 * Workspace: namoh_route_workspace_size(B, max_seqlen, H, K).
 * Requires 1 <= max_seqlen <= total_tokens, total_tokens*K < 2^31.
 * ------------------------------------------------------------------------- */
NAMOH_API int namoh_route_varlen(const float *scores, const float *bias, const int32_t *cu_seqlens, int B,
                                 int total_tokens, int max_seqlen, int H, int K, int32_t *topk_head, float *gate,
                                 int32_t *rank, int32_t *row, int32_t *seg_offsets, int32_t *row_src,
                                 void *workspace, size_t workspace_bytes, uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * namoh_route_noalloc: namoh_route without a workspace argument.
 * The paper has no counterpart; this is a convenience of this library.
 *
 * For callers that cannot allocate device memory around the call: code running
 * inside a stream capture (cudaMalloc/cudaFree are not capturable and may
 * synchronise the device), latency-critical serving loops that must never
 * synchronise, and runtimes that own every byte of device memory through their
 * own pools and forbid side allocations.  The scratch that namoh_route takes
 * from `workspace` comes instead from a 4 MiB array compiled into the library
 * (every GPU that loads the library holds it until the process exits).
 *
 * Arguments, outputs and rules are those of namoh_route.  Shapes whose
 * namoh_route_workspace_size exceeds 4 MiB return NAMOH_ERR_WORKSPACE with
 * nothing enqueued (e.g. B*ceil(T/256)*H <= about 500000 fits).  The call
 * allocates nothing.  The first call on each device resolves the array's device
 * address (cudaGetSymbolAddress) with that device current; make that first call
 * before any stream capture.  Every call on a device shares the one array and
 * leaves its last contents there; every word of it is written before it is
 * read.  Calls that overlap on the GPU -- on
 * different streams, or from different host threads -- race on it and must be
 * serialised by the caller.  The resolved address is kept for the life of the
 * process: after cudaDeviceReset (or anything else that destroys and recreates
 * the device's primary context) it is stale, so do not call this entry point on
 * a device that has been reset since its first call.
 * ------------------------------------------------------------------------- */
NAMOH_API int namoh_route_noalloc(const float *scores, int B, int T, int H, int K, int32_t *topk_head, float *gate,
                                  int32_t *rank, int32_t *row, int32_t *seg_offsets, int32_t *row_src,
                                  uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * Prefill: head-relative RoPE, routed causal attention, gate-weighted combine.
 * Sec. 3.2, Eq. (namoh-head-rope): q~ = q R(rho), k~ = k R(rho), half-split
 *   pairs (j, j + d/2), theta_j = rope_base^(-2j/d).
 * Sec. 3.1, Eq. (namoh-attention): h_{t,i} = softmax(q~ k~^T / sqrt(d)) v over
 *   s in I_i, s <= t; the combine writes the per-slot term g_{t,i} h_{t,i}
 *   (the W_O projection is outside this path).
 * App. B.7 "Adopted KV-group routing": the g query heads of a group share its
 *   keys, values, gate and rank.
 * Sec. 3.2 "Efficient execution": length-aware scheduling of query tiles.
 *
 * q           [R*g, d] bf16: query of packed row r and group head j at row r*g + j.
 * k, v        [R, d]   bf16: packed rows in segment order (as produced by the
 *             routing above with H = Hr, K = Kr).
 * seg_offsets [B*Hr + 1], row_src [R], gate [R] (indexed by row_src value):
 *             namoh_route outputs for the Hr-way routing.
 * y           [B, T, K, d] bf16 out (= [B, T, Kr, g, d]): g_{t,i} h_{t,i} per slot.
 * k_cache     out: rotated keys k~ (bf16, d per row); v_cache out: values.
 * seg_base    NULL: the caches are packed like k/v ([R, d]); v_cache may then
 *             equal v (no copy).  Otherwise [B*Hr] int64 first cache row of
 *             each segment, with seg_cap [B*Hr] int32 its capacity in rows and
 *             cache_rows the rows allocated in each cache (for bounds); a
 *             segment longer than its capacity sets NAMOH_DEV_CAPACITY and its
 *             rows and outputs are skipped.
 * seg_len     NULL or [B*Hr] int32 out: n of each segment (decode state).
 * Supports d_head in {64, 128}, g in {1, 2, 4, 8}, rope_base > 1, T <= 2^20.
 * k_cache must not alias k.  Runs the three stages below in order.
 * ------------------------------------------------------------------------- */
NAMOH_API size_t namoh_prefill_workspace_size(int B, int T, int H, int K, int d_head, int group);
NAMOH_API int namoh_prefill(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int T, int H, int K,
                  int d_head, int group, float rope_base, const int32_t *seg_offsets, const int32_t *row_src,
                  const float *gate, uint16_t *y, uint16_t *k_cache, uint16_t *v_cache, const int64_t *seg_base,
                  const int32_t *seg_cap, int64_t cache_rows, int32_t *seg_len, void *workspace,
                  size_t workspace_bytes, uint32_t *dev_status, void *stream);
/* namoh_prefill_ex: namoh_prefill with rope_flags (NAMOH_ROPE_*; unknown bits are
 * NAMOH_ERR_INVALID_ARG).  Under NAMOH_ROPE_GLOBAL the position of packed row r is
 * t = (row_src[r] / Kr) % T.  namoh_prefill is namoh_prefill_ex with rope_flags = 0. */
NAMOH_API int namoh_prefill_ex(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int T, int H, int K,
                               int d_head, int group, float rope_base, unsigned rope_flags,
                               const int32_t *seg_offsets, const int32_t *row_src, const float *gate, uint16_t *y,
                               uint16_t *k_cache, uint16_t *v_cache, const int64_t *seg_base,
                               const int32_t *seg_cap, int64_t cache_rows, int32_t *seg_len, void *workspace,
                               size_t workspace_bytes, uint32_t *dev_status, void *stream);

/* namoh_prefill_varlen: namoh_prefill_ex over a ragged batch routed by
 * namoh_route_varlen.  total_tokens and max_seqlen are the host's copies of
 * cu_seqlens[B] and the longest length; R = total_tokens * Kr; y is
 * [total_tokens, K, d].  cu_seqlens ([B + 1], device) is read only for
 * NAMOH_ROPE_GLOBAL, where the position of a row is its token's index inside its
 * own sequence.  Workspace: namoh_prefill_varlen_workspace_size.  Requires
 * 1 <= max_seqlen <= min(total_tokens, 2^20).  The staged calls below are for
 * fixed-length batches only. */
NAMOH_API size_t namoh_prefill_varlen_workspace_size(int B, int total_tokens, int max_seqlen, int H, int K,
                                                     int d_head, int group);
NAMOH_API int namoh_prefill_varlen(const uint16_t *q, const uint16_t *k, const uint16_t *v, const int32_t *cu_seqlens,
                                   int B, int total_tokens, int max_seqlen, int H, int K, int d_head, int group,
                                   float rope_base, unsigned rope_flags, const int32_t *seg_offsets,
                                   const int32_t *row_src, const float *gate, uint16_t *y, uint16_t *k_cache,
                                   uint16_t *v_cache, const int64_t *seg_base, const int32_t *seg_cap,
                                   int64_t cache_rows, int32_t *seg_len, void *workspace, size_t workspace_bytes,
                                   uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * The three stages of namoh_prefill, callable one by one (same arguments and
 * rules as namoh_prefill unless stated).
 *
 * namoh_rope_pack (Sec. 3.2, Eq. namoh-head-rope): rotates every query row to
 *   its rank into q_rot [R*g, d] bf16 (caller-owned), writes k~ to k_cache and
 *   copies v to v_cache (unless v_cache == v, allowed only without seg_base).
 *   plan: NULL, or a buffer as namoh_attention_plan takes (plan_bytes long); the
 *   same launch then also writes the plan that namoh_attention_plan would write
 *   with seg_cap (or NULL when seg_base is NULL), saving one kernel launch.
 *
 * namoh_attention_plan (Sec. 3.2 "Efficient execution", length-aware
 *   scheduling): writes into `plan` (namoh_attention_plan_size bytes, 16-byte
 *   aligned, caller-owned) the list of 128-row query tiles of every segment and
 *   group head, longest causal workload first.  Segments longer than seg_cap
 *   (when seg_cap is not NULL) are left out.  A plan depends only on
 *   seg_offsets and may be reused by any number of namoh_attention calls on the
 *   same stream; two calls must not use one plan concurrently.
 *
 * namoh_attention (Sec. 3.1, Eq. namoh-attention and the combine): one
 *   persistent kernel (one CTA per SM) that takes tiles from the plan longest
 *   first and writes y = g_{t,i} h_{t,i}.  k_cache / v_cache hold k~ and v at
 *   seg_base (or packed rows when seg_base is NULL).
 * ------------------------------------------------------------------------- */
NAMOH_API int namoh_rope_pack(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int T, int H, int K,
                              int d_head, int group, float rope_base, const int32_t *seg_offsets, uint16_t *q_rot,
                              uint16_t *k_cache, uint16_t *v_cache, const int64_t *seg_base, const int32_t *seg_cap,
                              int64_t cache_rows, uint32_t *dev_status, void *plan, size_t plan_bytes,
                              void *stream);
/* namoh_rope_pack_ex: namoh_rope_pack with rope_flags (NAMOH_ROPE_*) and row_src
 * ([R] int32, the routing's inverse map; read only under NAMOH_ROPE_GLOBAL, where it
 * must not be NULL). */
NAMOH_API int namoh_rope_pack_ex(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int T, int H,
                                 int K, int d_head, int group, float rope_base, unsigned rope_flags,
                                 const int32_t *seg_offsets, const int32_t *row_src, uint16_t *q_rot,
                                 uint16_t *k_cache, uint16_t *v_cache, const int64_t *seg_base,
                                 const int32_t *seg_cap, int64_t cache_rows, uint32_t *dev_status, void *plan,
                                 size_t plan_bytes, void *stream);
NAMOH_API size_t namoh_attention_plan_size(int B, int T, int H, int K, int group);
NAMOH_API int namoh_attention_plan(const int32_t *seg_offsets, int B, int T, int H, int K, int group,
                                   const int32_t *seg_cap, void *plan, size_t plan_bytes, void *stream);
NAMOH_API int namoh_attention(const uint16_t *q_rot, const uint16_t *k_cache, const uint16_t *v_cache, int B, int T,
                              int H, int K, int d_head, int group, const int32_t *seg_offsets, const int32_t *row_src,
                              const float *gate, const int64_t *seg_base, int64_t cache_rows, void *plan,
                              size_t plan_bytes, uint16_t *y, uint32_t *dev_status, void *stream);

/* namoh_attention_timeout_probe: a check of the kernels' bounded waits, for tests (no
 * counterpart in the paper).  Every wait of the attention kernel gives up after a limit
 * (2 s), reports NAMOH_DEV_TIMEOUT and lets every role drain and exit, so that a stalled
 * pipeline returns an error instead of hanging the GPU.  This call runs namoh_attention
 * (packed caches, seg_base NULL) with the first query tile of every CTA withheld: the
 * MMA issuer's wait for it runs out after wait_limit_ns (1 us .. 2 s) and sets in
 * *dev_status NAMOH_DEV_TIMEOUT, bits 16-22 = 4 (the query tile's barrier, the fifth
 * word of the kernel's barrier block) and bits 24-31 = 5 (the MMA issuer's warp).  y is
 * left unspecified; the plan and the context stay usable.  Argument errors as
 * namoh_attention, plus NAMOH_ERR_INVALID_ARG for a limit out of range. */
NAMOH_API int namoh_attention_timeout_probe(const uint16_t *q_rot, const uint16_t *k_cache, const uint16_t *v_cache,
                                            int B, int T, int H, int K, int d_head, int group,
                                            const int32_t *seg_offsets, const int32_t *row_src, const float *gate,
                                            void *plan, size_t plan_bytes, uint16_t *y, uint64_t wait_limit_ns,
                                            uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * Decode: one new token per sequence.
 * Sec. 3.1 (last paragraph): the token appends to and attends within only its
 *   selected heads' caches; prefill and incremental decoding are the same
 *   causal computation.  Sec. 3.2: the new token's rank is the current length.
 * Sec. 3.2 "Efficient execution": only active head queries run and only their
 *   caches are read or updated.
 *
 * topk_head, gate [B, Kr]: routing of the new tokens (namoh_route with T = 1).
 * q [B, K, d], k [B, Kr, d], v [B, Kr, d] bf16: projections of the new tokens
 *   for the selected (group) heads, in slot order.
 * For each (b, slot) with head h, segment s = b*Hr + h, rho = seg_len[s]:
 *   k~ = k R(rho) and v are written at cache row seg_base[s] + rho, every q of
 *   the group is rotated to rho and attends over the rho + 1 rows, and
 *   y[b, slot*g + j] = gate * h; finally seg_len[s] = rho + 1.
 * A full segment (rho >= seg_cap[s]) sets NAMOH_DEV_CAPACITY; its y is zero
 *   and its length is unchanged.
 * Supports d_head in {64, 128}, g in {1, 2, 4, 8}.
 * ------------------------------------------------------------------------- */
NAMOH_API size_t namoh_decode_workspace_size(int B, int H, int K, int d_head, int group);
NAMOH_API int namoh_decode(const int32_t *topk_head, const float *gate, const uint16_t *q, const uint16_t *k,
                 const uint16_t *v, int B, int H, int K, int d_head, int group, float rope_base,
                 uint16_t *k_cache, uint16_t *v_cache, const int64_t *seg_base, int32_t *seg_len,
                 const int32_t *seg_cap, int64_t cache_rows, uint16_t *y, void *workspace,
                 size_t workspace_bytes, uint32_t *dev_status, void *stream);
/* namoh_decode_ex: namoh_decode with rope_flags (NAMOH_ROPE_*) and token_pos ([B]
 * int64, the new tokens' indices in their sequences, each in [0, 2^24)): NULL unless
 * NAMOH_ROPE_GLOBAL is set, and required when it is.  The new token is then rotated
 * to token_pos[b]; its cache row is still seg_base[s] + rho. */
NAMOH_API int namoh_decode_ex(const int32_t *topk_head, const float *gate, const uint16_t *q, const uint16_t *k,
                              const uint16_t *v, int B, int H, int K, int d_head, int group, float rope_base,
                              unsigned rope_flags, const int64_t *token_pos, uint16_t *k_cache, uint16_t *v_cache,
                              const int64_t *seg_base, int32_t *seg_len, const int32_t *seg_cap, int64_t cache_rows,
                              uint16_t *y, void *workspace, size_t workspace_bytes, uint32_t *dev_status,
                              void *stream);

/* ------------------------------------------------------------------------- *
 * Shared heads: the paper's shared-head variant (Sec. 4.4, "Shared heads for local
 * context"): Hs always-active heads, outside the routing, each attending to the full
 * causal prefix (window = 0) or to the most recent `window` tokens including the current
 * one, with RoPE at the token's global position and no gate.  Their outputs are summed
 * into o by the caller's projection, like the routed heads'.
 *
 * namoh_shared_prefill
 *   q, k, v     [B, Hs, T, d] bf16 (each head's sequence contiguous).
 *   y           [B, T, Hs, d] bf16 out: h of every (token, shared head).
 *   k_cache, v_cache, seg_base, seg_cap, cache_rows, seg_len: as namoh_prefill, segment
 *               (b, j) = shared head j of sequence b (B*Hs segments of T rows).
 *   rope_flags  NAMOH_ROPE_INTERLEAVED or 0 (positions are global already).
 *   Workspace: namoh_shared_workspace_size.  Supports d_head in {64, 128}, T <= 2^20.
 * namoh_shared_decode: one new token per sequence for every shared head: q, k, v and y
 *   [B, Hs, d]; appends k~ (at position seg_len, which is t) and v, attends over the last
 *   min(seg_len + 1, window) rows (all of them when window = 0), seg_len += 1.
 *   Workspace: namoh_shared_decode_workspace_size.
 * ------------------------------------------------------------------------- */
NAMOH_API size_t namoh_shared_workspace_size(int B, int T, int Hs, int d_head);
NAMOH_API int namoh_shared_prefill(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int T, int Hs,
                                   int d_head, int window, float rope_base, unsigned rope_flags, uint16_t *y,
                                   uint16_t *k_cache, uint16_t *v_cache, const int64_t *seg_base,
                                   const int32_t *seg_cap, int64_t cache_rows, int32_t *seg_len, void *workspace,
                                   size_t workspace_bytes, uint32_t *dev_status, void *stream);
NAMOH_API size_t namoh_shared_decode_workspace_size(int B, int Hs, int d_head);
NAMOH_API int namoh_shared_decode(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int Hs, int d_head,
                                  int window, float rope_base, unsigned rope_flags, uint16_t *k_cache,
                                  uint16_t *v_cache, const int64_t *seg_base, int32_t *seg_len,
                                  const int32_t *seg_cap, int64_t cache_rows, uint16_t *y, void *workspace,
                                  size_t workspace_bytes, uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * SA + NAMOH: block-selected sparse attention inside each routed history (App. B.8
 * "SA+NAMOH", with the selection model of App. B.3 "Block-Selected Sparse Attention",
 * Eqs. app-block-budget and app-selected-entries).  The routed history of each (batch,
 * head) is cut into blocks of `block` entries in its local order.  A query at one-based
 * local rank r keeps R(r) = ceil(alpha * ceil(r / block)) blocks, alpha = alpha_num /
 * alpha_den in (0, 1] (computed exactly): its current block, attended causally, and the
 * R(r) - 1 completed earlier blocks whose mean-pooled rotated key k~ has the largest dot
 * product with its rotated query q~ (fp32 scores; ties to the lower block index).  It then
 * attends over the entries of the kept blocks; the gate-weighted combine is namoh_prefill's.
 * alpha = 1 keeps every block (dense routed attention).
 *
 * namoh_sa_prefill
 *   Arguments as namoh_prefill_ex (routing outputs, caches, seg_len, workspace), plus:
 *   block       32, 64 or 128 keys per block; ceil(T / block) <= 1024.
 *   alpha_num, alpha_den  1 <= alpha_num <= alpha_den.
 *   sa_mask     [R*g, namoh_sa_mask_words(T, block)] uint32 out, 4-byte aligned: the kept
 *               earlier blocks of query (packed row r, group head j) at row r*g + j, bit
 *               b % 32 of word b / 32 for block b (the current block is implied).
 *   Workspace: namoh_sa_prefill_workspace_size (the rotated queries q~ [R*g, d] bf16, which the
 *   selection reads, the plan, and the pooled keys, (R / block + B*H/g) * d_head bf16).
 *   The block scores of each 128-query tile run on the tensor cores (bf16 q~ and pooled keys,
 *   fp32 sums); scores within 2^-13 of each other (relative) count as tied, ties to the lower
 *   block.  The attention does every causal key tile and masks the blocks not kept: the cost
 *   is that of namoh_prefill plus the selection.  Rows of a segment longer than its seg_cap
 *   are neither pooled nor attended; their sa_mask rows are zero.
 * namoh_sa_mask_words: words per query of sa_mask (0 for an unsupported block).
 * Errors: NAMOH_ERR_INVALID_ARG for an unsupported block or alpha, a null sa_mask, or the
 * argument errors of namoh_prefill_ex.
 * ------------------------------------------------------------------------- */
NAMOH_API int namoh_sa_mask_words(int T, int block);
NAMOH_API size_t namoh_sa_prefill_workspace_size(int B, int T, int H, int K, int d_head, int group, int block);
NAMOH_API int namoh_sa_prefill(const uint16_t *q, const uint16_t *k, const uint16_t *v, int B, int T, int H, int K,
                               int d_head, int group, float rope_base, unsigned rope_flags,
                               const int32_t *seg_offsets, const int32_t *row_src, const float *gate, int block,
                               int alpha_num, int alpha_den, uint32_t *sa_mask, uint16_t *y, uint16_t *k_cache,
                               uint16_t *v_cache, const int64_t *seg_base, const int32_t *seg_cap,
                               int64_t cache_rows, int32_t *seg_len, void *workspace, size_t workspace_bytes,
                               uint32_t *dev_status, void *stream);

/* ------------------------------------------------------------------------- *
 * The projections around the path (the full attention layer).
 * Sec. 3.1, Eq. (namoh-qkv): only an active token-head pair projects,
 *   q_{t,i} = x_t W_Q^(i), k_{t,i} = x_t W_K^(i), v_{t,i} = x_t W_V^(i), t in I_i.
 * Sec. 3.1, Eq. (namoh-attention): o_t = sum_{i in S_K(t)} g_{t,i} h_{t,i} W_O^(i).
 * App. B.7: a KV group projects one key, one value and g queries (one per query head).
 * Both run as one grouped GEMM over the packed rows of the routing (tcgen05 tiles of 128
 * rows, the A rows gathered from the token axis by 16-byte cp.async copies, the weight
 * tiles loaded by TMA), so they follow namoh_route or
 * namoh_route_varlen directly: seg_offsets [B*Hr + 1] and row_src [R] are its outputs,
 * R = total_tokens * Kr (total_tokens = B*T for a fixed-length batch).
 *
 * namoh_proj_qkv
 *   x      [total_tokens, d_model] bf16 token representations.
 *   w_qkv  [Hr, (g+2) d, d_model] bf16, one block per KV group i: rows j d .. j d + d - 1
 *          hold W_Q of query head i g + j transposed (row c = column c of W_Q), then d rows
 *          of W_K^(i) transposed, then d rows of W_V^(i) transposed.
 *   q [R*g, d], k [R, d], v [R, d] bf16 out: exactly namoh_prefill's inputs.
 * namoh_proj_out
 *   y      [total_tokens, K, d] bf16: namoh_prefill's output (per-slot g h).
 *   w_o    [Hr, d_model, g d] bf16, one block per group: row m holds column m of W_O of the
 *          group's query heads one after the other (W_O^(i g + j) row c at column j d + c).
 *   o      [total_tokens, d_model] fp32 out; accumulate = 0 overwrites it, 1 adds to it
 *          (e.g. onto a residual).  Two passes: each packed row's product with its group's
 *          W_O is rounded to bf16 into the workspace at its token-slot row, then each token's K
 *          rows are summed in slot order in fp32 (deterministic, no atomics).
 * Workspace: namoh_proj_workspace_size (one size serves both calls: the list of 128-row
 * tiles of the segments, plus the per-slot products of the output projection,
 * total_tokens*K/g*d_model bf16).
 * Supports d_head in {64, 128}, g in {1, 2, 4, 8}, d_model a multiple of 64 up to 65536, and
 * B*(H/g + 1) <= 51200.
 * x, w, q, k, v, y, o 16-byte aligned.  Rows of an inconsistent layout (a malformed
 * cu_seqlens) are computed from clamped indices and write nothing outside the outputs.
 * ------------------------------------------------------------------------- */
NAMOH_API size_t namoh_proj_workspace_size(int B, int total_tokens, int d_model, int H, int K, int group);
NAMOH_API int namoh_proj_qkv(const uint16_t *x, int total_tokens, int d_model, const uint16_t *w_qkv, int B, int H,
                             int K, int d_head, int group, const int32_t *seg_offsets, const int32_t *row_src,
                             uint16_t *q, uint16_t *k, uint16_t *v, void *workspace, size_t workspace_bytes,
                             uint32_t *dev_status, void *stream);
NAMOH_API int namoh_proj_out(const uint16_t *y, int total_tokens, int d_model, const uint16_t *w_o, int B, int H,
                             int K, int d_head, int group, const int32_t *seg_offsets, const int32_t *row_src,
                             float *o, int accumulate, void *workspace, size_t workspace_bytes,
                             uint32_t *dev_status, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* NAMOH_H */
