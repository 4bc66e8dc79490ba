// sa_select.cuh -- the per-query block selection of SA + NAMOH (App. B.8, with the selection model of
// App. B.3, Eqs. app-block-budget and app-selected-entries): how one thread picks the kept blocks of its
// query from its row of block scores in TMEM.
//
// A query at one-based local rank r sees N_B(r) = ceil(r / block) blocks and keeps R(r) =
// ceil(alpha N_B(r)) of them: its current block and the R(r) - 1 completed blocks whose mean-pooled key
// scores highest against the query.  Each block's score is keyed by its fp32 value mapped to an
// order-preserving integer, with the low 10 bits replaced by 1023 - b: a larger key is a higher score,
// and scores equal to within the 10 dropped bits (2^-13 relative, far inside the bf16 rounding the
// inputs already carry) go to the lower block index.  Keys are unique, so "kept" is "key >= the k-th
// largest key".  With k = R(r) - 1 kept of the c = N_B(r) - 1 completed blocks, a thread finds the
// min(k, c - k)-th extreme key (of the kept set, or of the dropped one) with a sorted register list of
// 2, 4 or 8 entries (the shortest the warp's largest count allows) fed by a branch-free insertion
// network, or, past 8, by bisection over the 32-bit key range.
#pragma once

#include "common.cuh"

namespace namoh {
namespace sa {

constexpr int kListLen = 8;  // register list of the streaming selection

// Kept historical blocks of a query whose current block is `cur`: ceil(alpha (cur + 1)) - 1, exact.
__device__ __forceinline__ int kept_blocks(int cur, int alpha_num, int alpha_den) {
  return (int)(((long long)(cur + 1) * alpha_num + alpha_den - 1) / alpha_den) - 1;
}

// Selection key of block b with fp32 score s (see the file header).  -0 and +0 map alike.
__device__ __forceinline__ uint32_t score_key(float s, int b) {
  uint32_t u = __float_as_uint(s + 0.0f);
  u = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return (u & ~0x3FFu) | (uint32_t)(0x3FF - b);
}

// 16 block scores of this thread's row (TMEM lane), columns taddr .. taddr + 15.  The passes below
// walk the scores 16 columns at a time in a loop that is not unrolled, which keeps the code small
// (every CTA runs it once, from a cold instruction cache).
constexpr int kSelGroup = 16;
__device__ __forceinline__ void load_scores(uint32_t taddr, uint32_t (&r)[kSelGroup]) {
  tmem_ld16(taddr, r);
  tmem_wait_ld();
}

// The kx-th largest key (x = key ^ flip) among blocks 0 .. cand - 1 of this thread's row, kept in a
// sorted LL-entry register list fed by a branch-free insertion network; lanes with use = false
// take part in the warp-collective loads only.  LL >= every participating lane's kx.  The columns
// stop at the warp's largest candidate count.
template <int LL>
__device__ __forceinline__ uint32_t list_pass(uint32_t taddr, int cand, int kx, uint32_t flip, bool use) {
  uint32_t best[LL];
#pragma unroll
  for (int i = 0; i < LL; ++i) best[i] = 0u;
  const int wmax = (int)__reduce_max_sync(0xffffffffu, use ? (unsigned)cand : 0u);
#pragma unroll 1
  for (int g0 = 0; g0 < wmax; g0 += kSelGroup) {
    uint32_t v[kSelGroup];
    load_scores(taddr + (uint32_t)g0, v);
#pragma unroll
    for (int i = 0; i < kSelGroup; ++i) {
      const int b = g0 + i;
      uint32_t x = (use && b < cand) ? score_key(__uint_as_float(v[i]), b) ^ flip : 0u;
#pragma unroll
      for (int e = 0; e < LL; ++e) {  // insertion into the sorted list, branch-free
        const uint32_t hi = max(best[e], x);
        x = min(best[e], x);
        best[e] = hi;
      }
    }
  }
  uint32_t tau = 0xFFFFFFFFu;
#pragma unroll
  for (int e = 0; e < LL; ++e)
    if (use && e == kx - 1) tau = best[e];
  return tau;
}

// The kept blocks of one query from its row of block scores in TMEM (lane = this thread, columns
// taddr .. taddr + 32 nchunks - 1): candidates are blocks 0 .. cand - 1, `keep` of them are kept.
// emit(c, w) receives mask word c (bit i: block 32 c + i kept) for c = 0 .. nchunks - 1.
// Warp-collective: tcgen05.ld needs every lane of the warp, so every lane calls this with the same
// nchunks (a lane without a query passes cand = keep = 0) and the lanes' own work is predicated.
// Scores are read only below the warp's largest candidate count, which the caller's TMEM
// allocation covers.  The list is as short as the warp's largest kx allows (2, 4 or kListLen
// entries).
template <typename Emit>
__device__ __forceinline__ void select_from_tmem(uint32_t taddr, int nchunks, int cand, int keep, Emit&& emit) {
  const bool drop_mode = 2 * keep > cand;          // find the dropped blocks instead
  const int kx = drop_mode ? cand - keep : keep;   // extreme keys to find
  const uint32_t flip = drop_mode ? 0xFFFFFFFFu : 0u;
  const bool use_list = kx > 0 && kx <= kListLen;
  const int need = (int)__reduce_max_sync(0xffffffffu, use_list ? (unsigned)kx : 0u);
  uint32_t tau = 0xFFFFFFFFu;                      // the kx-th largest key (x = key ^ flip)
  if (need > 4) tau = list_pass<kListLen>(taddr, cand, kx, flip, use_list);
  else if (need > 2) tau = list_pass<4>(taddr, cand, kx, flip, use_list);
  else if (need > 0) tau = list_pass<2>(taddr, cand, kx, flip, use_list);
  if (__any_sync(0xffffffffu, kx > kListLen)) {
    // bisection for the lanes that need more than kListLen keys: the largest t with #{x >= t} >= kx,
    // which (keys unique) is the kx-th largest key
    const bool bis = kx > kListLen;
    const int wmax = (int)__reduce_max_sync(0xffffffffu, bis ? (unsigned)cand : 0u);
    uint32_t lo = 0u, hi = 0xFFFFFFFFu;
    for (int it = 0; it < 32; ++it) {
      const uint32_t mid = lo + ((hi - lo) >> 1) + ((hi - lo) & 1u);
      int cnt = 0;
#pragma unroll 1
      for (int g0 = 0; g0 < wmax; g0 += kSelGroup) {
        uint32_t v[kSelGroup];
        load_scores(taddr + (uint32_t)g0, v);
#pragma unroll
        for (int i = 0; i < kSelGroup; ++i) {
          const int b = g0 + i;
          cnt += (b < cand && (score_key(__uint_as_float(v[i]), b) ^ flip) >= mid) ? 1 : 0;
        }
      }
      if (lo < hi) {
        if (cnt >= kx) lo = mid;
        else hi = mid - 1u;
      }
    }
    if (bis) tau = lo;
  }
  // the mask: block b kept iff key >= tau (kept mode), ~key < tau (drop mode); the columns stop at
  // the warp's largest candidate count
  const int wmax = (int)__reduce_max_sync(0xffffffffu, keep > 0 ? (unsigned)cand : 0u);
#pragma unroll 1
  for (int c = 0; c < nchunks; ++c) {
    uint32_t w = 0u;
#pragma unroll
    for (int h = 0; h < 32 / kSelGroup; ++h) {
      const int g0 = c * 32 + h * kSelGroup;
      if (g0 >= wmax) break;
      uint32_t v[kSelGroup];
      load_scores(taddr + (uint32_t)g0, v);
#pragma unroll
      for (int i = 0; i < kSelGroup; ++i) {
        const int b = g0 + i;
        const uint32_t x = score_key(__uint_as_float(v[i]), b) ^ flip;
        const bool kept = b < cand && keep > 0 && (drop_mode ? x < tau : x >= tau);
        w |= (kept ? 1u : 0u) << (h * kSelGroup + i);
      }
    }
    emit(c, w);
  }
}

}  // namespace sa
}  // namespace namoh
