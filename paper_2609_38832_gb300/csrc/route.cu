// route.cu -- routing and dispatch (Sec. 3.1 Eq. namoh-gates; Sec. 3.2 Eq. namoh-head-rope).
//
// Every token selects exactly K heads, so sequence b's rows start at (its first token)*K --
// b*T*K, or cu_seqlens[b]*K in a ragged batch -- and each sequence's segment offsets depend
// only on that sequence's own head counts.
//
// The packed layout takes two launches, chained by programmatic dependent launch (the
// second is resident and waiting before the first ends):
//   1. route_local_kernel  one block per 256-token chunk, one thread per token: TopK of the
//                          fp32 logits (descending, ties to the lower head index), fp32
//                          softmax gates over all H, the chunk's head counts, and each
//                          (token, slot)'s rank among the chunk's earlier tokens for its head
//                          (warp ballots; written to `rank` for the second pass).
//   2. route_final_kernel  one block per chunk: sums its sequence's chunk-count table (chunk
//                          base per head, n[b, h], segment offsets), then the final rank, row
//                          and row_src of its tokens.
// When the count tables are large (many chunks x heads) a third launch between the two,
// route_scan_kernel (one block per sequence), scans them once and the final pass reads the
// chunk bases.  Without the packed layout (e.g. one decode token) only route_topk_kernel runs.
// All integer work is exact, so the packed layout is deterministic and bit-identical to
// a sequential append in token order, on either path.
#include <float.h>

#include <mutex>
#include <type_traits>

#include "common.cuh"

namespace namoh {
namespace {

constexpr int kChunk = 256;  // tokens per block in the top-K and rank kernels

constexpr float kLog2e = 1.4426950408889634f;

// Token range [start, start + len) of sequence b: b*T and T, or from cu_seqlens in a ragged
// batch (T = the longest sequence then).  A malformed cu_seqlens entry (decreasing, outside
// [0, total], cu_seqlens[0] != 0, cu_seqlens[B] != total, or longer than T) clears `ok`; the
// range is clamped into [0, total] and to T tokens, so every access stays inside the arrays.
struct SeqRange {
  int start, len;
  bool ok;
};
__device__ __forceinline__ SeqRange seq_range(const int32_t* __restrict__ cu, int b, int B, int T, int total) {
  if (!cu) return {b * T, T, true};
  int s0 = __ldg(cu + b), s1 = __ldg(cu + b + 1);
  const bool ok = s0 >= 0 && s1 >= s0 && s1 <= total && s1 - s0 <= T && (b > 0 || s0 == 0) &&
                  (b < B - 1 || s1 == total);
  s0 = min(max(s0, 0), total);
  s1 = min(max(s1, s0), total);
  s1 = min(s1, s0 + T);
  return {s0, s1 - s0, ok};
}

// The H logits of token `tok` in registers (independent loads, all in flight together).
// Non-finite logits become -FLT_MAX and set `bad`.
template <int HMAX>
__device__ __forceinline__ void load_logits(const float* __restrict__ scores, size_t tok, int H, float (&sc)[HMAX],
                                            bool& bad) {
  const float* src = scores + tok * H;
  if ((H & 3) == 0 && (reinterpret_cast<uintptr_t>(src) & 15u) == 0) {
#pragma unroll
    for (int h4 = 0; h4 < HMAX / 4; ++h4) {
      float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
      if (h4 * 4 < H) x = __ldg(reinterpret_cast<const float4*>(src) + h4);
      sc[4 * h4 + 0] = x.x;
      sc[4 * h4 + 1] = x.y;
      sc[4 * h4 + 2] = x.z;
      sc[4 * h4 + 3] = x.w;
    }
  } else {
#pragma unroll
    for (int h = 0; h < HMAX; ++h) sc[h] = (h < H) ? __ldg(src + h) : 0.f;
  }
  // one sum decides whether any logit needs looking at (it is non-finite when one is, or on
  // overflow, where the per-logit check then finds nothing to replace)
  uint64_t total2 = 0ull;
#pragma unroll
  for (int h = 0; h < HMAX; h += 2)
    total2 = f2_add(total2, f2_pack(h < H ? sc[h] : 0.f, h + 1 < H ? sc[h + 1] : 0.f));
  float ta, tb;
  f2_unpack(total2, ta, tb);
  const float total = ta + tb;
  bad = false;
  if (!isfinite(total)) {
#pragma unroll
    for (int h = 0; h < HMAX; ++h) {
      if (h < H && !isfinite(sc[h])) {
        bad = true;
        sc[h] = -FLT_MAX;
      }
    }
  }
}

// Softmax normaliser over all H logits (Sec. 3.1 Eq. namoh-gates), fp32: the max and
// 1 / sum_h exp(sc_h - max), each exponential as exp2((sc_h - max) * log2 e).
// The subtract and scale run on fp32 pairs (f32x2), each lane rounded as the scalar form
// would be; even heads sum into one partial and odd heads into the other.
template <int HMAX>
__device__ __forceinline__ void softmax_norm(const float (&sc)[HMAX], int H, float& mx, float& inv_z) {
  mx = -FLT_MAX;
#pragma unroll
  for (int h = 0; h < HMAX; h += 2)
    mx = fmax3(mx, h < H ? sc[h] : -FLT_MAX, h + 1 < H ? sc[h + 1] : -FLT_MAX);
  const uint64_t nmx2 = f2_pack(-mx, -mx), l2e2 = f2_pack(kLog2e, kLog2e);
  uint64_t z2 = 0ull;
#pragma unroll
  for (int h = 0; h < HMAX; h += 2) {
    if (h < H) {
      float x0, x1;
      f2_unpack(f2_mul(f2_add(f2_pack(sc[h], h + 1 < H ? sc[h + 1] : mx), nmx2), l2e2), x0, x1);
      z2 = f2_add(z2, f2_pack(fast_exp2(x0), h + 1 < H ? fast_exp2(x1) : 0.f));
    }
  }
  float z0, z1;
  f2_unpack(z2, z0, z1);
  inv_z = 1.0f / (z0 + z1);
}

// Top-K in registers: insertion into a list kept in (score desc, index asc) order.  Heads
// arrive in increasing index, so a head displaces only strictly smaller scores.  Empty
// entries hold -inf, which every (finite) logit beats; entries past K are scratch.
template <int HMAX, int KMAX>
__device__ __forceinline__ void topk_sorted(const float (&sc)[HMAX], int H, int (&hk)[KMAX], float (&vk)[KMAX]) {
#pragma unroll
  for (int k = 0; k < KMAX; ++k) {
    hk[k] = 0;
    vk[k] = -INFINITY;
  }
#pragma unroll
  for (int h = 0; h < HMAX; ++h) {
    if (h < H) {
      const float x = sc[h];
      bool beats[KMAX];
#pragma unroll
      for (int k = 0; k < KMAX; ++k) beats[k] = x > vk[k];
      // entry k takes entry k-1 when x beats that too, else x when x beats entry k
#pragma unroll
      for (int k = KMAX - 1; k >= 1; --k) {
        vk[k] = beats[k - 1] ? vk[k - 1] : (beats[k] ? x : vk[k]);
        hk[k] = beats[k - 1] ? hk[k - 1] : (beats[k] ? h : hk[k]);
      }
      vk[0] = beats[0] ? x : vk[0];
      hk[0] = beats[0] ? h : hk[0];
    }
  }
}

// Top-4 (score desc, index asc) with few instructions per head, for K <= 4:
//   1. the four largest values as a multiset, by a min / max insertion chain (no indices);
//   2. the heads at or above the fourth value t3, in ascending index order: every head above t3
//      (exactly as many as there are values above t3 in the multiset), then heads equal to t3 in
//      index order until four -- ties go to the lower index;
//   3. a stable sort of the four picks by value, descending (equal values keep index order).
// Entries past H (H < 4) hold head 0 and -inf, as the insertion list does.
// kSmemLoc: step 2 reads a pick's value by its head index from srow, this thread's row of
// loc_stride(HMAX) floats in shared memory (the candidates' values are stored there), instead of from a
// register copy.  The rows are padded by one float, so the threads of a warp use different banks.
// Measured at a 131072-token prefix (H 32): the biased selection's pass 452 us against 469 us, the
// plain one's 346 us against 333 us, so only the biased kernels take it.
__host__ __device__ constexpr int loc_stride(int hmax) { return hmax + 1; }
template <int HMAX, bool kSmemLoc>
__device__ __forceinline__ void topk4_sorted(const float (&sc)[HMAX], int H, int (&hk)[4], float (&vk)[4],
                                             float* srow) {
  float t0 = -INFINITY, t1 = -INFINITY, t2 = -INFINITY, t3 = -INFINITY;
#pragma unroll
  for (int h = 0; h < HMAX; ++h) {
    if (h < H) {
      float x = sc[h], m;
      m = fmaxf(t0, x); x = fminf(t0, x); t0 = m;
      m = fmaxf(t1, x); x = fminf(t1, x); t1 = m;
      m = fmaxf(t2, x); x = fminf(t2, x); t2 = m;
      t3 = fmaxf(t3, x);
    }
  }
  using Mask = typename std::conditional<(HMAX <= 32), uint32_t, uint64_t>::type;
  Mask ge = 0;     // heads at or above t3
  float loc[HMAX];  // a copy the picks are read back from by index (without kSmemLoc)
#pragma unroll
  for (int h = 0; h < HMAX; ++h) {
    if constexpr (!kSmemLoc) loc[h] = sc[h];
    if (h < H && sc[h] >= t3) {
      ge |= (Mask)1 << h;
      if constexpr (kSmemLoc) srow[h] = sc[h];  // only the heads step 2 reads back
    }
  }
  int eq_left = 4 - ((t0 > t3) + (t1 > t3) + (t2 > t3));  // picks equal to t3
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    hk[k] = 0;
    vk[k] = -INFINITY;
  }
  int n = 0;
  while (ge && n < 4) {
    const int h = (sizeof(Mask) == 4 ? __ffs((int)ge) : __ffsll((long long)ge)) - 1;
    ge &= ge - 1;
    float x;
    if constexpr (kSmemLoc) x = srow[h];
    else x = loc[h];
    const bool take = x > t3 || eq_left > 0;
    if (!take) continue;
    if (!(x > t3)) --eq_left;
    if (n == 0) { hk[0] = h; vk[0] = x; }
    else if (n == 1) { hk[1] = h; vk[1] = x; }
    else if (n == 2) { hk[2] = h; vk[2] = x; }
    else { hk[3] = h; vk[3] = x; }
    ++n;
  }
  // odd-even transposition sort, swapping only on a strictly larger right value (stable)
  auto cas = [&](int a, int b) {
    const bool sw = vk[b] > vk[a];
    const float va = vk[a], vb = vk[b];
    const int ia = hk[a], ib = hk[b];
    vk[a] = sw ? vb : va;
    vk[b] = sw ? va : vb;
    hk[a] = sw ? ib : ia;
    hk[b] = sw ? ia : ib;
  };
  cas(0, 1); cas(2, 3);
  cas(1, 2);
  cas(0, 1); cas(2, 3);
  cas(1, 2);
}

// Top-K for any K <= H: pass k picks the best head strictly after the previous pick in the
// total order (score desc, index asc) and writes it out with its gate.  Returns the picked
// heads as a bit mask.
template <int HMAX, bool kBiased>
__device__ __forceinline__ uint64_t topk_passes(const float (&sc)[HMAX], const float (&a)[HMAX], int H, int K,
                                                float mx, float inv_z, size_t tok, int32_t* __restrict__ topk_head,
                                                float* __restrict__ gate) {
  float pv = 0.f;
  int pi = -1;
  uint64_t mask = 0;
  const size_t base = tok * K;
  for (int k = 0; k < K; ++k) {
    float bv = 0.f;
    int bi = -1;
#pragma unroll
    for (int h = 0; h < HMAX; ++h) {
      const float x = sc[h];
      const bool elig = (h < H) && (pi < 0 || x < pv || (x == pv && h > pi));
      const bool better = elig && (bi < 0 || x > bv);
      bv = better ? x : bv;
      bi = better ? h : bi;
    }
    topk_head[base + k] = bi;
    gate[base + k] = kBiased ? a[bi] : fast_exp2((bv - mx) * kLog2e) * inv_z;
    mask |= 1ull << bi;
    pv = bv;
    pi = bi;
  }
  return mask;
}

// TopK and gates of token `tok` (Sec. 3.1 Eq. namoh-gates), written to topk_head and gate
// ([tok, K] rows).  With KMAX > 0 (K <= KMAX) the picks also stay in hk for the caller;
// with KMAX == 0 any K is taken, the picks only go to memory.  kBiased: selection on the
// biased affinities a + b, gates still a (App. A, Eq. namoh-biased-routing).  Returns the
// picked heads as a bit mask.
template <int HMAX, int KMAX, bool kBiased>
__device__ __forceinline__ uint64_t topk_token(const float* __restrict__ scores, const float* __restrict__ bias,
                                               size_t tok, int H, int K, int32_t* __restrict__ topk_head,
                                               float* __restrict__ gate, int* s_bad,
                                               int (&hk)[KMAX > 0 ? KMAX : 1], float* srow) {
  float sc[HMAX];
  bool bad;
  load_logits<HMAX>(scores, tok, H, sc, bad);
  if (bad) *s_bad = 1;
  float mx, inv_z;
  softmax_norm<HMAX>(sc, H, mx, inv_z);
  // biased selection ranks the affinities a_h plus the head biases b_h; without a bias the
  // logits themselves are ranked (softmax is monotone)
  // the affinity of head h: exp2((logit - max) log2 e) / z, the logit as loaded (non-finite -> -FLT_MAX)
  auto affinity = [&](float l) { return fast_exp2((l - mx) * kLog2e) * inv_z; };
  float a[HMAX];
  if constexpr (kBiased) {
#pragma unroll
    for (int h = 0; h < HMAX; ++h) {
      a[h] = h < H ? affinity(sc[h]) : 0.f;
      sc[h] = h < H ? a[h] + __ldg(bias + h) : 0.f;
    }
  }
  if constexpr (KMAX == 0) {
    return topk_passes<HMAX, kBiased>(sc, a, H, K, mx, inv_z, tok, topk_head, gate);
  } else {
    float vk[KMAX];
    if constexpr (KMAX == 4) topk4_sorted<HMAX, kBiased && HMAX <= 32>(sc, H, hk, vk, srow);
    else topk_sorted<HMAX, KMAX>(sc, H, hk, vk);
    float g[KMAX];
    uint64_t mask = 0;
#pragma unroll
    for (int k = 0; k < KMAX; ++k) {
      if constexpr (kBiased) {
        // the picked head's affinity again from its logit (the row is in L1), rather than a
        // select over all H registers
        float l = __ldg(scores + tok * H + hk[k]);
        if (!isfinite(l)) l = -FLT_MAX;
        g[k] = affinity(l);
      } else {
        g[k] = fast_exp2((vk[k] - mx) * kLog2e) * inv_z;
      }
      if (k < K) mask |= 1ull << hk[k];
    }
    const size_t base = tok * K;
    if (KMAX == 4 && K == 4 && (reinterpret_cast<uintptr_t>(topk_head + base) & 15u) == 0 &&
        (reinterpret_cast<uintptr_t>(gate + base) & 15u) == 0) {
      *reinterpret_cast<int4*>(topk_head + base) = make_int4(hk[0], hk[KMAX > 1 ? 1 : 0], hk[KMAX > 2 ? 2 : 0],
                                                             hk[KMAX > 3 ? 3 : 0]);
      *reinterpret_cast<float4*>(gate + base) = make_float4(g[0], g[KMAX > 1 ? 1 : 0], g[KMAX > 2 ? 2 : 0],
                                                            g[KMAX > 3 ? 3 : 0]);
    } else {
#pragma unroll
      for (int k = 0; k < KMAX; ++k) {
        if (k < K) {
          topk_head[base + k] = hk[k];
          gate[base + k] = g[k];
        }
      }
    }
    return mask;
  }
}

// TopK and gates only (no packed layout), one thread per token.  kFullH: H == HMAX, so every
// per-head guard folds away at compile time.
template <int HMAX, int KMAX, bool kBiased, bool kFullH>
__global__ void __launch_bounds__(kChunk) route_topk_kernel(const float* __restrict__ scores,
                                                            const float* __restrict__ bias, int T, int H_, int K,
                                                            int32_t* __restrict__ topk_head, float* __restrict__ gate,
                                                            uint32_t* __restrict__ status) {
  __shared__ int s_bad;
  __shared__ float s_loc[KMAX == 4 && kBiased && HMAX <= 32 ? kChunk * loc_stride(HMAX) : 1];
  const int H = kFullH ? HMAX : H_;
  const int t = blockIdx.x * kChunk + threadIdx.x;
  if (threadIdx.x == 0) s_bad = 0;
  __syncthreads();
  int hk[KMAX > 0 ? KMAX : 1];
  if (t < T)
    topk_token<HMAX, KMAX, kBiased>(scores, bias, (size_t)blockIdx.y * T + t, H, K, topk_head, gate, &s_bad, hk,
                                    s_loc + (KMAX == 4 && kBiased && HMAX <= 32 ? threadIdx.x * loc_stride(HMAX) : 0));
  __syncthreads();
  if (threadIdx.x == 0 && s_bad) report(status, NAMOH_DEV_NONFINITE_SCORE);
}

// One block per sequence b: for every head, exclusive scan of the chunk counts over chunks
// (thread (h, p) owns the chunk range [p*per, (p+1)*per)) -> chunk bases and n[b, h]; then
// seg_offsets[b*H + h] = b*T*K + sum of n[b, h'] over h' < h.
__global__ void __launch_bounds__(1024) route_scan_kernel(const int32_t* __restrict__ chunk_count, int B, int T,
                                                          int H, int K, int nchunks, int32_t* __restrict__ chunk_base,
                                                          int32_t* __restrict__ seg_offsets,
                                                          const int32_t* __restrict__ cu_seqlens, int total) {
  __shared__ int s_part[1024];
  __shared__ int s_n[NAMOH_MAX_HEADS];
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  pdl_launch_dependents();
  pdl_wait();  // pass 1 complete and visible
  const int P = blockDim.x / H;  // parts per head (blockDim is a multiple of H)
  const int h = tid % H, p = tid / H;
  const int per = (nchunks + P - 1) / P;
  const int c0 = min(nchunks, p * per), c1 = min(nchunks, c0 + per);
  const int32_t* cc = chunk_count + (size_t)b * nchunks * H;
  int sum = 0;
  for (int c = c0; c < c1; ++c) sum += __ldg(cc + (size_t)c * H + h);
  s_part[tid] = sum;
  __syncthreads();
  int before = 0;
  for (int q = 0; q < p; ++q) before += s_part[q * H + h];
  int run = before;
  int32_t* out = chunk_base + (size_t)b * nchunks * H;
  for (int c = c0; c < c1; ++c) {
    out[(size_t)c * H + h] = run;
    run += __ldg(cc + (size_t)c * H + h);
  }
  if (p == P - 1) s_n[h] = run;
  __syncthreads();
  if (tid == 0) {
    int off = seq_range(cu_seqlens, b, B, T, total).start * K;  // < 2^31: checked on the host
    for (int hh = 0; hh < H; ++hh) {
      seg_offsets[(size_t)b * H + hh] = off;
      off += s_n[hh];
    }
    if (b == B - 1) seg_offsets[(size_t)B * H] = off;
  }
}

// Pass 1 of the packed layout (one block per chunk, one thread per token): TopK and gates,
// the chunk's head counts, and rank_local = the (token, slot)'s rank among this chunk's
// earlier tokens for its head (Sec. 3.2 Eq. namoh-head-rope restricted to the chunk).
// rank_local goes to `rank`, which the final pass turns into the full rank.
template <int HMAX, int KMAX, bool kBiased, bool kFullH>
__global__ void __launch_bounds__(kChunk) route_local_kernel(const float* __restrict__ scores,
                                                             const float* __restrict__ bias, int T, int H_, int K,
                                                             int nchunks, int32_t* __restrict__ topk_head,
                                                             float* __restrict__ gate, int32_t* __restrict__ rank,
                                                             int32_t* __restrict__ chunk_count,
                                                             uint32_t* __restrict__ status,
                                                             const int32_t* __restrict__ cu_seqlens, int B,
                                                             int total) {
  __shared__ uint32_t s_bal[kChunk / 32][NAMOH_MAX_HEADS];
  __shared__ int s_pre[kChunk / 32][NAMOH_MAX_HEADS];
  __shared__ int s_bad;
  __shared__ float s_loc[KMAX == 4 && kBiased && HMAX <= 32 ? kChunk * loc_stride(HMAX) : 1];
  const int H = kFullH ? HMAX : H_;  // (kFullH: a compile-time head count)
  pdl_launch_dependents();
  const int c = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t = c * kChunk + tid;
  if (tid == 0) s_bad = 0;
  __syncthreads();
  // the logits may come from the kernel just before this one, and that kernel may still
  // read this call's outputs: nothing global is touched before the wait
  pdl_wait();
  const SeqRange sr = seq_range(cu_seqlens, b, B, T, total);
  if (!sr.ok && c == 0 && tid == 0) report(status, NAMOH_DEV_BAD_SEQLENS);
  const bool valid = t < sr.len;
  const size_t tok = (size_t)sr.start + t;
  uint64_t mask = 0;
  int hk[KMAX > 0 ? KMAX : 1];
  if (valid)
    mask = topk_token<HMAX, KMAX, kBiased>(scores, bias, tok, H, K, topk_head, gate, &s_bad, hk,
                                           s_loc + (KMAX == 4 && kBiased && HMAX <= 32 ? tid * loc_stride(HMAX) : 0));
  // s_bal[warp][h] = the warp's ballot of "selects head h": the 32 x 32 bit matrix of the lanes'
  // head masks transposed in five shuffle stages (each swaps the off-diagonal blocks of size j)
#pragma unroll
  for (int half = 0; half < (HMAX > 32 ? 2 : 1); ++half) {
    uint32_t m = (uint32_t)(mask >> (32 * half));
#pragma unroll
    for (int j = 16; j > 0; j >>= 1) {
      const uint32_t lowj = j == 16 ? 0x0000FFFFu : j == 8 ? 0x00FF00FFu : j == 4 ? 0x0F0F0F0Fu
                            : j == 2 ? 0x33333333u : 0x55555555u;
      const uint32_t y = __shfl_xor_sync(0xffffffffu, m, j);
      m = (lane & j) ? ((m & ~lowj) | ((y >> j) & lowj)) : ((m & lowj) | ((y << j) & ~lowj));
    }
    if (32 * half + lane < H) s_bal[warp][32 * half + lane] = m;
  }
  __syncthreads();
  if (tid < H) {
    // s_pre[w][h]: tokens of warps before w that picked head h; the chunk's count
    int n = 0;
#pragma unroll
    for (int w = 0; w < kChunk / 32; ++w) {
      s_pre[w][tid] = n;
      n += __popc(s_bal[w][tid]);
    }
    chunk_count[((size_t)b * nchunks + c) * H + tid] = n;
  }
  __syncthreads();
  if (tid == 0 && s_bad) report(status, NAMOH_DEV_NONFINITE_SCORE);
  if (!valid) return;
  const uint32_t lt = (1u << lane) - 1u;
  auto local_rank = [&](int h) { return s_pre[warp][h] + __popc(s_bal[warp][h] & lt); };
  const size_t base = tok * K;
  if constexpr (KMAX > 0) {
    int rk[KMAX];
#pragma unroll
    for (int k = 0; k < KMAX; ++k) rk[k] = k < K ? local_rank(hk[k]) : 0;
    if (KMAX == 4 && K == 4 && (reinterpret_cast<uintptr_t>(rank + base) & 15u) == 0) {
      *reinterpret_cast<int4*>(rank + base) = make_int4(rk[0], rk[KMAX > 1 ? 1 : 0], rk[KMAX > 2 ? 2 : 0],
                                                        rk[KMAX > 3 ? 3 : 0]);
    } else {
#pragma unroll
      for (int k = 0; k < KMAX; ++k)
        if (k < K) rank[base + k] = rk[k];
    }
  } else {
    for (int k = 0; k < K; ++k) rank[base + k] = local_rank(topk_head[base + k]);  // written above by this thread
  }
}

// Pass 2 (one block per chunk): this chunk's base rank per head and the sequence's
// segment offsets -- from the chunk-count table (chunk_base == nullptr: thread (h, p)
// sums chunks p, p + P, ...), or as written by route_scan_kernel -- then
// rank = base + rank_local, row = seg_offsets[b*H + head] + rank, row_src[row].
__global__ void __launch_bounds__(kChunk) route_final_kernel(const int32_t* __restrict__ topk_head, int T, int H,
                                                             int K, int nchunks, const int32_t* chunk_count,
                                                             const int32_t* chunk_base, int32_t* __restrict__ rank,
                                                             int32_t* __restrict__ row, int32_t* seg_offsets,
                                                             int32_t* __restrict__ row_src, int B,
                                                             const int32_t* __restrict__ cu_seqlens, int total) {
  __shared__ int s_tot[kChunk];
  __shared__ int s_bef[kChunk];
  __shared__ int s_cbase[NAMOH_MAX_HEADS];
  __shared__ int s_soff[NAMOH_MAX_HEADS];
  __shared__ int s_pos[NAMOH_MAX_HEADS];  // (K = 4) first staging slot of each head's rows
  __shared__ int32_t s_src[kChunk * 4];   // (K = 4) row_src values, grouped by head in rank order
  __shared__ int32_t s_dst[kChunk * 4];   // (K = 4) and the rows they go to
  pdl_launch_dependents();
  const int c = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x;
  const int t = c * kChunk + tid;
  pdl_wait();  // pass 1 (and the scan, when there is one) complete and visible
  const SeqRange sr = seq_range(cu_seqlens, b, B, T, total);
  const bool valid = t < sr.len;
  const size_t tok = (size_t)sr.start + t;
  const size_t base = tok * K;
  // this token's heads and local ranks first: their loads overlap the count-table work
  const bool vec4 = K == 4 && (reinterpret_cast<uintptr_t>(topk_head + base) & 15u) == 0 &&
                    (reinterpret_cast<uintptr_t>(rank + base) & 15u) == 0 &&
                    (reinterpret_cast<uintptr_t>(row + base) & 15u) == 0;
  int4 h4 = make_int4(0, 0, 0, 0), r4 = make_int4(0, 0, 0, 0);
  if (valid && vec4) {
    h4 = __ldcg(reinterpret_cast<const int4*>(topk_head + base));
    r4 = __ldcg(reinterpret_cast<const int4*>(rank + base));
  }
  // (K = 4) the chunk's head counts, for the staging slots below
  if (K == 4 && tid < H) s_pos[tid] = __ldcg(chunk_count + ((size_t)b * nchunks + c) * H + tid);
  if (chunk_base) {
    if (tid < H) {
      s_cbase[tid] = chunk_base[((size_t)b * nchunks + c) * H + tid];
      s_soff[tid] = seg_offsets[(size_t)b * H + tid];
    }
  } else {
    const int P = kChunk / H;
    const int h = tid % H, p = tid / H;
    int tot = 0, bef = 0;
    if (p < P) {
      const int32_t* cc = chunk_count + (size_t)b * nchunks * H + h;
      for (int cj = p; cj < nchunks; cj += P) {
        const int v = __ldcg(cc + (size_t)cj * H);
        tot += v;
        bef += (cj < c) ? v : 0;
      }
    }
    s_tot[tid] = tot;
    s_bef[tid] = bef;
    __syncthreads();
    if (tid < H) {
      int n = 0, cb = 0;
      for (int q = 0; q < P; ++q) {
        n += s_tot[q * H + tid];
        cb += s_bef[q * H + tid];
      }
      s_cbase[tid] = cb;
      s_tot[tid] = n;  // rows q >= 1 of s_tot are no longer read
    }
    __syncthreads();
    if (tid == 0) {
      int off = sr.start * K;  // < 2^31: checked on the host
      for (int hh = 0; hh < H; ++hh) {
        s_soff[hh] = off;
        off += s_tot[hh];
      }
    }
    __syncthreads();
    if (c == 0 && tid < H) seg_offsets[(size_t)b * H + tid] = s_soff[tid];
    if (c == 0 && b == B - 1 && tid == 0) seg_offsets[(size_t)B * H] = (sr.start + sr.len) * K;
  }
  // every thread: the count-table results above are visible after this barrier
  const bool staged = __syncthreads_and(!valid || vec4);
  if (K == 4 && staged) {
    // row_src through shared memory: this chunk's rows of head h are the contiguous run
    // seg_offsets + chunk base .. + count of segment h, so staging the values by head (at their
    // local rank) and writing the staged array in order turns 4 scattered stores per token into
    // runs of consecutive rows
    // the exclusive prefix of the chunk's head counts (warp 0, two scans of up to 32 heads)
    if (tid < 32) {
      const int lane = tid;
      int carry = 0;
#pragma unroll
      for (int half = 0; half < 2; ++half) {
        const int h = 32 * half + lane;
        const int v = h < H ? s_pos[h] : 0;
        int inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, inc, o);
          if (lane >= o) inc += y;
        }
        if (h < H) s_pos[h] = carry + inc - v;
        carry += __shfl_sync(0xffffffffu, inc, 31);
      }
    }
    __syncthreads();
    if (valid) {
      const int hs[4] = {h4.x, h4.y, h4.z, h4.w}, ls[4] = {r4.x, r4.y, r4.z, r4.w};
      int rho[4], rw[4];
#pragma unroll
      for (int k = 0; k < 4; ++k) {
        rho[k] = s_cbase[hs[k]] + ls[k];
        rw[k] = s_soff[hs[k]] + rho[k];
        const int e = s_pos[hs[k]] + ls[k];
        s_src[e] = (int32_t)(base + k);
        s_dst[e] = rw[k];
      }
      *reinterpret_cast<int4*>(rank + base) = make_int4(rho[0], rho[1], rho[2], rho[3]);
      *reinterpret_cast<int4*>(row + base) = make_int4(rw[0], rw[1], rw[2], rw[3]);
    }
    __syncthreads();
    const int nent = 4 * max(0, min(kChunk, sr.len - c * kChunk));  // this chunk's (token, slot) rows
    for (int e = tid; e < nent; e += kChunk) row_src[s_dst[e]] = s_src[e];
    return;
  }
  if (!valid) return;
  for (int k = 0; k < K; ++k) {
    const size_t i = base + k;
    const int h = topk_head[i];
    const int rho = s_cbase[h] + rank[i];
    const int r = s_soff[h] + rho;
    rank[i] = rho;
    row[i] = r;
    row_src[r] = (int32_t)i;
  }
}

struct RouteArgs {
  const float* scores;
  const float* bias;  // [H] or nullptr
  const int32_t* cu_seqlens;  // [B + 1] for a ragged batch (T = longest sequence), or nullptr
  int total;                  // tokens in all (ragged batch)
  int B, T, H, K, nchunks;
  int32_t *topk_head, *rank, *row, *seg_offsets, *row_src;
  float* gate;
  int32_t *chunk_count, *chunk_base;
  uint32_t* status;
};

// Count tables up to this many entries per sequence are summed by every block of the final
// pass; larger ones are scanned once by route_scan_kernel.
constexpr int kFinalMaxTable = 1 << 12;

template <int HMAX, int KMAX, bool kBiased, bool kFullH = false>
int launch_route(const RouteArgs& a, cudaStream_t stream) {
  const dim3 chunks((unsigned)a.nchunks, (unsigned)a.B);
  if (a.seg_offsets == nullptr) {
    route_topk_kernel<HMAX, KMAX, kBiased, kFullH><<<chunks, kChunk, 0, stream>>>(a.scores, a.bias, a.T, a.H, a.K,
                                                                                  a.topk_head, a.gate, a.status);
    return cuda_check_launch("route_topk_kernel launch");
  }
  cudaError_t e = launch_pdl(route_local_kernel<HMAX, KMAX, kBiased, kFullH>, chunks, dim3(kChunk), 0, stream, a.scores,
                             a.bias,
                             a.T, a.H, a.K, a.nchunks, a.topk_head, a.gate, a.rank, a.chunk_count, a.status,
                             a.cu_seqlens, a.B, a.total);
  if (e != cudaSuccess) return cuda_fail(e, "route_local_kernel launch");
  const bool scan = (long long)a.nchunks * a.H > kFinalMaxTable;
  if (scan) {
    const int scan_threads = 1024 - (1024 % a.H);
    e = launch_pdl(route_scan_kernel, dim3((unsigned)a.B), dim3((unsigned)scan_threads), 0, stream,
                   (const int32_t*)a.chunk_count, a.B, a.T, a.H, a.K, a.nchunks, a.chunk_base, a.seg_offsets,
                   a.cu_seqlens, a.total);
    if (e != cudaSuccess) return cuda_fail(e, "route_scan_kernel launch");
  }
  e = launch_pdl(route_final_kernel, chunks, dim3(kChunk), 0, stream, (const int32_t*)a.topk_head, a.T, a.H, a.K,
                 a.nchunks, (const int32_t*)a.chunk_count, (const int32_t*)(scan ? a.chunk_base : nullptr), a.rank,
                 a.row, a.seg_offsets, a.row_src, a.B, a.cu_seqlens, a.total);
  if (e != cudaSuccess) return cuda_fail(e, "route_final_kernel launch");
  return NAMOH_OK;
}

// picks held in registers for K <= 8; larger K takes K passes over the logits.  K <= 4 with H a
// power of two takes the kernels with a compile-time head count.
template <int HMAX, bool kBiased>
int launch_route_k4(const RouteArgs& a, cudaStream_t stream) {
  return a.H == HMAX ? launch_route<HMAX, 4, kBiased, true>(a, stream) : launch_route<HMAX, 4, kBiased>(a, stream);
}
template <bool kBiased>
int launch_route_h(const RouteArgs& a, cudaStream_t stream) {
  const int H = a.H, K = a.K;
  if (H <= 8) return K <= 4 ? launch_route_k4<8, kBiased>(a, stream) : launch_route<8, 8, kBiased>(a, stream);
  if (H <= 16)
    return K <= 4 ? launch_route_k4<16, kBiased>(a, stream)
                  : K <= 8 ? launch_route<16, 8, kBiased>(a, stream) : launch_route<16, 0, kBiased>(a, stream);
  if (H <= 32)
    return K <= 4 ? launch_route_k4<32, kBiased>(a, stream)
                  : K <= 8 ? launch_route<32, 8, kBiased>(a, stream) : launch_route<32, 0, kBiased>(a, stream);
  return K <= 4 ? launch_route_k4<64, kBiased>(a, stream)
                : K <= 8 ? launch_route<64, 8, kBiased>(a, stream) : launch_route<64, 0, kBiased>(a, stream);
}

}  // namespace
}  // namespace namoh

using namespace namoh;

extern "C" size_t namoh_route_workspace_size(int B, int T, int H, int K) {
  if (B < 1 || T < 1 || H < 1 || K < 1) return 0;
  const size_t nchunks = ((size_t)T + kChunk - 1) / kChunk;
  WorkspaceCarver ws{nullptr, 0, 0};
  ws.take<int32_t>((size_t)B * nchunks * H);  // chunk counts
  ws.take<int32_t>((size_t)B * nchunks * H);  // chunk bases
  return align_up(ws.used, 256);
}

namespace namoh {
namespace {
// Shared body of the routing entry points.  cu_seqlens == nullptr: B sequences of T tokens;
// else a ragged batch of `total` tokens whose longest sequence has T tokens.
int route_impl(const float* scores, const float* bias, const int32_t* cu_seqlens, int B, int T, int total, int H,
               int K, int32_t* topk_head, float* gate, int32_t* rank, int32_t* row, int32_t* seg_offsets,
               int32_t* row_src, void* workspace, size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!scores || !topk_head || !gate || !dev_status) return NAMOH_ERR_INVALID_ARG;
  if (B < 1 || T < 1 || H < 1 || K < 1 || K > H || H > NAMOH_MAX_HEADS) return NAMOH_ERR_INVALID_ARG;
  const long long tokens = cu_seqlens ? (long long)total : (long long)B * T;
  if (tokens * K >= (1ll << 31) || (long long)B * H >= (1ll << 20)) return NAMOH_ERR_INVALID_ARG;
  if (cu_seqlens && total < T) return NAMOH_ERR_INVALID_ARG;
  const bool compact = seg_offsets != nullptr;
  if (compact != (rank != nullptr) || compact != (row != nullptr) || compact != (row_src != nullptr))
    return NAMOH_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  RouteArgs a{};
  a.scores = scores;
  a.bias = bias;
  a.cu_seqlens = cu_seqlens;
  a.total = total;
  a.B = B;
  a.T = T;
  if (cu_seqlens && !compact) {  // picks only: one flat sequence of every token
    a.cu_seqlens = nullptr;
    a.B = 1;
    a.T = total;
  }
  a.H = H;
  a.K = K;
  a.nchunks = (a.T + kChunk - 1) / kChunk;
  a.topk_head = topk_head;
  a.gate = gate;
  a.rank = rank;
  a.row = row;
  a.seg_offsets = seg_offsets;
  a.row_src = row_src;
  a.status = dev_status;
  if (compact) {
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
    WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
    a.chunk_count = ws.take<int32_t>((size_t)B * a.nchunks * H);
    a.chunk_base = ws.take<int32_t>((size_t)B * a.nchunks * H);
    if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  }
  return a.bias ? launch_route_h<true>(a, stream) : launch_route_h<false>(a, stream);
}
}  // namespace
}  // namespace namoh

extern "C" int namoh_route_biased(const float* scores, const float* bias, int B, int T, int H, int K,
                                  int32_t* topk_head, float* gate, int32_t* rank, int32_t* row, int32_t* seg_offsets,
                                  int32_t* row_src, void* workspace, size_t workspace_bytes, uint32_t* dev_status,
                                  void* stream_v) {
  return route_impl(scores, bias, nullptr, B, T, 0, H, K, topk_head, gate, rank, row, seg_offsets, row_src, workspace,
                    workspace_bytes, dev_status, stream_v);
}

extern "C" int namoh_route_varlen(const float* scores, const float* bias, const int32_t* cu_seqlens, int B,
                                  int total_tokens, int max_seqlen, int H, int K, int32_t* topk_head, float* gate,
                                  int32_t* rank, int32_t* row, int32_t* seg_offsets, int32_t* row_src,
                                  void* workspace, size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!cu_seqlens || total_tokens < 1) return NAMOH_ERR_INVALID_ARG;
  return route_impl(scores, bias, cu_seqlens, B, max_seqlen, total_tokens, H, K, topk_head, gate, rank, row,
                    seg_offsets, row_src, workspace, workspace_bytes, dev_status, stream_v);
}

extern "C" int namoh_route(const float* scores, int B, int T, int H, int K, int32_t* topk_head, float* gate,
                           int32_t* rank, int32_t* row, int32_t* seg_offsets, int32_t* row_src, void* workspace,
                           size_t workspace_bytes, uint32_t* dev_status, void* stream) {
  return namoh_route_biased(scores, nullptr, B, T, H, K, topk_head, gate, rank, row, seg_offsets, row_src, workspace,
                            workspace_bytes, dev_status, stream);
}

// ---------------------------------------------------------------------------
// Routing with built-in scratch (no caller workspace, no allocation).
// The scratch is a file-scope device array; host code only ever passes the
// device address obtained from cudaGetSymbolAddress, never the array's name.
// ---------------------------------------------------------------------------

namespace namoh {
namespace {
constexpr size_t kRouteStaticScratchBytes = 4u << 20;  // 4 MiB on every device that loads the library
static __device__ __align__(256) unsigned char g_route_scratch[kRouteStaticScratchBytes];

constexpr int kMaxScratchDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxScratchDevices] = {};

// Device address of g_route_scratch on the current device (resolved once per device).
void* route_scratch_address() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxScratchDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_addr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_route_scratch) != cudaSuccess) return nullptr;
    g_scratch_addr[dev] = ptr;
  }
  return g_scratch_addr[dev];
}
}  // namespace
}  // namespace namoh

extern "C" int namoh_route_noalloc(const float* scores, int B, int T, int H, int K, int32_t* topk_head, float* gate,
                                   int32_t* rank, int32_t* row, int32_t* seg_offsets, int32_t* row_src,
                                   uint32_t* dev_status, void* stream) {
  if (!scores || !topk_head || !gate || !dev_status) return NAMOH_ERR_INVALID_ARG;
  if (B < 1 || T < 1 || H < 1 || K < 1 || K > H || H > NAMOH_MAX_HEADS) return NAMOH_ERR_INVALID_ARG;
  if (seg_offsets && namoh_route_workspace_size(B, T, H, K) > kRouteStaticScratchBytes) return NAMOH_ERR_WORKSPACE;
  void* scratch = route_scratch_address();
  if (!scratch) return cuda_fail(cudaErrorInvalidSymbol, "cudaGetSymbolAddress of the routing scratch");
  return namoh_route(scores, B, T, H, K, topk_head, gate, rank, row, seg_offsets, row_src, scratch,
                     kRouteStaticScratchBytes, dev_status, stream);
}
