// sa_select.cu -- block selection of SA + NAMOH (App. B.8 "SA+NAMOH", with the selection model of
// App. B.3 "Block-Selected Sparse Attention", Eqs. app-block-budget and app-selected-entries).
//
// Within each routed history (a segment of packed rows in local order), the keys form blocks of
// `block` entries.  A query at one-based local rank r sees N_B(r) = ceil(r / block) blocks and keeps
// R(r) = ceil(alpha N_B(r)) of them: its current block (attended causally by the attention kernel)
// and the R(r) - 1 completed blocks whose mean-pooled key scores highest against the query (the
// MoBA selector of App. B.3).  Ties go to the lower block index; alpha = alpha_num / alpha_den.
//
//   sa_pool_kernel    one warp per (segment, complete block): the block's rotated keys (bf16, from
//                     the cache) summed in fp32 in row order and scaled by 1 / block (exact: block
//                     is a power of two) -> kbar[blk_base(s) + b], blk_base(s) = seg_offsets[s] /
//                     block + s (disjoint per segment, at most R / block + nseg rows).
//   sa_select_kernel  one warp per query (packed row, group head j): for each group of 32 blocks
//                     before the current one, lane l multiplies its d / 32 columns of q~ with those
//                     columns of every block's pooled key (one coalesced row read per block), and a
//                     warp reduce-scatter (31 shuffles) leaves block 32 i + l's fp32 score in lane l.
//                     R(r) - 1 rounds of a warp arg-max then pick the kept blocks; the mask row
//                     [row * g + j] gets one bit per kept block (bit b % 32 of word b / 32).
#include "common.cuh"

namespace namoh {
namespace sa {

constexpr int kMaxBlocks = 1024;            // blocks per history the selector holds (32 per lane)
constexpr int kPerLane = kMaxBlocks / 32;

__device__ __forceinline__ int blk_base(const int32_t* seg_offsets, int s, int lg) {
  return (seg_offsets[s] >> lg) + s;
}

// A segment is live when its rows are in the cache: always for the packed layout; with seg_base only
// when n <= seg_cap (the RoPE pass skips the others' rows and the plan leaves them out).
__device__ __forceinline__ bool seg_live(const int32_t* seg_offsets, const int64_t* seg_base,
                                         const int32_t* seg_cap, int s) {
  return !seg_base || seg_offsets[s + 1] - seg_offsets[s] <= seg_cap[s];
}

__global__ void __launch_bounds__(256) sa_pool_kernel(const uint16_t* __restrict__ k_cache,
                                                      const int32_t* __restrict__ seg_offsets,
                                                      const int64_t* __restrict__ seg_base,
                                                      const int32_t* __restrict__ seg_cap, long long cache_rows,
                                                      int d, int lg, float* __restrict__ kbar) {
  const int s = blockIdx.y;
  const int b = blockIdx.x * 8 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  const int n = seg_offsets[s + 1] - seg_offsets[s];
  if (b >= (n >> lg) || !seg_live(seg_offsets, seg_base, seg_cap, s)) return;
  const long long row0 = (seg_base ? seg_base[s] : (long long)seg_offsets[s]) + ((long long)b << lg);
  // rows outside the cache were never written (the RoPE pass reports them): nothing to pool
  if (row0 < 0 || row0 + (1ll << lg) > cache_rows) return;
  const int per = d / 32;  // columns per lane (2 or 4)
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
  for (int t = 0; t < (1 << lg); ++t) {
    const uint16_t* src = k_cache + (row0 + t) * d + lane * per;
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (i < per) acc[i] += __uint_as_float((uint32_t)src[i] << 16);
  }
  const float inv = 1.0f / (float)(1 << lg);
  float* dst = kbar + ((long long)blk_base(seg_offsets, s, lg) + b) * d + lane * per;
#pragma unroll
  for (int i = 0; i < 4; ++i)
    if (i < per) dst[i] = acc[i] * inv;
}

__global__ void __launch_bounds__(256) sa_select_kernel(const uint16_t* __restrict__ q_rot,
                                                        const int32_t* __restrict__ seg_offsets, int nseg,
                                                        const int64_t* __restrict__ seg_base,
                                                        const int32_t* __restrict__ seg_cap,
                                                        const float* __restrict__ kbar, int d, int g, int lg,
                                                        int alpha_num, int alpha_den, long long nq,
                                                        uint32_t* __restrict__ mask, int words) {
  const int wib = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const long long qi = (long long)blockIdx.x * 8 + wib;  // query number: packed row * g + j
  if (qi >= nq) return;
  const long long row = qi / g;
  // the segment holding this row
  int lo = 0, hi = nseg;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (seg_offsets[mid] <= row) lo = mid;
    else hi = mid;
  }
  const int r = (int)(row - seg_offsets[lo]);  // zero-based local rank
  const int cur = r >> lg;                      // current block = N_B(r + 1) - 1
  // kept historical blocks: ceil(alpha (cur + 1)) - 1, computed exactly; none in a segment that
  // is not in the cache (its pooled keys were never written and the attention skips it)
  const int keep = seg_live(seg_offsets, seg_base, seg_cap, lo)
                       ? (int)(((long long)(cur + 1) * alpha_num + alpha_den - 1) / alpha_den) - 1
                       : 0;
  const int per = d / 32;  // columns of q~ and of the pooled keys per lane (2 or 4)
  float ql[4];
#pragma unroll
  for (int e = 0; e < 4; ++e)
    ql[e] = e < per ? __uint_as_float((uint32_t)q_rot[qi * d + lane * per + e] << 16) : 0.f;
  const float* kb = kbar + (long long)blk_base(seg_offsets, lo, lg) * d + lane * per;
  // score slots in use: blocks i * 32 + lane < cur (warp-uniform count; the loops below stop there)
  const int nslot = keep > 0 ? (cur + 31) >> 5 : 0;
  float sc[kPerLane];
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    if (i >= nslot) break;
    float v[32];  // this lane's partial dot products for blocks 32 i + t
#pragma unroll
    for (int t = 0; t < 32; ++t) {
      const int b = i * 32 + t;
      float a = 0.f;
      if (b < cur) {
        const float* kr = kb + (long long)b * d;
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (e < per) a = fmaf(ql[e], __ldg(kr + e), a);
      }
      v[t] = a;
    }
    // reduce-scatter: at the step of offset o a lane keeps the half of its live values whose
    // block index has bit o equal to its own lane bit, adding the partner's copy of that half;
    // afterwards v[0] of lane l is the whole sum for block 32 i + l
#pragma unroll
    for (int o = 16, n = 32; o > 0; o >>= 1, n >>= 1) {
      const bool up = (lane & o) != 0;
#pragma unroll
      for (int jj = 0; jj < n / 2; ++jj) {
        const float send = up ? v[jj] : v[jj + n / 2];
        const float mine = up ? v[jj + n / 2] : v[jj];
        v[jj] = mine + __shfl_xor_sync(0xffffffffu, send, o);
      }
    }
    sc[i] = i * 32 + lane < cur ? v[0] : -INFINITY;
  }
  uint32_t taken = 0;  // bit i: block i * 32 + lane kept
  for (int m = 0; m < keep; ++m) {
    // this lane's best remaining block (highest score, lowest index), then the warp's
    float best = -INFINITY;
    int bi = -1;
#pragma unroll
    for (int i = 0; i < kPerLane; ++i) {
      if (i >= nslot) break;
      const int b = i * 32 + lane;
      if (b < cur && !((taken >> i) & 1u) && (bi < 0 || sc[i] > best)) {
        best = sc[i];
        bi = i;
      }
    }
    int bb = bi < 0 ? 0x7fffffff : bi * 32 + lane;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float ob = __shfl_xor_sync(0xffffffffu, best, o);
      const int obb = __shfl_xor_sync(0xffffffffu, bb, o);
      if (obb != 0x7fffffff && (bb == 0x7fffffff || ob > best || (ob == best && obb < bb))) {
        best = ob;
        bb = obb;
      }
    }
    if (bb == 0x7fffffff) break;  // cannot happen: keep <= cur
    if ((bb & 31) == lane) taken |= 1u << (bb >> 5);
  }
  uint32_t* mrow = mask + qi * words;
#pragma unroll
  for (int i = 0; i < kPerLane; ++i) {
    if (i >= words) break;
    const uint32_t w = __ballot_sync(0xffffffffu, (taken >> i) & 1u);
    if (lane == 0) mrow[i] = w;
  }
}

}  // namespace sa

int launch_sa_select(const uint16_t* q_rot, const uint16_t* k_cache, const int32_t* seg_offsets,
                     const int64_t* seg_base, const int32_t* seg_cap, long long cache_rows, int nseg, int T,
                     long long R, int d, int g, int lg, int alpha_num, int alpha_den, float* kbar, uint32_t* mask,
                     int words, cudaStream_t stream) {
  const int max_blocks = (T + (1 << lg) - 1) >> lg;
  if (nseg > 0 && max_blocks > 0) {
    dim3 grid((max_blocks + 7) / 8, nseg);
    sa::sa_pool_kernel<<<grid, 256, 0, stream>>>(k_cache, seg_offsets, seg_base, seg_cap, cache_rows, d, lg, kbar);
    if (const int st = cuda_check_launch("sa_pool_kernel launch")) return st;
  }
  const long long nq = R * g;
  if (nq > 0) {
    sa::sa_select_kernel<<<(unsigned)((nq + 7) / 8), 256, 0, stream>>>(q_rot, seg_offsets, nseg, seg_base, seg_cap, kbar,
                                                                       d, g, lg, alpha_num, alpha_den, nq, mask,
                                                                       words);
    if (const int st = cuda_check_launch("sa_select_kernel launch")) return st;
  }
  return NAMOH_OK;
}

}  // namespace namoh
