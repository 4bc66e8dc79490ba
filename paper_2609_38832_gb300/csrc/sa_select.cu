// sa_select.cu -- block selection of SA + NAMOH (App. B.8 "SA+NAMOH", with the selection model of
// App. B.3 "Block-Selected Sparse Attention", Eqs. app-block-budget and app-selected-entries).
//
// Within each routed history (a segment of packed rows in local order), the keys form blocks of
// `block` entries.  A query at one-based local rank r sees N_B(r) = ceil(r / block) blocks and keeps
// R(r) = ceil(alpha N_B(r)) of them: its current block (attended causally by the attention kernel)
// and the R(r) - 1 completed blocks whose mean-pooled key scores highest against the query (the
// MoBA selector of App. B.3).  alpha = alpha_num / alpha_den.
//
//   sa_pool_kernel        one warp per (segment, complete block): the block's rotated keys (bf16, from
//                         the cache) summed in fp32, scaled by 1 / block (exact: block is a power of two)
//                         and rounded to bf16 -> kbar[blk_base(s) + b], blk_base(s) = seg_offsets[s] /
//                         block + s (disjoint per segment, at most R / block + nseg rows).  Lanes read
//                         whole 16-byte pieces (two or four rows per warp instruction) and the lanes
//                         holding one piece of different rows add up by a butterfly.
//   sa_select_tc_kernel   one CTA per item of the attention plan (128 query rows of one segment and
//                         group head j).  The block scores of the tile are one dense contraction,
//                         S = Q~[128 x d] K̄^T[d x nb], run as tcgen05.mma (bf16, fp32 accumulate into
//                         TMEM; Q~ and the pooled keys staged by TMA).  Thread i owns query row i (TMEM
//                         lane i) and picks its kept blocks from its row of S (below).
//   sa_select_kernel      the rows whose current block lies past the kSelMaxCols scores one CTA holds
//                         in TMEM: one warp per query, scores on the CUDA cores (lane l: d / 32 columns,
//                         warp reduce-scatter per 32 blocks), R(r) - 1 rounds of a warp arg-max.
//
// The per-query selection itself (keys, register list, bisection) is in sa_select.cuh.
#include <algorithm>

#include "common.cuh"
#include "sa_select.cuh"

namespace namoh {
namespace sa {

constexpr int kMaxBlocks = 1024;            // blocks per history the selectors hold (32 per lane)
constexpr int kPerLane = kMaxBlocks / 32;
constexpr int kSelMaxCols = 512;            // block scores one select CTA keeps in TMEM
constexpr int kSelThreads = 128;            // one thread per query row of a 128-row tile
constexpr int kSelTileRows = 128;
constexpr int kKbBox = 64;                  // pooled-key rows per TMA box

__device__ __forceinline__ int blk_base(const int32_t* seg_offsets, int s, int lg) {
  return (seg_offsets[s] >> lg) + s;
}

// A segment is live when its rows are in the cache: always for the packed layout; with seg_base only
// when n <= seg_cap (the RoPE pass skips the others' rows and the plan leaves them out).
__device__ __forceinline__ bool seg_live(const int32_t* seg_offsets, const int64_t* seg_base,
                                         const int32_t* seg_cap, int s) {
  return !seg_base || seg_offsets[s + 1] - seg_offsets[s] <= seg_cap[s];
}

template <int D, int LG>
__global__ void __launch_bounds__(256) sa_pool_kernel(const uint16_t* __restrict__ k_cache,
                                                      const int32_t* __restrict__ seg_offsets,
                                                      const int64_t* __restrict__ seg_base,
                                                      const int32_t* __restrict__ seg_cap, long long cache_rows,
                                                      int g, uint16_t* __restrict__ kbar, uint32_t* __restrict__ mask,
                                                      int words) {
  constexpr int d = D, lg = LG;
  pdl_launch_dependents();
  pdl_wait();  // the rotated keys come from the RoPE pass before it
  const int s = blockIdx.y;
  const int lane = threadIdx.x & 31;
  const int n = seg_offsets[s + 1] - seg_offsets[s];
  if (!seg_live(seg_offsets, seg_base, seg_cap, s)) {
    // a segment not in the cache keeps no block: its mask rows are zero
    if (blockIdx.x == 0) {
      const long long m0 = (long long)seg_offsets[s] * g * words, m1 = (long long)seg_offsets[s + 1] * g * words;
      for (long long i = m0 + threadIdx.x; i < m1; i += blockDim.x) mask[i] = 0u;
    }
    return;
  }
  const int b = blockIdx.x * 8 + (threadIdx.x >> 5);
  if (b >= (n >> lg)) return;
  const long long row0 = (seg_base ? seg_base[s] : (long long)seg_offsets[s]) + ((long long)b << lg);
  // rows outside the cache were never written (the RoPE pass reports them): nothing to pool
  if (row0 < 0 || row0 + (1ll << lg) > cache_rows) return;
  // lane l reads the 16-byte piece l % P of row t + l / P, P = d / 8 pieces per row; every load of
  // the block is issued before the first is used (the block's rows a lane reads: 2^lg / (32 / P))
  constexpr int P = D / 8;            // 8 or 16
  constexpr int rows_per = 32 / P;    // rows per warp instruction: 4 or 2
  constexpr int nld = (1 << LG) / rows_per;
  const int piece = lane % P, sub = lane / P;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  const uint4* src = reinterpret_cast<const uint4*>(k_cache + row0 * d) + piece + (long long)sub * P;
  constexpr int kBatch = nld < 16 ? nld : 16;
#pragma unroll
  for (int i0 = 0; i0 < nld; i0 += kBatch) {
    uint4 w[kBatch];
#pragma unroll
    for (int i = 0; i < kBatch; ++i) w[i] = __ldg(src + (long long)(i0 + i) * rows_per * P);
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const uint32_t wv[4] = {w[i].x, w[i].y, w[i].z, w[i].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        acc[2 * e] += bf16_lo(wv[e]);
        acc[2 * e + 1] += bf16_hi(wv[e]);
      }
    }
  }
  // lanes holding the same piece of different rows add up (fixed order: a butterfly over `sub`)
#pragma unroll
  for (int o = P; o < 32; o <<= 1)
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], o);
  if (sub == 0) {
    const float inv = 1.0f / (float)(1 << lg);
    uint4 o;
    o.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
    o.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
    o.z = pack_bf16x2(acc[4] * inv, acc[5] * inv);
    o.w = pack_bf16x2(acc[6] * inv, acc[7] * inv);
    reinterpret_cast<uint4*>(kbar + ((long long)blk_base(seg_offsets, s, lg) + b) * d)[piece] = o;
  }
}

struct SelParams {
  const int4* items;   // the attention plan's items {segment * g + j, query tile, seg_offsets[s], n}
  const int* nitems;
  uint32_t* mask;      // [(row * g + j), words]
  uint32_t* status;
  int g, lg, alpha_num, alpha_den, words;
  int kb_rows;         // pooled-key rows of the streaming buffer (kKbBox)
};

template <int D>
__global__ void __launch_bounds__(kSelThreads) sa_select_tc_kernel(const __grid_constant__ CUtensorMap tm_q,
                                                                   const __grid_constant__ CUtensorMap tm_kb,
                                                                   SelParams p) {
  constexpr int kAtoms = D / 64;                          // 128-byte swizzle atoms per row
  constexpr int kQAtomBytes = kSelTileRows * 128;         // 16 KB
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int kb_atom_bytes = p.kb_rows * 128;
  uint8_t* sq = smem;
  uint8_t* skb = smem + kAtoms * kQAtomBytes;
  __shared__ uint64_t bar_load, bar_mma, bar_drain;
  __shared__ uint32_t tmem_base;
  __shared__ int abort_flag;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  pdl_launch_dependents();
  pdl_wait();  // plan, Q~ and the pooled keys come from the kernels before it
  // the item count and this CTA's item load together (the plan holds one item per CTA of the grid)
  const int nitems = *p.nitems;
  const int4 item = p.items[blockIdx.x];
  if ((int)blockIdx.x >= nitems) return;
  const int s = item.x / p.g, j = item.x - s * p.g, qt = item.y, off = item.z, n = item.w;
  const int row0 = qt * kSelTileRows;
  const int r = row0 + (int)threadIdx.x;            // this thread's query rank
  const bool valid = r < n;
  const int cur = r >> p.lg;                         // current block of this query
  const int last_cur = (min(row0 + kSelTileRows, n) - 1) >> p.lg;
  const int nb = min(last_cur, kSelMaxCols);         // block scores this CTA computes
  uint32_t* mrow = p.mask + ((long long)(off + r) * p.g + j) * p.words;
  const int keep_all = valid ? kept_blocks(cur, p.alpha_num, p.alpha_den) : 0;
  if (nb == 0 || __syncthreads_and(keep_all == 0)) {
    // no query of the tile keeps an earlier block: zero mask rows
    if (valid)
      for (int w = 0; w < p.words; ++w) mrow[w] = 0u;
    return;
  }
  const int ncols = (nb + 15) & ~15;                 // N of the MMA (multiple of 16)
  uint32_t alloc = 32;
  while ((int)alloc < ncols) alloc <<= 1;
  const int kbase = (off >> p.lg) + s;  // first pooled-key row of the segment
  // the first loads (the query tile and the first box of pooled keys) go out before the TMEM
  // allocation and the barrier, which they then overlap
  auto issue_loads = [&](int n0) {
    mbar_arrive_expect_tx(&bar_load, (uint32_t)(kAtoms * ((n0 == 0 ? kQAtomBytes : 0) + kKbBox * 128)));
    for (int a = 0; a < kAtoms; ++a) {
      if (n0 == 0) tma_load_2d(sq + a * kQAtomBytes, &tm_q, j * D + a * 64, off + row0, &bar_load);
      tma_load_2d(skb + a * kb_atom_bytes, &tm_kb, a * 64, kbase + n0, &bar_load);
    }
  };
  if (threadIdx.x == 0) {
    mbar_init(&bar_load, 1);
    mbar_init(&bar_mma, 1);
    mbar_init(&bar_drain, 1);
    abort_flag = 0;
    mbar_fence_init();
    issue_loads(0);
  }
  if (warp == 0) {
    tmem_alloc(&tmem_base, alloc);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_base;
  bool ok = true;
  if (warp == 0) {
    // The pooled keys stream through one buffer of kKbBox rows: load a box of blocks, issue its
    // MMAs into the next kKbBox score columns, wait for them, then reuse the buffer.
    const uint64_t q_desc = make_smem_desc_sw128(smem_u32(sq), 16, 1024);
    const uint64_t kb_desc = make_smem_desc_sw128(smem_u32(skb), 16, 1024);
    uint32_t phase = 0;
    for (int n0 = 0; n0 < ncols && ok; n0 += kKbBox, ++phase) {
      if (lane == 0 && n0 > 0) issue_loads(n0);
      __syncwarp();
      ok = __all_sync(0xffffffffu, mbar_wait(&bar_load, phase & 1, &abort_flag, p.status));
      if (!ok) break;
      tc_fence_after();
      const int N = min(kKbBox, ncols - n0);  // a multiple of 16
      const uint32_t idesc = make_idesc_bf16(kSelTileRows, N, false, false);
      // K steps of 16 elements: 32 bytes within the 128-byte atom, then the next atom
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        const uint64_t qo = (uint64_t)(((kk >> 2) * kQAtomBytes + (kk & 3) * 32) >> 4);
        const uint64_t ko = (uint64_t)(((kk >> 2) * kb_atom_bytes + (kk & 3) * 32) >> 4);
        mma_bf16_ss(tmem + (uint32_t)n0, q_desc + qo, kb_desc + ko, idesc, kk > 0 ? 1u : 0u);
      }
      mma_commit(&bar_mma);
      ok = __all_sync(0xffffffffu, mbar_wait(&bar_mma, phase & 1, &abort_flag, p.status));  // buffer free again
    }
  }
  tc_fence_before();
  ok = __syncthreads_and(ok);  // the scores are complete (the MMA warp saw its last commit)
  tc_fence_after();
  if (ok) {
    const uint32_t lane_addr = tmem + ((uint32_t)(warp * 32) << 16);
    const int nchunks = (nb + 31) >> 5;
    // rows handled here: current block within the TMEM scores; the rest go to sa_select_kernel
    const bool mine = valid && cur <= kSelMaxCols;
    const int keep = mine ? keep_all : 0;
    const int cand = mine ? cur : 0;                 // candidate blocks 0 .. cur - 1
    select_from_tmem(lane_addr, nchunks, cand, keep, [&](int c, uint32_t w) {
      if (mine && c < p.words) mrow[c] = w;
    });
    if (mine)
      for (int w = nchunks; w < p.words; ++w) mrow[w] = 0u;
  } else if (warp == 0) {
    // a wait gave up: let an MMA already issued finish before TMEM is released
    mma_commit(&bar_drain);
    const uint64_t t0 = global_timer_ns();
    while (!mbar_try_wait(&bar_drain, 0) && global_timer_ns() - t0 < 100000000ull) {
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, alloc);
}

// Rows whose current block is past kSelMaxCols (histories longer than kSelMaxCols blocks).
__global__ void __launch_bounds__(256) sa_select_kernel(const uint16_t* __restrict__ q_rot,
                                                        const int32_t* __restrict__ seg_offsets, int nseg,
                                                        const int64_t* __restrict__ seg_base,
                                                        const int32_t* __restrict__ seg_cap,
                                                        const uint16_t* __restrict__ kbar, int d, int g, int lg,
                                                        int alpha_num, int alpha_den, long long nq,
                                                        uint32_t* __restrict__ mask, int words) {
  pdl_launch_dependents();
  pdl_wait();
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
  if (cur <= kSelMaxCols || !seg_live(seg_offsets, seg_base, seg_cap, lo)) return;  // done elsewhere
  const int keep = kept_blocks(cur, alpha_num, alpha_den);
  const int per = d / 32;  // columns of q~ and of the pooled keys per lane (2 or 4)
  float ql[4];
#pragma unroll
  for (int e = 0; e < 4; ++e)
    ql[e] = e < per ? __uint_as_float((uint32_t)q_rot[qi * d + lane * per + e] << 16) : 0.f;
  const uint16_t* kb = kbar + (long long)blk_base(seg_offsets, lo, lg) * d + lane * per;
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
        const uint16_t* kr = kb + (long long)b * d;
#pragma unroll
        for (int e = 0; e < 4; ++e)
          if (e < per) a = fmaf(ql[e], __uint_as_float((uint32_t)__ldg(kr + e) << 16), a);
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
    sc[i] = v[0];
  }
  uint32_t taken = 0;  // bit i: block i * 32 + lane kept
  for (int m = 0; m < keep; ++m) {
    // this lane's best remaining block (highest key), then the warp's
    uint32_t best = 0u;
#pragma unroll
    for (int i = 0; i < kPerLane; ++i) {
      if (i >= nslot) break;
      const int b = i * 32 + lane;
      if (b < cur && !((taken >> i) & 1u)) best = max(best, score_key(sc[i], b));
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) best = max(best, __shfl_xor_sync(0xffffffffu, best, o));
    if (best == 0u) break;  // cannot happen: keep <= cur
    const int bb = 0x3FF - (int)(best & 0x3FFu);
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

bool encode_kbar_map(CUtensorMap* map, const void* base, long long rows, int d) {
  EncodeTiledFn enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)d * 2};
  cuuint32_t box[2] = {64u, (cuuint32_t)kKbBox};
  cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
int launch_select_tc(const CUtensorMap& tq, const CUtensorMap& tkb, const SelParams& p, int grid, cudaStream_t stream) {
  const int smem = 1024 + (D / 64) * (kSelTileRows * 128 + p.kb_rows * 128);
  cudaError_t e = cudaFuncSetAttribute(sa_select_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e == cudaSuccess) e = launch_pdl(sa_select_tc_kernel<D>, dim3(grid), dim3(kSelThreads), (size_t)smem, stream,
                                       tq, tkb, p);
  if (e == cudaSuccess) e = cudaGetLastError();
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, "sa_select_tc_kernel launch");
}

}  // namespace sa

// Pooled keys (unless the RoPE pass pooled them: pooled = true), then the selection: the tensor-core
// selector over the attention plan's items, and for histories longer than kSelMaxCols blocks the
// per-query selector for the rows past that.
// q_rot_map is the attention's tensor map of Q~ ([R, g d] rows, 64 x 128 boxes).  kbar holds
// kbar_rows bf16 rows of d.
int launch_sa_select(const CUtensorMap& q_rot_map, const uint16_t* q_rot, const uint16_t* k_cache,
                     const int32_t* seg_offsets, const int64_t* seg_base, const int32_t* seg_cap,
                     long long cache_rows, int nseg, int T, long long R, int d, int g, int lg, int alpha_num,
                     int alpha_den, uint16_t* kbar, long long kbar_rows, uint32_t* mask, int words, const void* plan,
                     int max_items, uint32_t* status, cudaStream_t stream, bool pooled) {
  const int max_blocks = (T + (1 << lg) - 1) >> lg;
  if (nseg > 0 && max_blocks > 0 && !pooled) {
    dim3 grid((max_blocks + 7) / 8, nseg);
    auto pool = d == 128 ? (lg == 5 ? sa::sa_pool_kernel<128, 5> : lg == 6 ? sa::sa_pool_kernel<128, 6>
                                                                            : sa::sa_pool_kernel<128, 7>)
                         : (lg == 5 ? sa::sa_pool_kernel<64, 5> : lg == 6 ? sa::sa_pool_kernel<64, 6>
                                                                           : sa::sa_pool_kernel<64, 7>);
    const cudaError_t e = launch_pdl(pool, grid, dim3(256), 0, stream, k_cache, seg_offsets, seg_base, seg_cap,
                                     cache_rows, g, kbar, mask, words);
    if (e != cudaSuccess) return cuda_fail(e, "sa_pool_kernel launch");
  }
  if (R <= 0 || max_items <= 0) return NAMOH_OK;
  CUtensorMap tkb;
  if (!sa::encode_kbar_map(&tkb, kbar, kbar_rows, d)) return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled");
  sa::SelParams p;
  p.items = reinterpret_cast<const int4*>(static_cast<const char*>(plan) + 16);
  p.nitems = static_cast<const int*>(plan) + 2;
  p.mask = mask;
  p.status = status;
  p.g = g;
  p.lg = lg;
  p.alpha_num = alpha_num;
  p.alpha_den = alpha_den;
  p.words = words;
  p.kb_rows = sa::kKbBox;  // the pooled keys stream through a buffer of one TMA box
  int rc = d == 128 ? sa::launch_select_tc<128>(q_rot_map, tkb, p, max_items, stream)
                    : sa::launch_select_tc<64>(q_rot_map, tkb, p, max_items, stream);
  if (rc != NAMOH_OK) return rc;
  if (max_blocks - 1 > sa::kSelMaxCols) {
    const long long nq = R * g;
    const cudaError_t e = launch_pdl(sa::sa_select_kernel, dim3((unsigned)((nq + 7) / 8)), dim3(256), 0, stream,
                                     q_rot, seg_offsets, nseg, seg_base, seg_cap, (const uint16_t*)kbar, d, g, lg,
                                     alpha_num, alpha_den, nq, mask, words);
    if (e != cudaSuccess) return cuda_fail(e, "sa_select_kernel launch");
  }
  return NAMOH_OK;
}

}  // namespace namoh
