// rope_pack.cu -- head-relative RoPE at the packed rank (Sec. 3.2, Eq. namoh-head-rope).
//
// Packed rows are contiguous in q, k and v, so each block streams chunks of packed rows
// (their g query rows, the key row and, when it is copied, the value row) into shared
// memory with 1D bulk copies through a kRopeStages-deep mbarrier pipeline, and rotates them
// from there: the loads of several chunks are in flight at any time, with no per-thread
// load latency on the way.  A group of D/16 threads owns one packed row of a chunk (for
// g >= 4, half of its query heads or less): the row's segment s comes from a binary search
// over seg_offsets (staged in shared memory), rho = r - seg_offsets[s], and each thread
// rotates 8 pairs (j, j + D/2) with angles it computes once for the row; KV-group routing
// shares the rank between the key and the row's g query heads (App. B.7).
// Variants: the interleaved pairing (2j, 2j+1) keeps the same 16-byte accesses (elements
// [8l, 8l+8) and [D/2 + 8l, D/2 + 8l + 8) for lane l of a group) and pairs adjacent elements
// inside them, so the lane's angles are j = 4l..4l+3 and D/4 + 4l..D/4 + 4l+3; global
// positions (Sec. 3.2: rho_i(t) replaced by t) take t = (row_src[r] / Kr) % T from the
// routing's inverse map, loaded one chunk ahead -- in a ragged batch t = row_src[r] / Kr -
// cu_seqlens[b], b = segment / Hr; the cache row is still the rank.
// Outputs: Q~ (bf16 scratch for the attention kernel), K~ into the key cache, and V copied
// into the value cache unless the caller passed v_cache == v.  Given a plan buffer, block 0
// builds the attention work list in the same launch.  Launched with programmatic dependent
// launch: set-up overlaps the routing kernel's tail, and every read of routing outputs or
// inputs comes after pdl_wait().
// Pooling variants (SA + NAMOH, App. B.8 with the mean-pooled keys of App. B.3): the chunks start at
// multiples of the chunk height within each segment, so each block of 2^lg <= kRows keys lies in
// one chunk; the pass sums the rotated keys it wrote (as bf16) per block and column and stores the
// block means, the pooled keys the selection kernel reads.
#include <type_traits>

#include "common.cuh"
#include "plan.cuh"

namespace namoh {

constexpr int kRopeThreads = 256;
constexpr int kRopeStages = 3;
constexpr int kRopeStageMax = 8192;  // seg_offsets entries staged in shared memory (32 KB)
constexpr size_t kSmemPerSm = 233472;  // shared memory per SM (228 KB); each resident block also takes 1 KB
// the least dynamic shared memory with which three blocks no longer fit on one SM
constexpr size_t kSmemThirdPlus = kSmemPerSm / 3 - 1024 + 16;

template <int D, int G>
struct RopeChunk {
  static constexpr int kLpr = D / 16;                    // threads per group (8 pairs each)
  static constexpr int kGroups = kRopeThreads / kLpr;    // 32 (D = 128) or 64 (D = 64)
  static constexpr int kGpr = G >= 4 ? G / 2 : 1;        // groups per packed row
  static constexpr int kHeads = G / kGpr;                // query heads per group
  static constexpr int kRows = kGroups / kGpr;           // packed rows per chunk
  static constexpr int kRowsLg = kRows == 64 ? 6 : kRows == 32 ? 5 : kRows == 16 ? 4 : 3;
  static constexpr int kWarps = kRopeThreads / 32;
  static constexpr int kPartStride = D + 4;  // floats per row of per-warp column sums (padded: no bank conflicts)
  // pooling: two sets of per-warp column sums, each stage's chunk {segment, first row, rows}, and the
  // angle table (theta_hi, theta_lo)
  static constexpr int kPartBytes = 2 * kWarps * kPartStride * 4 + 64 + 2 * 64 * 4;
  static constexpr int kQBytes = kRows * G * D * 2;
  static constexpr int kKBytes = kRows * D * 2;
  static constexpr int kStageBytes = kQBytes + 2 * kKBytes;  // Q, K, V
  static_assert(kStageBytes % 128 == 0, "stage alignment");
  static_assert((1 << kRowsLg) == kRows, "chunk height");
};

__host__ __device__ constexpr size_t rope_offs_bytes(int nseg) {
  return nseg + 1 <= kRopeStageMax ? ((size_t)(nseg + 1) * 4 + 15) / 16 * 16 : 0;
}

// shared memory: the stages, the pooling sums (pool variants), the staged seg_offsets, the barriers
template <int D, int G>
__host__ __device__ constexpr size_t rope_smem_bytes(int nseg, bool pool) {
  return (size_t)kRopeStages * RopeChunk<D, G>::kStageBytes + (pool ? RopeChunk<D, G>::kPartBytes : 0) +
         rope_offs_bytes(nseg) + kRopeStages * sizeof(uint64_t);
}

// Packed rows per chunk of the RoPE pass (host): blocks of SA + NAMOH up to this size pool in the pass.
int rope_chunk_rows(int D, int g) {
  const int lpr = D / 16, groups = kRopeThreads / lpr, gpr = g >= 4 ? g / 2 : 1;
  return groups / gpr;
}

// kFlags: NAMOH_ROPE_INTERLEAVED, NAMOH_ROPE_GLOBAL, kRopeRagged (global positions in a ragged
// batch) and kRopePool (SA + NAMOH block pooling), compile-time so that no variant carries another's
// branches
constexpr unsigned kRopeRagged = 0x4u;
constexpr unsigned kRopePool = 0x8u;

template <int D, int G, unsigned kFlags>
__global__ void __launch_bounds__(kRopeThreads) rope_pack_kernel(
    const uint16_t* __restrict__ q, const uint16_t* __restrict__ k, const uint16_t* __restrict__ v, int R,
    const int32_t* __restrict__ seg_offsets, int nseg, const int64_t* __restrict__ seg_base,
    const int32_t* __restrict__ seg_cap, long long cache_rows, uint16_t* __restrict__ q_rot,
    uint16_t* __restrict__ k_cache, uint16_t* __restrict__ v_cache, int copy_v, RopeTable tab,
    uint32_t* __restrict__ status, int* __restrict__ plan_header, int4* __restrict__ plan_items,
    const int32_t* __restrict__ plan_cap, int plan_qtiles, const int32_t* __restrict__ pos_row_src,
    FastDiv pos_k, FastDiv pos_t, const int32_t* __restrict__ pos_cu, FastDiv pos_hr, RopePool pool) {
  using C = RopeChunk<D, G>;
  constexpr int HALF = D / 2;
  constexpr bool kInterleaved = (kFlags & NAMOH_ROPE_INTERLEAVED) != 0;
  constexpr bool kGlobal = (kFlags & NAMOH_ROPE_GLOBAL) != 0;
  constexpr bool kRagged = (kFlags & kRopeRagged) != 0;
  constexpr bool kPool = (kFlags & kRopePool) != 0;
  extern __shared__ __align__(128) uint8_t smem_raw[];
  __shared__ int s_abort;
  pdl_launch_dependents();  // the attention kernel may start launching; it waits for this grid
  const int first = plan_header ? 1 : 0;
  if ((int)blockIdx.x < first) {
    pdl_wait();
    build_plan(seg_offsets, nseg, plan_cap, G, plan_qtiles, plan_header, plan_items, reinterpret_cast<int*>(smem_raw));
    return;
  }
  const int nblk = gridDim.x - first, blk = blockIdx.x - first;
  // chunk numbers: kRows consecutive packed rows each; with pooling, segment s owns the numbers
  // seg_offsets[s] / kRows + s + i (chunk i of the segment starts at its row i kRows), at least
  // ceil(n_s / kRows) of them, so the last number of a segment may hold no row
  const int nchunks = kPool ? (R >> C::kRowsLg) + nseg : (R + C::kRows - 1) / C::kRows;
  constexpr int kPartBytes = kPool ? C::kPartBytes : 0;
  uint8_t* stages = smem_raw;
  float* part = reinterpret_cast<float*>(smem_raw + kRopeStages * C::kStageBytes);  // [2][kWarps][kPartStride]
  int4* s_chunk = reinterpret_cast<int4*>(smem_raw + kRopeStages * C::kStageBytes + 2 * C::kWarps * C::kPartStride * 4);
  float* s_theta = reinterpret_cast<float*>(s_chunk + 4);  // pooling variants: [theta_hi[64], theta_lo[64]]
  int32_t* s_offs = reinterpret_cast<int32_t*>(smem_raw + kRopeStages * C::kStageBytes + kPartBytes);
  uint64_t* full =
      reinterpret_cast<uint64_t*>(smem_raw + kRopeStages * C::kStageBytes + kPartBytes + rope_offs_bytes(nseg));
  const bool staged = nseg + 1 <= kRopeStageMax;

  // rows r0 .. r0 + rows - 1 of chunk c (rows <= 0: none) and, with pooling, their segment s
  auto locate = [&](int c, const int32_t* o, int& s, int& r0) -> int {
    if constexpr (!kPool) {
      s = 0;
      r0 = c * C::kRows;
      return min(C::kRows, R - r0);
    } else {
      int lo = 0, hi = nseg;  // last s with seg_offsets[s] / kRows + s <= c
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if ((o[mid] >> C::kRowsLg) + mid <= c) lo = mid; else hi = mid;
      }
      const int base = o[lo];
      s = lo;
      r0 = base + ((c - (base >> C::kRowsLg) - lo) << C::kRowsLg);
      return r0 < 0 ? 0 : min(min(C::kRows, o[lo + 1] - r0), R - r0);
    }
  };
  // chunk c into stage st: its rows' Q (g rows each), K and V, one bulk copy per array
  auto issue = [&](int c, int st, const int32_t* o) {
    int s_ = 0, r0 = c * C::kRows;
    const int rows = kPool ? max(locate(c, o, s_, r0), 0) : min(C::kRows, R - r0);
    // the chunk's place, for the threads that wait on this stage (the arrive below releases it)
    if constexpr (kPool) s_chunk[st] = make_int4(s_, r0, rows, 0);
    uint8_t* base = stages + st * C::kStageBytes;
    const uint32_t qb = (uint32_t)rows * G * D * 2, kb = (uint32_t)rows * D * 2;
    mbar_arrive_expect_tx(&full[st], qb + kb + (copy_v ? kb : 0u));  // no bytes: the phase completes here
    if (!kPool || rows > 0) {
      bulk_load(base, q + (size_t)r0 * G * D, qb, &full[st]);
      bulk_load(base + C::kQBytes, k + (size_t)r0 * D, kb, &full[st]);
      if (copy_v) bulk_load(base + C::kQBytes + C::kKBytes, v + (size_t)r0 * D, kb, &full[st]);
    }
  };
  if (threadIdx.x == 0) {
    for (int i = 0; i < kRopeStages; ++i) mbar_init(&full[i], 1);
    s_abort = 0;
    mbar_fence_init();
  }
  pdl_wait();  // routing outputs (and q, k, v) are visible from here
  if (threadIdx.x == 0)
    for (int i = 0; i < kRopeStages; ++i)
      if (blk + i * nblk < nchunks) issue(blk + i * nblk, i, seg_offsets);
  if (staged)
    for (int i = threadIdx.x; i <= nseg; i += blockDim.x) s_offs[i] = __ldg(seg_offsets + i);
  if constexpr (kPool) {
    if (threadIdx.x < 64) {
      s_theta[threadIdx.x] = tab.theta_hi[threadIdx.x];
      s_theta[64 + threadIdx.x] = tab.theta_lo[threadIdx.x];
    }
  }
  __syncthreads();
  const int32_t* offs = staged ? s_offs : seg_offsets;

  const int grp = threadIdx.x / C::kLpr, lig = threadIdx.x % C::kLpr;
  const int prow = grp / C::kGpr;  // packed row within the chunk
  const int hsub = grp % C::kGpr;  // which share of the row's query heads
  const int j0 = lig * 8;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float th_hi[8], th_lo[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int j = kInterleaved ? (i < 4 ? 4 * lig + i : D / 4 + 4 * lig + i - 4) : j0 + i;
    if constexpr (kPool) {
      // from shared memory: a value loaded from the parameter bank may be loaded again in every
      // chunk, and per-lane indices there serialise
      th_hi[i] = s_theta[j];
      th_lo[i] = s_theta[64 + j];
    } else {
      th_hi[i] = opaque_f32(tab.theta_hi[j]);  // kept in registers across the chunk loop
      th_lo[i] = opaque_f32(tab.theta_lo[j]);
    }
  }
  bool ok = true;
  int it = 0;
  // global positions: row_src of this thread's row in the next chunk, loaded a chunk ahead
  int token_next = 0;
  if constexpr (kGlobal && kPool) {
    int s_, r0;
    if (blk < nchunks && prow < locate(blk, offs, s_, r0)) token_next = __ldg(pos_row_src + r0 + prow);
  } else if (kGlobal) {
    const long long r_first = (long long)blk * C::kRows + prow;
    if (blk < nchunks && r_first < R) token_next = __ldg(pos_row_src + r_first);
  }
  for (int c = blk; c < nchunks; c += nblk, ++it) {
    const int st = it % kRopeStages;
    int token_src = 0;  // row_src of this thread's row: (b*T + t)*Kr + slot
    if constexpr (kGlobal && kPool) {
      token_src = token_next;
      int s_, r0n;
      if (c + nblk < nchunks && prow < locate(c + nblk, offs, s_, r0n)) token_next = __ldg(pos_row_src + r0n + prow);
    } else if (kGlobal) {
      token_src = token_next;
      const long long r_next = (long long)(c + nblk) * C::kRows + prow;
      if (c + nblk < nchunks && r_next < R) token_next = __ldg(pos_row_src + r_next);
    }
    ok = mbar_wait(&full[st], (it / kRopeStages) & 1, &s_abort, status);
    if (!__syncthreads_and(ok)) {
      ok = false;
      break;
    }
    const uint8_t* base = stages + st * C::kStageBytes;
    int cseg = 0, cr0 = 0, crows = 0;
    if constexpr (kPool) {
      const int4 ci = s_chunk[st];
      cseg = ci.x;
      cr0 = ci.y;
      crows = ci.z;
    }
    const long long r = kPool ? (long long)cr0 + prow : (long long)c * C::kRows + prow;
    float pk[16];  // pooling: this thread's columns of its rotated key row, 0 without one
#pragma unroll
    for (int e = 0; e < 16; ++e) pk[e] = 0.f;
    // pooling: the blocks of a segment pool only when all its rows are in the cache
    const bool live = !kPool || !seg_base || offs[cseg + 1] - offs[cseg] <= __ldg(seg_cap + cseg);
    if (kPool ? prow < crows : r < R) {
      // segment of row r: last s with seg_offsets[s] <= r (with pooling, the chunk's segment)
      int lo = cseg;
      if constexpr (!kPool) {
        int hi = nseg;
        lo = 0;
        while (hi - lo > 1) {
          const int mid = (lo + hi) >> 1;
          if (offs[mid] <= r) lo = mid; else hi = mid;
        }
      }
      const int rho = (int)(r - offs[lo]);
      // position: the rank, or the token's index t in its sequence
      float pos = (float)rho;
      if (kGlobal) {
        const uint32_t tok = fastdiv((uint32_t)token_src, pos_k);  // b*T + t, or the flat token index
        if constexpr (kRagged)
          pos = (float)((int)tok - __ldg(pos_cu + fastdiv((uint32_t)lo, pos_hr)));
        else
          pos = (float)(tok - fastdiv(tok, pos_t) * pos_t.d);
      }
      float sn[8], cs[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) rope_sincos(pos, th_hi[i], th_lo[i], tab, &sn[i], &cs[i]);

      // x'_j = x_j cos - x_{j+D/2} sin ;  x'_{j+D/2} = x_{j+D/2} cos + x_j sin
      // (interleaved: the same with x_{2j} and x_{2j+1}, one bf16x2 word per pair)
      // pooled (pool variants, key rows): the rotated bf16 values of columns j0 .. j0 + 7, then
      // D/2 + j0 .. D/2 + j0 + 7, added to the pooling sums (both pairings write those columns)
      auto rotate = [&](const uint8_t* src_row, uint16_t* dst_row, bool pooled) {
        if constexpr (kInterleaved) {
          const uint4 a = *reinterpret_cast<const uint4*>(src_row + j0 * 2);
          const uint4 b = *reinterpret_cast<const uint4*>(src_row + (HALF + j0) * 2);
          const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
          uint32_t o[8];
#pragma unroll
          for (int p = 0; p < 8; ++p) {
            const float x0 = bf16_lo(w[p]), x1 = bf16_hi(w[p]);
            o[p] = pack_bf16x2(fmaf(x0, cs[p], -x1 * sn[p]), fmaf(x1, cs[p], x0 * sn[p]));
          }
          *reinterpret_cast<uint4*>(dst_row + j0) = make_uint4(o[0], o[1], o[2], o[3]);
          *reinterpret_cast<uint4*>(dst_row + HALF + j0) = make_uint4(o[4], o[5], o[6], o[7]);
          if constexpr (kPool) {
            if (pooled) {
#pragma unroll
              for (int p = 0; p < 8; ++p) {
                pk[2 * p] = bf16_lo(o[p]);
                pk[2 * p + 1] = bf16_hi(o[p]);
              }
            }
          }
        } else {
          const uint4 a = *reinterpret_cast<const uint4*>(src_row + j0 * 2);
          const uint4 b = *reinterpret_cast<const uint4*>(src_row + (HALF + j0) * 2);
          const uint32_t av[4] = {a.x, a.y, a.z, a.w};
          const uint32_t bv[4] = {b.x, b.y, b.z, b.w};
          uint32_t oa[4], ob[4];
#pragma unroll
          for (int p = 0; p < 4; ++p) {
            const float x0 = bf16_lo(av[p]), x1 = bf16_hi(av[p]);
            const float y0 = bf16_lo(bv[p]), y1 = bf16_hi(bv[p]);
            const int i0 = 2 * p, i1 = 2 * p + 1;
            oa[p] = pack_bf16x2(fmaf(x0, cs[i0], -y0 * sn[i0]), fmaf(x1, cs[i1], -y1 * sn[i1]));
            ob[p] = pack_bf16x2(fmaf(y0, cs[i0], x0 * sn[i0]), fmaf(y1, cs[i1], x1 * sn[i1]));
          }
          *reinterpret_cast<uint4*>(dst_row + j0) = make_uint4(oa[0], oa[1], oa[2], oa[3]);
          *reinterpret_cast<uint4*>(dst_row + HALF + j0) = make_uint4(ob[0], ob[1], ob[2], ob[3]);
          if constexpr (kPool) {
            if (pooled) {
#pragma unroll
              for (int p = 0; p < 4; ++p) {
                pk[2 * p] = bf16_lo(oa[p]);
                pk[2 * p + 1] = bf16_hi(oa[p]);
                pk[8 + 2 * p] = bf16_lo(ob[p]);
                pk[8 + 2 * p + 1] = bf16_hi(ob[p]);
              }
            }
          }
        }
      };
#pragma unroll
      for (int h = 0; h < C::kHeads; ++h) {
        const int head = hsub * C::kHeads + h;
        rotate(base + ((size_t)prow * G + head) * D * 2, q_rot + ((size_t)r * G + head) * D, false);
      }
      if (hsub == 0) {
        long long dst = r;
        bool write_cache = true;
        if (seg_base) {
          dst = __ldg(seg_base + lo) + rho;
          if (rho >= __ldg(seg_cap + lo) || dst < 0 || dst >= cache_rows) {
            write_cache = false;
            if (lig == 0) report(status, NAMOH_DEV_CAPACITY);
          }
        }
        if (write_cache) {
          rotate(base + C::kQBytes + (size_t)prow * D * 2, k_cache + (size_t)dst * D, live);
          if (copy_v) {
            const uint4* vs = reinterpret_cast<const uint4*>(base + C::kQBytes + C::kKBytes + (size_t)prow * D * 2);
            uint4* vd = reinterpret_cast<uint4*>(v_cache + (size_t)dst * D);
            vd[lig] = vs[lig];
            vd[lig + C::kLpr] = vs[lig + C::kLpr];
          }
        }
      }
      if constexpr (kPool) {
        // a segment not in the cache keeps no block: its rows' mask words are zero
        if (!live && pool.mask) {
          uint32_t* mrow = pool.mask + r * G * pool.words;
          for (int i = hsub * C::kLpr + lig; i < G * pool.words; i += C::kLpr * C::kGpr) mrow[i] = 0u;
        }
      }
    }
    if constexpr (kPool) {
      // The warp's rows lie in one block (blocks hold 32 rows or more, a warp's rows are
      // consecutive).  Their column sums by a reduce-scatter over the lane bits above lig: at each
      // step a lane keeps half of its values (the upper half when its bit is set) and adds the
      // partner's copy of that half, so each sum is formed once, in a fixed order.  Afterwards lane
      // l holds kNf consecutive columns of the warp's sums and stores them.
      constexpr int kRounds = C::kLpr == 8 ? 2 : 3;  // log2(32 / kLpr)
      constexpr int kNf = 16 >> kRounds;
      int e0 = 0;  // first of this lane's kept values (index into pk)
#pragma unroll
      for (int rd = 0; rd < kRounds; ++rd) {
        const int o = C::kLpr << rd, half = 16 >> (rd + 1);
        const bool up = (lane & o) != 0;
        e0 += up ? half : 0;
#pragma unroll
        for (int j = 0; j < half; ++j) {
          const float send = up ? pk[j] : pk[j + half];
          const float keep = up ? pk[j + half] : pk[j];
          pk[j] = keep + __shfl_xor_sync(0xffffffffu, send, o);
        }
      }
      const int col0 = e0 < 8 ? j0 + e0 : HALF + j0 + e0 - 8;
      float* pw = part + ((it & 1) * C::kWarps + warp) * C::kPartStride + col0;
      if constexpr (kNf == 4) *reinterpret_cast<float4*>(pw) = make_float4(pk[0], pk[1], pk[2], pk[3]);
      else *reinterpret_cast<float2*>(pw) = make_float2(pk[0], pk[1]);
    }
    __syncthreads();  // stage st fully read: refill it
    if (threadIdx.x == 0 && c + kRopeStages * nblk < nchunks) issue(c + kRopeStages * nblk, st, offs);
    if constexpr (kPool) {
      // The chunk's complete blocks: nsplit adjacent threads share (block i, column col), each
      // adding its run of the block's warps in order, then a butterfly over the nsplit lanes (the
      // same sum on each of them); the first scales by 1 / 2^lg (exact), rounds to bf16 and stores.
      // The sums of the next chunk go to the other half of `part`, and the barrier after them
      // orders these reads before that half's reuse.
      const int bpc = C::kRows >> pool.lg;  // blocks per chunk
      const int nsplit = kRopeThreads / (bpc * D), wpb = C::kWarps / bpc, wper = wpb / nsplit;
      const int pair = (int)threadIdx.x / nsplit, sub = (int)threadIdx.x % nsplit;
      const int i = pair / D, col = pair % D;
      const float* pc = part + (it & 1) * C::kWarps * C::kPartStride + col;
      float acc = 0.f;
      for (int w = i * wpb + sub * wper; w < i * wpb + (sub + 1) * wper; ++w) acc += pc[w * C::kPartStride];
      for (int o = 1; o < nsplit; o <<= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
      if (sub == 0 && live && crows > 0) {
        const int s0 = offs[cseg], n = offs[cseg + 1] - s0;
        const int b = ((cr0 - s0) >> pool.lg) + i;  // block of the segment
        if (((b + 1) << pool.lg) <= n) {
          const uint32_t pb = pack_bf16x2(acc * (1.0f / (float)(1 << pool.lg)), 0.f);
          pool.kbar[((long long)(s0 >> pool.lg) + cseg + b) * D + col] = (uint16_t)(pb & 0xFFFFu);
        }
      }
    }
  }
  if (!ok && threadIdx.x == 0) {
    // a wait gave up: let bulk copies still in flight land before the block exits
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 1000000ull) {
    }
  }
}

// The launch of one variant: a grid of two blocks per SM (one when the shared memory does not fit
// twice), plus the plan block.
template <int D, int G, unsigned F>
cudaError_t launch_rope_variant(int sm_count, int nseg, size_t plan_smem, bool with_plan, cudaStream_t stream,
                                const uint16_t* q, const uint16_t* k, const uint16_t* v, int R,
                                const int32_t* seg_offsets, const int64_t* seg_base, const int32_t* seg_cap,
                                long long cache_rows, uint16_t* q_rot, uint16_t* k_cache, uint16_t* v_cache,
                                int copy_v, const RopeTable& tab, uint32_t* status, int* plan_header,
                                int4* plan_items, const int32_t* plan_cap, int plan_qtiles,
                                const int32_t* pos_row_src, FastDiv pos_k, FastDiv pos_t, const int32_t* pos_cu,
                                FastDiv pos_hr, const RopePool& pool) {
  using C = RopeChunk<D, G>;
  constexpr bool kPool = (F & kRopePool) != 0;
  if constexpr (kPool && C::kRows < 32) {
    return cudaErrorInvalidValue;  // chunks shorter than the smallest block: pooling runs on its own
  } else {
    const auto kernel = rope_pack_kernel<D, G, F>;
    const size_t rope_smem = rope_smem_bytes<D, G>(nseg, kPool);
    const size_t smem0 = rope_smem > plan_smem ? rope_smem : plan_smem;
    // two blocks per SM when their shared memory fits (228 KB per SM, 1 KB reserved per block); the
    // block scheduler packs blocks as deep as resources allow, so each block also asks for more than
    // a third of the SM, which keeps it to two per SM and spreads the grid over every SM
    const int per_sm = (smem0 + 1024) * 2 <= kSmemPerSm ? 2 : 1;
    const size_t smem = per_sm == 2 && smem0 < kSmemThirdPlus ? kSmemThirdPlus : smem0;
    const long long nchunks = kPool ? ((long long)R >> C::kRowsLg) + nseg : ((long long)R + C::kRows - 1) / C::kRows;
    // the plan block takes one of the per_sm * sm_count slots: the whole grid is resident at once
    long long blocks = (long long)per_sm * sm_count - (with_plan ? 1 : 0);
    if (blocks > nchunks) blocks = nchunks;
    const long long grid = blocks + (with_plan ? 1 : 0);
    if (grid == 0) return cudaSuccess;
    if (smem > 48 * 1024) {
      cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
      if (e != cudaSuccess) return e;
    }
    return launch_pdl(kernel, dim3((unsigned)grid), dim3(kRopeThreads), smem, stream, q, k, v, R, seg_offsets, nseg,
                      seg_base, seg_cap, cache_rows, q_rot, k_cache, v_cache, copy_v, tab, status, plan_header,
                      plan_items, plan_cap, plan_qtiles, pos_row_src, pos_k, pos_t, pos_cu, pos_hr, pool);
  }
}

// pool: with a non-null kbar the pass also pools the SA + NAMOH blocks (2^lg <= rope_chunk_rows(D, g))
cudaError_t launch_rope_pack(int D, const uint16_t* q, const uint16_t* k, const uint16_t* v, int R, int g,
                             const int32_t* seg_offsets, int nseg, const int64_t* seg_base, const int32_t* seg_cap,
                             long long cache_rows, uint16_t* q_rot, uint16_t* k_cache, uint16_t* v_cache, bool copy_v,
                             const RopeTable& tab, uint32_t* status, int sm_count, cudaStream_t stream,
                             void* plan, int plan_qtiles, const int32_t* plan_cap, const int32_t* pos_row_src,
                             int pos_k, int pos_t, const int32_t* pos_cu, int pos_hr, bool interleaved,
                             const RopePool* pool) {
  int* plan_header = static_cast<int*>(plan);
  int4* plan_items = plan ? reinterpret_cast<int4*>(static_cast<char*>(plan) + 16) : nullptr;
  const size_t plan_smem = plan ? (size_t)plan_smem_ints(plan_qtiles, nseg) * sizeof(int) : 0;
  if (R == 0 && !plan) return cudaSuccess;
  const bool pooled = pool && pool->kbar;
  if (pooled && (1 << pool->lg) > rope_chunk_rows(D, g)) return cudaErrorInvalidValue;
  const RopePool pl = pooled ? *pool : RopePool{nullptr, nullptr, 0, 0};
  const unsigned flags = (interleaved ? NAMOH_ROPE_INTERLEAVED : 0u) | (pos_row_src ? NAMOH_ROPE_GLOBAL : 0u) |
                         (pos_row_src && pos_cu ? kRopeRagged : 0u);
  auto go = [&](auto d_tag, auto f_tag) -> cudaError_t {
    constexpr int DD = decltype(d_tag)::value;
    constexpr unsigned FF = decltype(f_tag)::value;
    auto one = [&](auto g_tag) {
      return launch_rope_variant<DD, decltype(g_tag)::value, FF>(
          sm_count, nseg, plan_smem, plan != nullptr, stream, q, k, v, R, seg_offsets, seg_base, seg_cap, cache_rows,
          q_rot, k_cache, v_cache, copy_v ? 1 : 0, tab, status, plan_header, plan_items, plan_cap, plan_qtiles,
          pos_row_src, make_fastdiv((uint32_t)pos_k), make_fastdiv((uint32_t)pos_t), pos_cu,
          make_fastdiv((uint32_t)pos_hr), pl);
    };
    switch (g) {
      case 1: return one(std::integral_constant<int, 1>{});
      case 2: return one(std::integral_constant<int, 2>{});
      case 4: return one(std::integral_constant<int, 4>{});
      case 8: return one(std::integral_constant<int, 8>{});
      default: return cudaErrorInvalidValue;
    }
  };
  using D64 = std::integral_constant<int, 64>;
  using D128 = std::integral_constant<int, 128>;
  auto by_d = [&](auto f_tag) { return D == 128 ? go(D128{}, f_tag) : go(D64{}, f_tag); };
  auto by_flags = [&](auto pool_tag) -> cudaError_t {
    constexpr unsigned P = decltype(pool_tag)::value;
    switch (flags) {
      case 0u: return by_d(std::integral_constant<unsigned, 0u | P>{});
      case 1u: return by_d(std::integral_constant<unsigned, 1u | P>{});
      case 2u: return by_d(std::integral_constant<unsigned, 2u | P>{});
      case 3u: return by_d(std::integral_constant<unsigned, 3u | P>{});
      case 6u: return by_d(std::integral_constant<unsigned, 6u | P>{});
      default: return by_d(std::integral_constant<unsigned, 7u | P>{});
    }
  };
  return pooled ? by_flags(std::integral_constant<unsigned, kRopePool>{})
                : by_flags(std::integral_constant<unsigned, 0u>{});
}

}  // namespace namoh
