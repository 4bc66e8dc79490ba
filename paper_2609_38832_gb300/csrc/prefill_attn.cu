// prefill_attn.cu -- routed causal attention over packed (batch, head) segments with the
// gate-weighted combine fused into the epilogue (Sec. 3.1, Eq. namoh-attention; Sec. 3.2
// "Efficient execution": packed variable-length subsequences and length-aware scheduling;
// App. C "Adopted KV-group routing" for g > 1).
//
// Work unit ("item"): one 128-row query tile of one segment for one group head j.  Within
// a segment, queries and keys share local ranks, so query tile qt needs key tiles 0..qt
// and only tile qt is masked (key rank <= query rank).
//
// Schedule (length-aware, longest first): a one-block "plan" kernel lists the items in
// order of decreasing cost (qt + 1 key tiles).  The persistent attention kernel launches
// one CTA per SM; each CTA's producer warp takes the next item from an atomic counter
// (greedy list scheduling in longest-first order) and hands it to the other warps through
// a two-slot ring in shared memory.  The last CTA to finish resets the counter, so a plan
// can be reused by later launches on the same stream.
//
// Attention CTA (192 threads, one CTA per SM):
//   warp 0      TMA producer: Q tile, then K and V tiles into 2-stage rings (128B swizzle)
//   warp 1      MMA issuer (one lane) and TMEM owner: S = Q K^T into one of two TMEM
//               S buffers, then O += P V into the TMEM O accumulator (tcgen05, M = 128)
//   warps 2-5   softmax / epilogue: thread i owns query row i (TMEM lane i).  Online
//               softmax in fp32 with exp2; the running max is only moved when it grows by
//               more than 2^8 (then O in TMEM is rescaled); P is written to shared memory
//               as bf16 in the MMA operand layout.  The epilogue divides by the row sum,
//               multiplies by the routing gate and scatters bf16 rows to y[row_src].
// TMEM: S0 = cols [0,128), S1 = [128,256), O = [256, 256 + D).
// Every mbarrier wait is bounded (NAMOH_DEV_TIMEOUT, then all roles drain and exit).
#include "common.cuh"

namespace namoh {

cudaError_t launch_rope_pack(int D, const uint16_t* q, const uint16_t* k, const uint16_t* v, int R, int g,
                             const int32_t* seg_offsets, int nseg, const int64_t* seg_base, const int32_t* seg_cap,
                             long long cache_rows, uint16_t* q_rot, uint16_t* k_cache, uint16_t* v_cache, bool copy_v,
                             const RopeTable& tab, uint32_t* status, int sm_count, cudaStream_t stream);

namespace attn {

constexpr int BM = 128;             // query rows per tile
constexpr int BN = 128;             // keys per tile
constexpr int kThreads = 192;       // 6 warps
constexpr int kTmemCols = 512;
constexpr int kTmemS0 = 0, kTmemS1 = 128, kTmemO = 256;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

template <int D>
struct Smem {
  static constexpr int kAtoms = D / 64;                  // 64-column (128-byte) swizzle atoms per row
  static constexpr int kTileBytes = BM * D * 2;          // one Q / K / V tile
  static constexpr int kAtomBytes = BM * 128;            // 16 KB: 128 rows x 128 bytes
  static constexpr int kQ = 0;
  static constexpr int kK0 = kQ + kTileBytes;
  static constexpr int kV0 = kK0 + 2 * kTileBytes;
  static constexpr int kP = kV0 + 2 * kTileBytes;
  static constexpr int kPBytes = BM * BN * 2;
  static constexpr int kBar = kP + kPBytes;
  static constexpr int kBytes = kBar + 256;
  static constexpr int kAlloc = kBytes + 1024;           // slack for 1024-byte alignment
};

struct Bars {
  uint64_t item_full[2], item_empty[2];
  uint64_t q_full, q_empty;
  uint64_t k_full[2], k_empty[2];
  uint64_t v_full[2], v_empty[2];
  uint64_t s_full[2], s_free[2];
  uint64_t p_full, o_ready, o_free;
  uint64_t drain;
  int2 item_slot[2];
  uint32_t tmem_base;
  int abort_flag;
};

struct Params {
  const int32_t* seg_offsets;  // [nseg + 1]
  const int64_t* seg_base;     // [nseg] or null (cache rows = packed rows)
  const int32_t* row_src;      // [R]
  const float* gate;           // [R] indexed by row_src value
  const int2* items;           // {segment * g + j, qt}, longest first
  const int* nitems;
  int* sched;                  // [0] next item, [1] CTAs finished
  uint16_t* y;                 // [R * g, D] indexed by row_src * g + j
  int g;
  float scale_log2;            // log2(e) / sqrt(D)
  uint32_t* status;
};

// All lanes of a warp wait and agree on the outcome, so warp-collective tcgen05
// instructions after the wait never diverge on a timeout race.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, uint32_t* status) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status);
  return __all_sync(0xffffffffu, ok);
}

// Consumer side of the item ring: every lane waits, reads the item, one lane releases the slot.
__device__ __forceinline__ bool take_item(Bars* bars, uint32_t idx, int2* item, volatile int* abort_flag,
                                          uint32_t* status) {
  const int slot = idx & 1;
  if (!warp_wait(&bars->item_full[slot], (idx >> 1) & 1, abort_flag, status)) return false;
  const volatile int* src = reinterpret_cast<const volatile int*>(&bars->item_slot[slot]);
  item->x = src[0];
  item->y = src[1];
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&bars->item_empty[slot]);
  return true;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                    const __grid_constant__ CUtensorMap tm_v, Params p) {
  using L = Smem<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + L::kBar);
  volatile int* abort_flag = &bars->abort_flag;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int G = gridDim.x;
  const int nitems = *p.nitems;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->item_full[i], 1);
      mbar_init(&bars->item_empty[i], 5);  // MMA warp + 4 softmax warps
    }
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->k_full[i], 1);
      mbar_init(&bars->k_empty[i], 1);
      mbar_init(&bars->v_full[i], 1);
      mbar_init(&bars->v_empty[i], 1);
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_free[i], 4);
    }
    mbar_init(&bars->p_full, 4);
    mbar_init(&bars->o_ready, 1);
    mbar_init(&bars->o_free, 4);
    mbar_init(&bars->drain, 1);
    bars->abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;

  if (warp == 0) {
    // ------------------------------------------------------------------ producer
    if (lane == 0) {
      uint32_t kv_iter = 0, item_iter = 0;
      bool ok = true;
      while (ok) {
        const int it = atomicAdd(p.sched, 1);
        const int2 item = it < nitems ? p.items[it] : make_int2(-1, -1);
        const int slot = item_iter & 1;
        if (item_iter >= 2) ok = mbar_wait(&bars->item_empty[slot], ((item_iter >> 1) - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        bars->item_slot[slot] = item;
        mbar_arrive(&bars->item_full[slot]);
        if (item.x < 0) break;
        const int seg = item.x / p.g, j = item.x % p.g, qt = item.y;
        const int off = p.seg_offsets[seg];
        const long long kvb = p.seg_base ? p.seg_base[seg] : (long long)off;
        if (item_iter > 0) ok = mbar_wait(&bars->q_empty, (item_iter - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        mbar_arrive_expect_tx(&bars->q_full, L::kTileBytes);
        for (int a = 0; a < L::kAtoms; ++a)
          tma_load_2d(smem + L::kQ + a * L::kAtomBytes, &tm_q, j * D + a * 64, off + qt * BM, &bars->q_full);
        for (int kv = 0; kv <= qt && ok; ++kv, ++kv_iter) {
          const int st = kv_iter & 1;
          const uint32_t use = kv_iter >> 1;
          if (use > 0) ok = mbar_wait(&bars->k_empty[st], (use - 1) & 1, abort_flag, p.status);
          if (!ok) break;
          mbar_arrive_expect_tx(&bars->k_full[st], L::kTileBytes);
          for (int a = 0; a < L::kAtoms; ++a)
            tma_load_2d(smem + L::kK0 + st * L::kTileBytes + a * L::kAtomBytes, &tm_k, a * 64,
                        (int)(kvb + (long long)kv * BN), &bars->k_full[st]);
          if (use > 0) ok = mbar_wait(&bars->v_empty[st], (use - 1) & 1, abort_flag, p.status);
          if (!ok) break;
          mbar_arrive_expect_tx(&bars->v_full[st], L::kTileBytes);
          for (int a = 0; a < L::kAtoms; ++a)
            tma_load_2d(smem + L::kV0 + st * L::kTileBytes + a * L::kAtomBytes, &tm_v, a * 64,
                        (int)(kvb + (long long)kv * BN), &bars->v_full[st]);
        }
        ++item_iter;
      }
      if (!ok) {
        // drain: let copies already in flight land before the CTA exits
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 1000000ull) {
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_qk = make_idesc_bf16(BM, BN, false, false);
    constexpr uint32_t idesc_pv = make_idesc_bf16(BM, D, false, true);
    const uint32_t q_addr = smem_u32(smem + L::kQ);
    const uint32_t p_addr = smem_u32(smem + L::kP);
    uint32_t kv_iter = 0, s_iter = 0, pv_iter = 0, item_iter = 0;
    bool ok = true;
    while (ok) {
      int2 item;
      ok = take_item(bars, item_iter, &item, abort_flag, p.status);
      if (!ok || item.x < 0) break;
      const int seg = item.x / p.g, qt = item.y;
      const int n = p.seg_offsets[seg + 1] - p.seg_offsets[seg];
      const int nkv = qt + 1;
      ok = warp_wait(&bars->q_full, item_iter & 1, abort_flag, p.status);
      for (int jj = 0; jj <= nkv && ok; ++jj) {
        if (jj < nkv) {
          // S_jj = Q K_jj^T
          const uint32_t kvi = kv_iter + jj;
          const int st = kvi & 1;
          ok = warp_wait(&bars->k_full[st], (kvi >> 1) & 1, abort_flag, p.status);
          const int sb = s_iter & 1;
          if (ok && s_iter >= 2) ok = warp_wait(&bars->s_free[sb], ((s_iter >> 1) - 1) & 1, abort_flag, p.status);
          if (!ok) break;
          tc_fence_after();
          if (lane == 0) {
            const uint32_t k_addr = smem_u32(smem + L::kK0 + st * L::kTileBytes);
            const uint32_t d_tmem = tmem + (sb ? kTmemS1 : kTmemS0);
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint32_t off = (kk >> 2) * L::kAtomBytes + (kk & 3) * 32;
              mma_bf16_ss(d_tmem, make_smem_desc_sw128(q_addr + off, 16, 1024),
                          make_smem_desc_sw128(k_addr + off, 16, 1024), idesc_qk, kk > 0 ? 1u : 0u);
            }
            mma_commit(&bars->s_full[sb]);
            mma_commit(&bars->k_empty[st]);
            if (jj == nkv - 1) mma_commit(&bars->q_empty);
          }
          __syncwarp();
          ++s_iter;
        }
        if (jj >= 1) {
          // O += P_{jj-1} V_{jj-1}
          const int pj = jj - 1;
          const uint32_t kvi = kv_iter + pj;
          const int st = kvi & 1;
          ok = warp_wait(&bars->p_full, pv_iter & 1, abort_flag, p.status);
          if (ok) ok = warp_wait(&bars->v_full[st], (kvi >> 1) & 1, abort_flag, p.status);
          if (ok && pj == 0 && item_iter > 0) ok = warp_wait(&bars->o_free, (item_iter - 1) & 1, abort_flag, p.status);
          if (!ok) break;
          uint8_t* vtile = smem + L::kV0 + st * L::kTileBytes;
          const int valid_keys = n - pj * BN;  // keys of this tile inside the segment
          if (valid_keys < BN) {
            // rows past the segment end may hold anything (other segments, unwritten cache
            // rows): zero them so that 0-weight columns of P cannot meet NaN in V
            for (int a = 0; a < L::kAtoms; ++a) {
              uint4* base = reinterpret_cast<uint4*>(vtile + a * L::kAtomBytes);
              for (int i = valid_keys * 8 + lane; i < BN * 8; i += 32) base[i] = make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
          }
          __syncwarp();
          tc_fence_after();
          if (lane == 0) {
            const uint32_t v_addr = smem_u32(vtile);
#pragma unroll
            for (int kk = 0; kk < BN / 16; ++kk) {
              const uint32_t a_off = (kk >> 2) * L::kAtomBytes + (kk & 3) * 32;
              mma_bf16_ss(tmem + kTmemO, make_smem_desc_sw128(p_addr + a_off, 16, 1024),
                          make_smem_desc_sw128(v_addr + kk * 2048, L::kAtomBytes, 1024), idesc_pv,
                          (pj > 0 || kk > 0) ? 1u : 0u);
            }
            mma_commit(&bars->o_ready);
            mma_commit(&bars->v_empty[st]);
          }
          __syncwarp();
          ++pv_iter;
        }
      }
      kv_iter += nkv;
      ++item_iter;
    }
    if (!ok && lane == 0) {
      // wait (bounded) for MMAs already issued before TMEM is released
      mma_commit(&bars->drain);
      const uint64_t t0 = global_timer_ns();
      while (!mbar_try_wait(&bars->drain, 0) && global_timer_ns() - t0 < 100000000ull) {
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ softmax / epilogue
    const int quad = warp & 3;              // TMEM lane quadrant of this warp
    const int row = quad * 32 + lane;       // query row within the tile
    const uint32_t lane_addr = (uint32_t)(quad * 32) << 16;
    uint8_t* p_tile = smem + L::kP;
    uint32_t s_iter = 0, o_iter = 0, item_iter = 0;
    bool ok = true;
    while (ok) {
      int2 item;
      ok = take_item(bars, item_iter, &item, abort_flag, p.status);
      if (!ok || item.x < 0) break;
      ++item_iter;
      const int seg = item.x / p.g, j = item.x % p.g, qt = item.y;
      const int off = p.seg_offsets[seg];
      const int n = p.seg_offsets[seg + 1] - off;
      const int nkv = qt + 1;
      const int qrank = qt * BM + row;
      float m_use = 0.f, l_sum = 0.f;
      for (int jj = 0; jj < nkv && ok; ++jj) {
        const int sb = s_iter & 1;
        ok = warp_wait(&bars->s_full[sb], (s_iter >> 1) & 1, abort_flag, p.status);
        if (!ok) break;
        tc_fence_after();
        float s[BN];
#pragma unroll
        for (int c = 0; c < BN / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(tmem + lane_addr + (sb ? kTmemS1 : kTmemS0) + c * 32, r);
#pragma unroll
          for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(r[i]);
        }
        tmem_wait_ld();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->s_free[sb]);
        ++s_iter;

        // causal mask inside the diagonal tile: key rank jj*BN + c <= query rank
        if (jj == qt) {
#pragma unroll
          for (int c = 0; c < BN; ++c)
            if (c > row) s[c] = -INFINITY;
        }
        float mx = s[0];
#pragma unroll
        for (int c = 1; c < BN; ++c) mx = fmaxf(mx, s[c]);
        const float m_tile = mx * p.scale_log2;
        float alpha = 1.f;
        bool rescale = false;
        if (jj == 0) {
          m_use = m_tile;
        } else if (m_tile > m_use + kRescaleThreshold) {
          alpha = fast_exp2(m_use - m_tile);
          m_use = m_tile;
          rescale = true;
        }
        uint32_t pk[BN / 2];
        float rowsum = 0.f;
#pragma unroll
        for (int c = 0; c < BN; c += 2) {
          const float e0 = fast_exp2(fmaf(s[c], p.scale_log2, -m_use));
          const float e1 = fast_exp2(fmaf(s[c + 1], p.scale_log2, -m_use));
          rowsum += e0 + e1;
          pk[c / 2] = pack_bf16x2(e0, e1);
        }
        l_sum = l_sum * alpha + rowsum;

        // P buffer and O are free once PV of the previous tile completed
        if (jj > 0) {
          ok = warp_wait(&bars->o_ready, o_iter & 1, abort_flag, p.status);
          ++o_iter;
          if (!ok) break;
          tc_fence_after();
          if (__any_sync(0xffffffffu, rescale)) {
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
              uint32_t r[32];
              tmem_ld32(tmem + lane_addr + kTmemO + c * 32, r);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
              tmem_st32(tmem + lane_addr + kTmemO + c * 32, r);
            }
            tmem_wait_st();
          }
        }
        // P row -> shared memory, K-major 128B-swizzled (16-byte chunk index ^= row % 8)
#pragma unroll
        for (int ch = 0; ch < BN / 8; ++ch) {
          const int atom = ch >> 3, cc = ch & 7;
          uint4* dst = reinterpret_cast<uint4*>(p_tile + atom * L::kAtomBytes + row * 128 + ((cc ^ (row & 7)) << 4));
          *dst = make_uint4(pk[ch * 4 + 0], pk[ch * 4 + 1], pk[ch * 4 + 2], pk[ch * 4 + 3]);
        }
        fence_proxy_async_smem();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->p_full);
      }
      if (!ok) break;
      // epilogue: O / l * gate -> y[row_src]
      ok = warp_wait(&bars->o_ready, o_iter & 1, abort_flag, p.status);
      ++o_iter;
      if (!ok) break;
      tc_fence_after();
      const bool valid = qrank < n;
      const long long prow = (long long)off + qrank;
      long long dst_row = 0;
      float scale = 0.f;
      if (valid) {
        const int src = p.row_src[prow];
        dst_row = (long long)src * p.g + j;
        scale = p.gate[src] / l_sum;
      }
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tmem + lane_addr + kTmemO + c * 32, r);
        tmem_wait_ld();
        if (valid) {
          uint4* dst = reinterpret_cast<uint4*>(p.y + dst_row * D + c * 32);
#pragma unroll
          for (int q4 = 0; q4 < 4; ++q4) {
            uint32_t w[4];
#pragma unroll
            for (int e = 0; e < 4; ++e)
              w[e] = pack_bf16x2(__uint_as_float(r[q4 * 8 + 2 * e]) * scale,
                                 __uint_as_float(r[q4 * 8 + 2 * e + 1]) * scale);
            dst[q4] = make_uint4(w[0], w[1], w[2], w[3]);
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->o_free);
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, kTmemCols);
  if (threadIdx.x == 0) {
    // every fetch of this CTA happened before the barrier above; the last CTA resets
    __threadfence();
    if (atomicAdd(p.sched + 1, 1) == G - 1) {
      p.sched[0] = 0;
      p.sched[1] = 0;
      __threadfence();
    }
  }
}

// One block.  Items ordered by decreasing cost (qt descending), then (segment, j).
// Segments longer than their cache capacity are skipped (the RoPE stage reports them).
// Also zeroes the dynamic scheduler's counters.
__global__ void __launch_bounds__(1024) plan_kernel(const int32_t* __restrict__ seg_offsets, int nseg,
                                                    const int32_t* __restrict__ seg_cap, int g, int max_qtiles,
                                                    int* __restrict__ header, int2* __restrict__ items) {
  extern __shared__ int s_dyn[];
  int* s_count = s_dyn;               // [max_qtiles]: segments with more than q tiles
  int* s_start = s_dyn + max_qtiles;  // [max_qtiles]: first item of cost q + 1
  const int tid = threadIdx.x;
  for (int q = tid; q < max_qtiles; q += blockDim.x) s_count[q] = 0;
  __syncthreads();
  for (int s = tid; s < nseg; s += blockDim.x) {
    const int n = seg_offsets[s + 1] - seg_offsets[s];
    if (seg_cap && n > seg_cap[s]) continue;
    const int nt = min((n + BM - 1) / BM, max_qtiles);
    if (nt > 0) atomicAdd(&s_count[nt - 1], 1);  // histogram of tile counts
  }
  __syncthreads();
  if (tid == 0) {
    int above = 0, run = 0;  // above: segments with more than q tiles
    for (int q = max_qtiles - 1; q >= 0; --q) {
      above += s_count[q];
      s_count[q] = above;
      s_start[q] = run;
      run += above * g;
    }
    header[0] = 0;  // next item
    header[1] = 0;  // CTAs finished
    header[2] = run;
  }
  __syncthreads();
  for (int q = tid; q < max_qtiles; q += blockDim.x) {
    if (s_count[q] == 0) continue;
    int pos = s_start[q];
    for (int s = 0; s < nseg; ++s) {
      const int n = seg_offsets[s + 1] - seg_offsets[s];
      if (seg_cap && n > seg_cap[s]) continue;
      if (n > q * BM)
        for (int j = 0; j < g; ++j) items[pos++] = make_int2(s * g + j, q);
    }
  }
}

bool encode_rows_map(CUtensorMap* map, const void* base, long long rows, int row_elems) {
  EncodeTiledFn enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)row_elems, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)row_elems * 2};
  cuuint32_t box[2] = {64u, (cuuint32_t)BM};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                   CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

template <int D>
cudaError_t launch_attn(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p,
                        int grid, cudaStream_t stream) {
  const int smem = Smem<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  attn_fwd_kernel<D><<<grid, kThreads, smem, stream>>>(tq, tk, tv, p);
  return cudaGetLastError();
}

}  // namespace attn

namespace {
__global__ void seg_len_kernel(const int32_t* __restrict__ seg_offsets, int nseg, int32_t* __restrict__ seg_len) {
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s < nseg) seg_len[s] = seg_offsets[s + 1] - seg_offsets[s];
}

constexpr int kMaxPrefillT = 1 << 20;  // the plan keeps 2 ints per query tile in shared memory

bool supported_dims(int d_head, int g) {
  return (d_head == 64 || d_head == 128) && (g == 1 || g == 2 || g == 4 || g == 8);
}

// Shape checks shared by the prefill stages.  Fills Hr, Kr, R on success.
int check_shape(int B, int T, int H, int K, int d_head, int group, int* Hr, int* Kr, long long* R) {
  if (B < 1 || T < 1 || group < 1 || H < 1 || K < 1 || K > H || H % group || K % group) return NAMOH_ERR_INVALID_ARG;
  if (H / group > NAMOH_MAX_HEADS) return NAMOH_ERR_INVALID_ARG;
  if (d_head >= 0 && !supported_dims(d_head, group)) return NAMOH_ERR_UNSUPPORTED;
  if (T > kMaxPrefillT) return NAMOH_ERR_UNSUPPORTED;
  *Hr = H / group;
  *Kr = K / group;
  *R = (long long)B * T * *Kr;
  if (*R * group >= (1ll << 31) || (long long)B * *Hr >= (1ll << 24)) return NAMOH_ERR_INVALID_ARG;
  return NAMOH_OK;
}

size_t plan_bytes_for(int B, int T, int Hr, int Kr, int g) {
  const long long R = (long long)B * T * Kr;
  const long long max_items = ((R + attn::BM - 1) / attn::BM + (long long)B * Hr) * g;
  return 16 + (size_t)max_items * sizeof(int2);
}

int launch_plan(const int32_t* seg_offsets, int nseg, int T, int g, const int32_t* seg_cap, void* plan,
                cudaStream_t stream) {
  const int max_qtiles = (T + attn::BM - 1) / attn::BM;
  const int smem = 2 * max_qtiles * (int)sizeof(int);
  if (smem > 48 * 1024 &&
      cudaFuncSetAttribute(attn::plan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
    return NAMOH_ERR_CUDA;
  int* header = static_cast<int*>(plan);
  int2* items = reinterpret_cast<int2*>(static_cast<char*>(plan) + 16);
  attn::plan_kernel<<<1, 1024, smem, stream>>>(seg_offsets, nseg, seg_cap, g, max_qtiles, header, items);
  return cudaGetLastError() == cudaSuccess ? NAMOH_OK : NAMOH_ERR_CUDA;
}

int launch_attention(const uint16_t* q_rot, const uint16_t* k_cache, const uint16_t* v_cache, int B, int T, int Hr,
                     int Kr, int D, int g, const int32_t* seg_offsets, const int32_t* row_src, const float* gate,
                     const int64_t* seg_base, long long cache_rows, void* plan, uint16_t* y, uint32_t* dev_status,
                     const DeviceInfo& info, cudaStream_t stream) {
  const long long R = (long long)B * T * Kr;
  CUtensorMap tq, tk, tv;
  if (!attn::encode_rows_map(&tq, q_rot, R, g * D) || !attn::encode_rows_map(&tk, k_cache, cache_rows, D) ||
      !attn::encode_rows_map(&tv, v_cache, cache_rows, D))
    return NAMOH_ERR_CUDA;
  attn::Params p;
  p.seg_offsets = seg_offsets;
  p.seg_base = seg_base;
  p.row_src = row_src;
  p.gate = gate;
  p.sched = static_cast<int*>(plan);
  p.nitems = static_cast<int*>(plan) + 2;
  p.items = reinterpret_cast<const int2*>(static_cast<char*>(plan) + 16);
  p.y = y;
  p.g = g;
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  p.status = dev_status;
  const cudaError_t e = (D == 128) ? attn::launch_attn<128>(tq, tk, tv, p, info.sm_count, stream)
                                   : attn::launch_attn<64>(tq, tk, tv, p, info.sm_count, stream);
  return e == cudaSuccess ? NAMOH_OK : NAMOH_ERR_CUDA;
}

bool device_ok(DeviceInfo* info) {
  return current_device_info(info) && info->major == 10 &&
         (size_t)attn::Smem<128>::kAlloc <= info->max_smem_optin;
}
}  // namespace

}  // namespace namoh

using namespace namoh;

extern "C" int namoh_rope_pack(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H, int K,
                               int d_head, int group, float rope_base, const int32_t* seg_offsets, uint16_t* q_rot,
                               uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap,
                               int64_t cache_rows, uint32_t* dev_status, void* stream_v) {
  if (!q || !k || !v || !seg_offsets || !q_rot || !k_cache || !v_cache || !dev_status) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (!(rope_base > 1.0f) || !isfinite(rope_base)) return NAMOH_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(q_rot) || !aligned16(k_cache) ||
      !aligned16(v_cache))
    return NAMOH_ERR_INVALID_ARG;
  if (k_cache == k) return NAMOH_ERR_INVALID_ARG;
  if (seg_base) {
    if (!seg_cap || cache_rows < 1 || cache_rows >= (1ll << 31) || v_cache == v) return NAMOH_ERR_INVALID_ARG;
  } else {
    cache_rows = R;
  }
  DeviceInfo info;
  if (!current_device_info(&info)) return NAMOH_ERR_CUDA;
  RopeTable tab;
  fill_rope_table(&tab, d_head, (double)rope_base);
  const cudaError_t e = launch_rope_pack(d_head, q, k, v, (int)R, group, seg_offsets, B * Hr, seg_base, seg_cap,
                                         cache_rows, q_rot, k_cache, v_cache, v_cache != v, tab, dev_status,
                                         info.sm_count, reinterpret_cast<cudaStream_t>(stream_v));
  return e == cudaSuccess ? NAMOH_OK : NAMOH_ERR_CUDA;
}

extern "C" size_t namoh_attention_plan_size(int B, int T, int H, int K, int group) {
  int Hr, Kr;
  long long R;
  if (check_shape(B, T, H, K, -1, group, &Hr, &Kr, &R) != NAMOH_OK) return 0;
  return align_up(plan_bytes_for(B, T, Hr, Kr, group), 256);
}

extern "C" int namoh_attention_plan(const int32_t* seg_offsets, int B, int T, int H, int K, int group,
                                    const int32_t* seg_cap, void* plan, size_t plan_bytes, void* stream_v) {
  if (!seg_offsets) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, -1, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (!plan || (reinterpret_cast<uintptr_t>(plan) & 15u) || plan_bytes < plan_bytes_for(B, T, Hr, Kr, group))
    return NAMOH_ERR_WORKSPACE;
  return launch_plan(seg_offsets, B * Hr, T, group, seg_cap, plan, reinterpret_cast<cudaStream_t>(stream_v));
}

extern "C" int namoh_attention(const uint16_t* q_rot, const uint16_t* k_cache, const uint16_t* v_cache, int B, int T,
                               int H, int K, int d_head, int group, const int32_t* seg_offsets,
                               const int32_t* row_src, const float* gate, const int64_t* seg_base, int64_t cache_rows,
                               void* plan, size_t plan_bytes, uint16_t* y, uint32_t* dev_status, void* stream_v) {
  if (!q_rot || !k_cache || !v_cache || !seg_offsets || !row_src || !gate || !y || !dev_status)
    return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (!aligned16(q_rot) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(y)) return NAMOH_ERR_INVALID_ARG;
  if (seg_base) {
    if (cache_rows < 1 || cache_rows >= (1ll << 31)) return NAMOH_ERR_INVALID_ARG;
  } else {
    cache_rows = R;
  }
  if (!plan || (reinterpret_cast<uintptr_t>(plan) & 15u) || plan_bytes < plan_bytes_for(B, T, Hr, Kr, group))
    return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!device_ok(&info)) return NAMOH_ERR_UNSUPPORTED;
  return launch_attention(q_rot, k_cache, v_cache, B, T, Hr, Kr, d_head, group, seg_offsets, row_src, gate, seg_base,
                          cache_rows, plan, y, dev_status, info, reinterpret_cast<cudaStream_t>(stream_v));
}

extern "C" size_t namoh_prefill_workspace_size(int B, int T, int H, int K, int d_head, int group) {
  int Hr, Kr;
  long long R;
  if (check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R) != NAMOH_OK) return 0;
  WorkspaceCarver ws{nullptr, 0, 0};
  ws.take<uint16_t>((size_t)R * group * d_head);
  ws.take<char>(plan_bytes_for(B, T, Hr, Kr, group));
  return align_up(ws.used, 256);
}

extern "C" int namoh_prefill(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H, int K,
                             int d_head, int group, float rope_base, const int32_t* seg_offsets,
                             const int32_t* row_src, const float* gate, uint16_t* y, uint16_t* k_cache,
                             uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap, int64_t cache_rows,
                             int32_t* seg_len, void* workspace, size_t workspace_bytes, uint32_t* dev_status,
                             void* stream_v) {
  if (!q || !k || !v || !seg_offsets || !row_src || !gate || !y || !k_cache || !v_cache || !dev_status)
    return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (!(rope_base > 1.0f) || !isfinite(rope_base)) return NAMOH_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(y) || !aligned16(k_cache) || !aligned16(v_cache))
    return NAMOH_ERR_INVALID_ARG;
  if (k_cache == k) return NAMOH_ERR_INVALID_ARG;
  if (seg_base) {
    if (!seg_cap || cache_rows < 1 || cache_rows >= (1ll << 31) || v_cache == v) return NAMOH_ERR_INVALID_ARG;
  } else {
    cache_rows = R;
  }
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
  uint16_t* q_rot = ws.take<uint16_t>((size_t)R * group * d_head);
  const size_t pbytes = plan_bytes_for(B, T, Hr, Kr, group);
  void* plan = ws.take<char>(pbytes);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!device_ok(&info)) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);

  RopeTable tab;
  fill_rope_table(&tab, d_head, (double)rope_base);
  if (launch_rope_pack(d_head, q, k, v, (int)R, group, seg_offsets, B * Hr, seg_base, seg_cap, cache_rows, q_rot,
                       k_cache, v_cache, v_cache != v, tab, dev_status, info.sm_count, stream) != cudaSuccess)
    return NAMOH_ERR_CUDA;
  st = launch_plan(seg_offsets, B * Hr, T, group, seg_base ? seg_cap : nullptr, plan, stream);
  if (st != NAMOH_OK) return st;
  if (seg_len) {
    seg_len_kernel<<<(B * Hr + 255) / 256, 256, 0, stream>>>(seg_offsets, B * Hr, seg_len);
    if (cudaGetLastError() != cudaSuccess) return NAMOH_ERR_CUDA;
  }
  return launch_attention(q_rot, k_cache, v_cache, B, T, Hr, Kr, d_head, group, seg_offsets, row_src, gate, seg_base,
                          cache_rows, plan, y, dev_status, info, stream);
}
