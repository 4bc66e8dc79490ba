// prefill_attn.cu -- routed causal attention over packed (batch, head) segments with the
// gate-weighted combine fused into the epilogue (Sec. 3.1, Eq. namoh-attention; Sec. 3.2
// "Efficient execution": packed variable-length subsequences and length-aware scheduling;
// App. B.7 "Adopted KV-group routing" for g > 1).
//
// Work unit ("item"): one 128-row query tile t of one segment for one group head j.  Within
// a segment, queries and keys share local ranks, so tile t needs key tiles 0..t and only
// tile t is masked (key rank <= query rank).
//
// Schedule (length-aware, longest first): a one-block "plan" kernel lists the items in
// order of decreasing cost (t + 1 key tiles).  The persistent attention kernel launches
// one CTA per SM; each CTA's producer warp takes the next item from an atomic counter
// (greedy list scheduling in longest-first order) and hands it to the other warps through
// a two-slot ring in shared memory.  The last CTA to finish resets the counter, so a plan
// can be reused by later launches on the same stream.
//
// Attention CTA (192 threads, one CTA per SM):
//   warps 0-3   softmax / epilogue: thread i owns query row i (TMEM lane i).  Online
//               softmax in fp32 with exp2; the running max only moves when it grows by
//               more than 2^8 (O in TMEM is then rescaled).  P is written back to TMEM as
//               bf16 over the S columns it came from.  The epilogue reads O out of TMEM
//               (freeing it for the next item at once), divides by the row sum, multiplies
//               by the routing gate and writes bf16 rows to y[row_src], a 32-byte sector per
//               store.
//   warp 4      TMA producer: the Q tile, then K(0), K(1), V(0), K(2), V(1), ... through a
//               6-slot ring (128B swizzle) two key tiles ahead of the MMAs.
//   warp 5      MMA issuer (one lane) and TMEM owner.  tcgen05.mma instructions into one
//               accumulator run back to back while instructions into different
//               accumulators overlap, so with three S/P buffers the issuer interleaves
//               PV(kv) (A = P in TMEM, B = V as the MN-major operand) with S(kv+2) = Q K^T
//               instruction by instruction while the softmax works on S(kv+1).
// TMEM: S/P buffers at cols [0,128), [128,256), [256,384); O at [384, 384 + D).
// Shared memory (d = 128): Q 32 KB + 6 x 32 KB ring = 224 KB.
// Every mbarrier wait is bounded (NAMOH_DEV_TIMEOUT, then all roles drain and exit).
#include <cstddef>

#include "common.cuh"
#include "plan.cuh"

namespace namoh {

cudaError_t launch_rope_pack(int D, const uint16_t* q, const uint16_t* k, const uint16_t* v, int R, int g,
                             const int32_t* seg_offsets, int nseg, const int64_t* seg_base, const int32_t* seg_cap,
                             long long cache_rows, uint16_t* q_rot, uint16_t* k_cache, uint16_t* v_cache, bool copy_v,
                             const RopeTable& tab, uint32_t* status, int sm_count, cudaStream_t stream,
                             void* plan, int plan_qtiles, const int32_t* plan_cap, const int32_t* pos_row_src,
                             int pos_k, int pos_t, const int32_t* pos_cu, int pos_hr, bool interleaved,
                             const RopePool* pool);
int rope_chunk_rows(int D, int g);

int launch_window_attention(const uint16_t* q_rot, const uint16_t* k_cache, const uint16_t* v_cache, int B, int T,
                            int Hs, int D, int window, const int64_t* seg_base, long long cache_rows, uint16_t* y,
                            uint32_t* dev_status, int sm_count, cudaStream_t stream);
constexpr int kMaxBandWindow = 128;  // windows up to one key tile run as one 256-key band per query tile

int launch_sa_select(const CUtensorMap& q_rot_map, const uint16_t* q_rot, const uint16_t* k_cache,
                     const int32_t* seg_offsets, const int64_t* seg_base, const int32_t* seg_cap,
                     long long cache_rows, int nseg, int T, long long R, int d, int g, int lg, int alpha_num,
                     int alpha_den, uint16_t* kbar, long long kbar_rows, uint32_t* mask, int words, const void* plan,
                     int max_items, uint32_t* status, cudaStream_t stream, bool pooled);

namespace attn {

constexpr int BM = 128;              // query rows per tile (one tile per work item)
constexpr int BN = 128;              // keys per tile
constexpr int kItemRows = BM;
static_assert(kItemRows == kPlanTileRows, "the plan and the kernel must agree on the query tile");
constexpr int kSoftmaxWarps = 4;     // warps 0-3: thread i owns query row i (TMEM lane i)
constexpr int kWarpLoad = 4;
constexpr int kWarpMma = 5;
constexpr int kThreads = 192;
constexpr int kTmemCols = 512;
constexpr int kSBufs = 3;            // S/P buffers in TMEM
// TMEM columns: S/P buffers at 0, 128, 256; O at 384.  P (bf16, two per 32-bit column)
// overwrites the first BN/2 columns of the S buffer it was computed from.
__host__ __device__ constexpr uint32_t tmem_s_col(int b) { return 128u * (uint32_t)b; }
constexpr uint32_t kTmemO = 384;
constexpr float kRescaleThreshold = 8.0f;  // log2 units
constexpr int kRing = 6;                   // K/V ring: K(0), K(1), V(0), K(2), V(1), K(3), ...

template <int D>
struct Smem {
  static constexpr int kAtoms = D / 64;          // 64-column (128-byte) swizzle atoms per row
  static constexpr int kTileBytes = BM * D * 2;  // one Q / K / V tile
  static constexpr int kAtomBytes = BM * 128;    // 16 KB: 128 rows x 128 bytes
  static constexpr int kQ = 0;
  static constexpr int kRing0 = kTileBytes;
  static constexpr int kBar = kRing0 + kRing * kTileBytes;
  static constexpr int kBytes = kBar + 512;
  static constexpr int kAlloc = kBytes + 1024;   // slack for 1024-byte alignment
};

struct Bars {
  uint64_t item_full[2], item_empty[2];
  uint64_t q_full, q_empty;
  uint64_t ring_full[kRing], ring_empty[kRing];
  uint64_t s_full[kSBufs];  // S written into buffer b (one barrier per buffer: at an item
                            // boundary two S are issued back to back, and a parity wait
                            // must never fall two phases behind)
  uint64_t p_full[2];   // P of key tile i in TMEM (and O rescaled if needed): p_full[i & 1],
                        // phase i >> 1.  The softmax may run two tiles ahead of the MMA warp
                        // (S(i) is issued only after P(i-2) was taken), never more.
  uint64_t o_ready[2];  // PV number i (counted over the CTA's life) completed: o_ready[i & 1],
                        // phase i >> 1.  Two barriers, so that consumers may skip PVs they
                        // do not need and still wait on an exact phase.
  uint64_t o_free;      // epilogue finished reading O
  uint64_t drain;
  int4 item_slot[2];    // {segment * g + j, query tile, seg_offsets[segment], n}
  uint32_t tmem_base;
  int abort_flag;
};

static_assert(sizeof(Bars) <= 512, "barrier block");
static_assert(offsetof(Bars, q_full) == 32, "the timeout probe's documented barrier index (word 4)");

struct Params {
  const int32_t* seg_offsets;  // [nseg + 1]
  const int64_t* seg_base;     // [nseg] or null (cache rows = packed rows)
  const int32_t* row_src;      // [R]
  const float* gate;           // [R] indexed by row_src value
  const int4* items;           // {segment * g + j, query tile, seg_offsets[segment], n}, longest first
  const int* nitems;
  int* sched;                  // [0] next item, [1] CTAs finished
  uint16_t* y;                 // [R * g, D] indexed by row_src * g + j
  int rows;                    // R: a row_src value at or above it is skipped (inconsistent layout)
  int window;                  // 0: causal over the whole segment; w > 0: the last w keys only
  int g;
  int y_sector_aligned;        // y is 32-byte aligned: rows go out as whole 32-byte sectors
  float scale_log2;            // log2(e) / sqrt(D)
  uint32_t* status;
  // SA + NAMOH: kept historical blocks of each query [(row * g + j), sa_words] (bit b % 32 of
  // word b / 32), blocks of 2^sa_lg keys (32, 64 or 128); used by the kSA instantiation only
  const uint32_t* sa_mask;
  int sa_words;
  int sa_lg;
  // Test hook of the bounded waits: the MMA issuer's wait limit (kWaitLimitNs normally) and, when
  // withhold_q is set, the producer never loads a CTA's first query tile, so that the issuer's
  // wait for it runs out, reports NAMOH_DEV_TIMEOUT and every role drains and exits.
  uint64_t mma_wait_ns;
  int withhold_q;
};

// All lanes of a warp wait and agree on the outcome, so warp-collective tcgen05
// instructions after the wait never diverge on a timeout race.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, uint32_t* status,
                                          uint64_t limit_ns = kWaitLimitNs) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status, limit_ns);
  return __all_sync(0xffffffffu, ok);
}

// First key tile of query tile qt: 0, or under a sliding window of w keys the tile holding key
// qt*BM - w + 1 (the earliest key the tile's first query sees).  Every role uses this.
__device__ __forceinline__ int first_key_tile(int qt, int window) {
  return window > 0 ? max(0, (qt * BM - window + 1) / BN) : 0;
}

// Consumer side of the item ring: every lane waits, reads the item, one lane releases the slot.
__device__ __forceinline__ bool take_item(Bars* bars, uint32_t idx, int4* item, volatile int* abort_flag,
                                          uint32_t* status) {
  const int slot = idx & 1;
  if (!warp_wait(&bars->item_full[slot], (idx >> 1) & 1, abort_flag, status)) return false;
  const volatile int* src = reinterpret_cast<const volatile int*>(&bars->item_slot[slot]);
  item->x = src[0];
  item->y = src[1];
  item->z = src[2];
  item->w = src[3];
  __syncwarp();
  if ((threadIdx.x & 31) == 0) mbar_arrive(&bars->item_empty[slot]);
  return true;
}

// Online softmax of one S tile for this thread's query row (Sec. 3.1, causal scaled
// dot-product attention): S from TMEM, the causal mask on the diagonal tile, the running max
// (moved only when it grows by more than kRescaleThreshold) and row sum, P = exp2(S * scale - m)
// as bf16 over the first half of the S columns, and O rescaled when the max moved (after
// PV(tile - 1) completed, through wait_pv).  Returns false when a wait gave up.  Ends with the
// TMEM stores complete and fenced for the arrive on p_full.
// kv_rel is the tile's index within the item (0 = first), kv its index in the segment.
// kSA: allow4 bit w clear masks the tile's columns 32w..32w+31 (a block the query does not keep;
// blocks are at least 32 keys, so each 32-column group lies in one block).
template <int D, bool kSA, typename WaitPv>
__device__ __forceinline__ bool softmax_tile(uint32_t s_addr, uint32_t o_addr, int kv_rel, int kv, int qt, int row,
                                             int window, float scale_log2, float& m_use, float& l_sum,
                                             uint32_t tile, WaitPv&& wait_pv, uint32_t allow4 = 0xFu) {
  float sv[BN];
#pragma unroll
  for (int c = 0; c < BN / 32; ++c) {
    uint32_t r[32];
    tmem_ld32(s_addr + c * 32, r);
#pragma unroll
    for (int i = 0; i < 32; ++i) sv[c * 32 + i] = __uint_as_float(r[i]);
  }
  tmem_wait_ld();
  // sliding window: keys older than query rank - window + 1 are out
  if (window > 0) {
    const int lo = qt * BM + row - window + 1 - kv * BN;  // first column in the window
#pragma unroll
    for (int c = 0; c < BN; ++c)
      if (c < lo) sv[c] = -INFINITY;
  }
  // SA + NAMOH: keys of blocks the query does not keep are out
  if (kSA && allow4 != 0xFu) {
#pragma unroll
    for (int c = 0; c < BN; ++c)
      if (!((allow4 >> (c >> 5)) & 1u)) sv[c] = -INFINITY;
  }
  // causal mask on the diagonal tile: key rank kv*BN + c <= query rank
  if (kv == qt) {
#pragma unroll
    for (int c = 0; c < BN; ++c)
      if (c > row) sv[c] = -INFINITY;
  }
  // row max: three-input max instructions over eight independent accumulators
  float m8[8];
  static_assert(BN == 128, "the max tree below covers 128 columns");
#pragma unroll
  for (int i = 0; i < 8; ++i) m8[i] = fmax3(sv[i], sv[8 + i], sv[16 + i]);
#pragma unroll
  for (int c = 24; c < 120; c += 16) {
#pragma unroll
    for (int i = 0; i < 8; ++i) m8[i] = fmax3(m8[i], sv[c + i], sv[c + 8 + i]);
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) m8[i] = fmaxf(m8[i], sv[120 + i]);
  const float mx = fmax3(fmax3(m8[0], m8[1], m8[2]), fmax3(m8[3], m8[4], m8[5]), fmaxf(m8[6], m8[7]));
  // a row with every key of the tile outside the window (or in blocks it does not keep) gets a
  // finite floor, so that its P is exactly 0 and the next tile's rescale factor
  // exp2(m_use - m_tile) is 0
  const float m_tile = (kSA || window > 0) ? fmaxf(mx * scale_log2, -1e30f) : mx * scale_log2;
  float alpha = 1.f;
  bool rescale = false;
  if (kv_rel == 0) {
    m_use = m_tile;
  } else if (m_tile > m_use + kRescaleThreshold) {
    if ((kSA || window > 0) && m_use <= -1e30f) {
      // every earlier key of this row was masked: O and the row sum are exactly 0, so the
      // first tile with a visible key just sets the max (no rescale, no wait for the PV)
      alpha = 0.f;
    } else {
      alpha = fast_exp2(m_use - m_tile);
      rescale = true;
    }
    m_use = m_tile;
  }
  // P = exp2(S * scale - m_use): scale-and-subtract and the row sum on fp32 pairs
  uint32_t pk[BN / 2];
  uint64_t sum2[4] = {0ull, 0ull, 0ull, 0ull};
  const uint64_t sc2 = f2_pack(scale_log2, scale_log2), nm2 = f2_pack(-m_use, -m_use);
#pragma unroll
  for (int c = 0; c < BN; c += 2) {
    float x0, x1;
    f2_unpack(f2_fma(f2_pack(sv[c], sv[c + 1]), sc2, nm2), x0, x1);
    const float e0 = fast_exp2(x0), e1 = fast_exp2(x1);
    sum2[(c >> 1) & 3] = f2_add(sum2[(c >> 1) & 3], f2_pack(e0, e1));
    pk[c / 2] = pack_bf16x2(e0, e1);
  }
  float sa, sb;
  f2_unpack(f2_add(f2_add(sum2[0], sum2[1]), f2_add(sum2[2], sum2[3])), sa, sb);
  l_sum = l_sum * alpha + (sa + sb);
  // P over the S columns just read (every S value is in registers)
  {
    uint32_t r[32];
#pragma unroll
    for (int i = 0; i < 32; ++i) r[i] = pk[i];
    tmem_st32(s_addr, r);
#pragma unroll
    for (int i = 0; i < 32; ++i) r[i] = pk[32 + i];
    tmem_st32(s_addr + 32, r);
  }
  // O may only be rescaled once the previous PV completed; without a rescale this
  // tile's softmax does not touch O and overlaps that PV
  if (kv_rel > 0 && __any_sync(0xffffffffu, rescale)) {
    if (!wait_pv(tile - 1)) return false;
    tc_fence_after();
    {
#pragma unroll
      for (int c = 0; c < D / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(o_addr + c * 32, r);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * alpha);
        tmem_st32(o_addr + c * 32, r);
      }
    }
  }
  tmem_wait_st();
  tc_fence_before();
  return true;
}

template <int D, bool kSA>
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

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->item_full[i], 1);
      mbar_init(&bars->item_empty[i], 1 + kSoftmaxWarps);
    }
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&bars->ring_full[i], 1);
      mbar_init(&bars->ring_empty[i], 1);
    }
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int i = 0; i < kSBufs; ++i) mbar_init(&bars->s_full[i], 1);
    mbar_init(&bars->p_full[0], kSoftmaxWarps);
    mbar_init(&bars->p_full[1], kSoftmaxWarps);
    mbar_init(&bars->o_ready[0], 1);
    mbar_init(&bars->o_ready[1], 1);
    mbar_init(&bars->o_free, kSoftmaxWarps);
    mbar_init(&bars->drain, 1);
    bars->abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kWarpLoad && lane == 0) {
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_k);
    tma_prefetch_desc(&tm_v);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  // set-up above touched only this CTA's own state; the plan and Q~/K~ come from the kernel
  // before it (programmatic dependent launch)
  pdl_launch_dependents();
  pdl_wait();
  const int nitems = *p.nitems;

  if (warp == kWarpLoad) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t ring_iter = 0, item_iter = 0;
      bool ok = true;
      auto load_tile = [&](const CUtensorMap* tm, int32_t row) {
        const int slot = ring_iter % kRing;
        const uint32_t use = ring_iter / kRing;
        if (use > 0 && !mbar_wait(&bars->ring_empty[slot], (use - 1) & 1, abort_flag, p.status)) return false;
        mbar_arrive_expect_tx(&bars->ring_full[slot], L::kTileBytes);
        for (int a = 0; a < L::kAtoms; ++a)
          tma_load_2d(smem + L::kRing0 + slot * L::kTileBytes + a * L::kAtomBytes, tm, a * 64, row,
                      &bars->ring_full[slot]);
        ++ring_iter;
        return true;
      };
      while (ok) {
        // the first item is this CTA's own (the plan's G longest tiles go one per CTA), later
        // ones come from the counter; the segment's offset and length travel with the item
        const int it = item_iter == 0 ? (int)blockIdx.x : G + atomicAdd(p.sched, 1);
        int4 item = make_int4(-1, -1, 0, 0);
        int kvb = 0;
        if (it < nitems) {
          item = p.items[it];
          kvb = (int)(p.seg_base ? p.seg_base[item.x / p.g] : (long long)item.z);
        }
        const int slot = item_iter & 1;
        if (item_iter >= 2) ok = mbar_wait(&bars->item_empty[slot], ((item_iter >> 1) - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        bars->item_slot[slot] = item;
        mbar_arrive(&bars->item_full[slot]);
        if (item.x < 0) break;
        const int j = item.x % p.g, qt = item.y;
        const int off = item.z;
        const int kv0 = first_key_tile(qt, p.window);
        const int nkv = qt + 1 - kv0;
        kvb += kv0 * BN;  // the item's first key tile
        if (item_iter > 0) ok = mbar_wait(&bars->q_empty, (item_iter - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        if (!(p.withhold_q && item_iter == 0)) {
          mbar_arrive_expect_tx(&bars->q_full, L::kTileBytes);
          for (int a = 0; a < L::kAtoms; ++a)
            tma_load_2d(smem + L::kQ + a * L::kAtomBytes, &tm_q, j * D + a * 64, off + qt * BM, &bars->q_full);
        }
        // K(0), K(1), then V(kv), K(kv + 2) for kv = 0, 1, ...
        ok = load_tile(&tm_k, kvb);
        if (ok && nkv > 1) ok = load_tile(&tm_k, kvb + BN);
        for (int kv = 0; kv < nkv && ok; ++kv) {
          ok = load_tile(&tm_v, kvb + kv * BN);
          if (ok && kv + 2 < nkv) ok = load_tile(&tm_k, kvb + (kv + 2) * BN);
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
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------------ MMA issuer
    // tcgen05.mma instructions into one accumulator run back to back; instructions into
    // different accumulators overlap.  With three S/P buffers, PV(kv) (A = P from TMEM)
    // and S(kv+2) (into the buffer PV(kv-1) finished with) are independent, and are
    // issued interleaved instruction by instruction while the softmax works on S(kv+1).
    // The MMA queue is shallow: issuing a burst blocks until most of it has executed, so
    // whatever runs between two bursts leaves the tensor pipe idle.  The warp therefore
    // runs converged (one elected lane issues; descriptors are warp-uniform bases plus
    // constant offsets), the next step's K/V waits sit in the middle of the current
    // burst, and only P(kv+1) is waited between bursts (a softmax that rescales O waits
    // for PV(kv), so P(kv+1) cannot be required earlier).
    constexpr uint32_t idesc_qk = make_idesc_bf16(BM, BN, false, false);
    constexpr uint32_t idesc_pv = make_idesc_bf16(BM, D, false, true);
    const uint64_t q_desc = make_smem_desc_sw128(smem_u32(smem + L::kQ), 16, 1024);
    // descriptor offsets (16-byte units) of the K-extent steps: S walks the 128-byte swizzle
    // atom 32 bytes at a time, then the next 64-column atom; PV walks 16 keys = 2048 bytes
    auto qk_off = [](int kk) -> uint64_t { return (uint64_t)(((kk >> 2) * L::kAtomBytes + (kk & 3) * 32) >> 4); };
    auto pv_off = [](int kk) -> uint64_t { return (uint64_t)((kk * 2048) >> 4); };
    uint32_t ring_iter = 0, item_iter = 0, s_iter = 0, p_iter = 0;
    bool ok = true;
    auto slot_addr = [&](uint32_t r) { return smem_u32(smem + L::kRing0 + (r % kRing) * L::kTileBytes); };
    auto ring_ready = [&](uint32_t r) {
      return warp_wait(&bars->ring_full[r % kRing], (r / kRing) & 1, abort_flag, p.status);
    };
    auto p_ready = [&](uint32_t i) {  // P of tile number i
      return warp_wait(&bars->p_full[i & 1], (i >> 1) & 1, abort_flag, p.status);
    };
    // Ring entries a and b (b may equal a): both tries in flight together, one warp vote; the
    // bounded slow path only when one of them is not there yet.
    auto ring_ready2 = [&](uint32_t a, uint32_t b) {
      const bool fa = mbar_try_wait(&bars->ring_full[a % kRing], (a / kRing) & 1);
      const bool fb = mbar_try_wait(&bars->ring_full[b % kRing], (b / kRing) & 1);
      if (__all_sync(0xffffffffu, fa && fb)) return true;
      return ring_ready(a) && ring_ready(b);
    };

    while (ok) {
      int4 item;
      ok = take_item(bars, item_iter, &item, abort_flag, p.status);
      if (!ok || item.x < 0) break;
      const int qt = item.y;
      const int kv0 = first_key_tile(qt, p.window);
      const int nkv = qt + 1 - kv0;
      const int n = item.w - kv0 * BN;  // keys from the item's first key tile to the segment's end
      // ring entries of this item, in load order: K(0), K(1) if nkv > 1, then for each kv:
      // V(kv) followed by K(kv+2) while kv + 2 < nkv
      const uint32_t rk0 = ring_iter, rk1 = ring_iter + 1;
      const int m = nkv > 2 ? nkv - 2 : 0;  // key tiles followed by a K load
      const uint32_t base = ring_iter + (nkv > 1 ? 2u : 1u);
      auto rv = [&](int kv) -> uint32_t { return kv < m ? base + 2u * kv : base + 2u * m + (kv - m); };
      auto rk = [&](int kv) -> uint32_t { return base + 2u * (kv - 2) + 1u; };  // K(kv), kv >= 2

      // prologue: S(0) and S(1) interleaved (independent buffers), then PV(0)'s operands
      ok = warp_wait(&bars->q_full, item_iter & 1, abort_flag, p.status, p.mma_wait_ns) && ring_ready(rk0) &&
           (nkv == 1 || ring_ready(rk1));
      if (!ok) break;
      tc_fence_after();
      {
        const uint32_t s0 = tmem + tmem_s_col((int)(s_iter % kSBufs));
        const uint32_t s1 = tmem + tmem_s_col((int)((s_iter + 1) % kSBufs));
        const uint64_t k0 = make_smem_desc_sw128(slot_addr(rk0), 16, 1024);
        const uint64_t k1 = make_smem_desc_sw128(slot_addr(rk1), 16, 1024);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          mma_bf16_ss(s0, q_desc + qk_off(kk), k0 + qk_off(kk), idesc_qk, kk > 0 ? 1u : 0u);
          if (nkv > 1) mma_bf16_ss(s1, q_desc + qk_off(kk), k1 + qk_off(kk), idesc_qk, kk > 0 ? 1u : 0u);
        }
        mma_commit(&bars->s_full[s_iter % kSBufs]);
        mma_commit(&bars->ring_empty[rk0 % kRing]);
        if (nkv > 1) {
          mma_commit(&bars->s_full[(s_iter + 1) % kSBufs]);
          mma_commit(&bars->ring_empty[rk1 % kRing]);
        }
        if (nkv <= 2) mma_commit(&bars->q_empty);  // every S of this item issued
      }
      s_iter += nkv > 1 ? 2u : 1u;
      // rows past the segment end may hold anything (other segments, unwritten cache rows):
      // zero them in the last V tile so that 0-weight columns of P cannot meet NaN in V
      auto zero_v_tail = [&](uint32_t r, int valid_keys) {
        uint8_t* vtile = smem + L::kRing0 + (r % kRing) * L::kTileBytes;
        for (int a = 0; a < L::kAtoms; ++a) {
          uint4* vb = reinterpret_cast<uint4*>(vtile + a * L::kAtomBytes);
          for (int i = valid_keys * 8 + lane; i < BN * 8; i += 32) vb[i] = make_uint4(0, 0, 0, 0);
        }
        fence_proxy_async_smem();
        __syncwarp();
      };
      // step kv's ring entries: V(kv) and, while kv + 2 < nkv, K(kv+2)
      uint32_t r_v = rv(0);
      uint32_t r_k2 = nkv > 2 ? rk(2) : r_v;
      ok = ring_ready2(r_v, r_k2) &&
           (item_iter == 0 || warp_wait(&bars->o_free, (item_iter - 1) & 1, abort_flag, p.status)) && p_ready(p_iter);
      if (!ok) break;
      if (n < BN) zero_v_tail(r_v, n);  // the item's first key tile is the segment's last, partial one

      // Everything a step needs besides its commits and P(kv+1) -- the next step's ring
      // entries, their waits, a partial last V tile -- is done in the middle of the burst,
      // where the issuing thread would otherwise wait for the MMA queue.
      for (int kv = 0; kv < nkv; ++kv) {
        // here V(kv), K(kv+2), a free O and P(kv) are all in place
        const bool with_s = kv + 2 < nkv;
        const bool has_next = kv + 1 < nkv;
        const uint32_t pv_index = p_iter++;
        tc_fence_after();
        // P(kv) sits in the buffer of S(kv): S and P are counted alike across items
        const uint32_t pbuf = tmem + tmem_s_col((int)(pv_index % kSBufs));
        const uint32_t sbuf = tmem + tmem_s_col((int)(s_iter % kSBufs));
        const uint64_t v_desc = make_smem_desc_sw128(slot_addr(r_v), L::kAtomBytes, 1024);
        const uint64_t k_desc = make_smem_desc_sw128(slot_addr(r_k2), 16, 1024);
        const uint32_t acc0 = kv > 0 ? 1u : 0u;
        const uint32_t r_vn = has_next ? rv(kv + 1) : r_v;
        const uint32_t r_kn = kv + 3 < nkv ? rk(kv + 3) : r_vn;
        auto mid_burst = [&]() {
          if (has_next) {
            ok = ring_ready2(r_vn, r_kn);
            const int next_valid = n - (kv + 1) * BN;
            if (ok && next_valid < BN) zero_v_tail(r_vn, next_valid);
          }
        };
        if (with_s) {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            // PV: K extent = BN keys, 16 per instruction; S: K extent = D, 16 per instruction
            mma_bf16_ts(tmem + kTmemO, pbuf + kk * 8, v_desc + pv_off(kk), idesc_pv, kk > 0 ? 1u : acc0);
            if (kk < D / 16) mma_bf16_ss(sbuf, q_desc + qk_off(kk), k_desc + qk_off(kk), idesc_qk, kk > 0 ? 1u : 0u);
            if (kk == 3) mid_burst();
          }
        } else {
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            mma_bf16_ts(tmem + kTmemO, pbuf + kk * 8, v_desc + pv_off(kk), idesc_pv, kk > 0 ? 1u : acc0);
            if (kk == 3) mid_burst();
          }
        }
        mma_commit(&bars->o_ready[pv_index & 1]);
        mma_commit(&bars->ring_empty[r_v % kRing]);
        if (with_s) {
          mma_commit(&bars->s_full[s_iter % kSBufs]);
          mma_commit(&bars->ring_empty[r_k2 % kRing]);
          if (kv + 2 == nkv - 1) mma_commit(&bars->q_empty);
          ++s_iter;
        }
        if (ok && has_next) ok = p_ready(p_iter);
        if (!ok) break;
        r_v = r_vn;
        r_k2 = r_kn;
      }
      ring_iter += 2 * nkv;
      ++item_iter;
    }
    if (!ok) {
      // wait (bounded) for MMAs already issued before TMEM is released
      mma_commit(&bars->drain);
      const uint64_t t0 = global_timer_ns();
      while (!mbar_try_wait(&bars->drain, 0) && global_timer_ns() - t0 < 100000000ull) {
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ softmax / epilogue
    const int row = warp * 32 + lane;  // query row within the tile (warp w reads TMEM lanes 32w..32w+31)
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    const uint32_t o_addr = tmem + lane_addr + kTmemO;
    // s_iter counts key tiles over the CTA's life; tile i's S, P and PV all carry number i.
    uint32_t s_iter = 0, item_iter = 0;
    bool ok = true;
    // Waits for PV number i.  Exact whenever PV i-2 is known complete and PV i+2 is not yet
    // issued: true inside the softmax of tile i+1 (its S was committed after PV i-1) and in
    // the epilogue of an item whose last tile is i.
    auto wait_pv = [&](uint32_t i) { return warp_wait(&bars->o_ready[i & 1], (i >> 1) & 1, abort_flag, p.status); };
    while (ok) {
      int4 item;
      ok = take_item(bars, item_iter, &item, abort_flag, p.status);
      ++item_iter;
      if (!ok || item.x < 0) break;
      const int j = item.x % p.g, qt = item.y, off = item.z, n = item.w;
      // the output row now (its latency hides behind the first tile); the gate after it
      const int qrank = qt * BM + row;
      const bool valid = qrank < n;
      int src = 0;
      if (valid) src = ld_issue_s32(p.row_src + off + qrank);
      float gt = 0.f;
      float m_use = 0.f, l_sum = 0.f;
      const int kv0 = first_key_tile(qt, p.window);
      // SA + NAMOH: this query's kept-block words, one tile ahead of their use
      const uint32_t* mrow = nullptr;
      int cur_blk = 0;
      uint32_t w_next = ~0u;
      if (kSA && valid) {
        mrow = p.sa_mask + ((long long)(off + qrank) * p.g + j) * p.sa_words;
        cur_blk = qrank >> p.sa_lg;
        w_next = ld_issue_u32(mrow + (((kv0 * BN) >> p.sa_lg) >> 5));
      }
      for (int kv = kv0; kv <= qt && ok; ++kv) {
        const uint32_t s_addr = tmem + lane_addr + tmem_s_col((int)(s_iter % kSBufs));
        uint32_t allow4 = 0xFu;
        if (kSA && mrow) {
          const uint32_t w = w_next;
          if (kv < qt) w_next = ld_issue_u32(mrow + ((((kv + 1) * BN) >> p.sa_lg) >> 5));
          allow4 = 0u;
#pragma unroll
          for (int c = 0; c < 4; ++c) {
            const int blk = (kv * BN + 32 * c) >> p.sa_lg;
            if (blk == cur_blk || ((w >> (blk & 31)) & 1u)) allow4 |= 1u << c;
          }
        }
        ok = warp_wait(&bars->s_full[s_iter % kSBufs], (s_iter / kSBufs) & 1, abort_flag, p.status);
        const uint32_t tile = s_iter++;
        if (!ok) break;
        tc_fence_after();
        ok = softmax_tile<D, kSA>(s_addr, o_addr, kv - kv0, kv, qt, row, p.window, p.scale_log2, m_use, l_sum,
                                  tile, wait_pv, allow4);
        if (!ok) break;
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->p_full[tile & 1]);
        if (kv == kv0 && valid) {  // the gate, used in the epilogue only
          if ((unsigned)src < (unsigned)p.rows) gt = ld_issue_f32(p.gate + src);
          else src = -1;
        }
      }
      if (!ok) break;
      // epilogue: O out of TMEM (O is then free for the next item), O / l * gate as bf16
      // to y[row_src * g + j], 32 bytes (one whole sector) per store where y allows it
      ok = wait_pv(s_iter - 1);
      if (!ok) break;
      tc_fence_after();
      uint32_t o[D / 32][32];
#pragma unroll
      for (int c = 0; c < D / 32; ++c) tmem_ld32(o_addr + c * 32, o[c]);
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->o_free);
      if (valid && src >= 0) {
        const float scale = gt / l_sum;
        uint32_t w[D / 2];
#pragma unroll
        for (int e = 0; e < D / 2; ++e)
          w[e] = pack_bf16x2(__uint_as_float(o[e / 16][(e % 16) * 2]) * scale,
                             __uint_as_float(o[e / 16][(e % 16) * 2 + 1]) * scale);
        uint16_t* dst = p.y + ((long long)src * p.g + j) * D;
        if (p.y_sector_aligned) {
#pragma unroll
          for (int c = 0; c < D / 16; ++c) st_global_v8(dst + c * 16, w + c * 8);
        } else {
#pragma unroll
          for (int c = 0; c < D / 8; ++c)
            *reinterpret_cast<uint4*>(dst + c * 8) = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kWarpMma) tmem_dealloc(tmem, kTmemCols);
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

// One block builds the work list (see build_plan) and zeroes the scheduler's counters.
__global__ void __launch_bounds__(1024) plan_kernel(const int32_t* __restrict__ seg_offsets, int nseg,
                                                    const int32_t* __restrict__ seg_cap, int g, int max_qtiles,
                                                    int* __restrict__ header, int4* __restrict__ items) {
  extern __shared__ int s_dyn[];
  build_plan(seg_offsets, nseg, seg_cap, g, max_qtiles, header, items, s_dyn);
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

template <int D, bool kSA>
cudaError_t launch_attn(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p,
                        int grid, cudaStream_t stream) {
  const int smem = Smem<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel<D, kSA>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(attn_fwd_kernel<D, kSA>, dim3(grid), dim3(kThreads), (size_t)smem, stream, tq, tk, tv, p);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace attn

namespace {
__global__ void seg_len_kernel(const int32_t* __restrict__ seg_offsets, int nseg, int32_t* __restrict__ seg_len) {
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s < nseg) seg_len[s] = max(seg_offsets[s + 1] - seg_offsets[s], 0);
}

constexpr int kMaxPrefillT = 1 << 20;  // the plan keeps 2 ints per query tile in shared memory
constexpr int kMaxPrefillSegments = 1 << 15;  // and one int per segment

bool supported_dims(int d_head, int g) {
  return (d_head == 64 || d_head == 128) && (g == 1 || g == 2 || g == 4 || g == 8);
}

// Shape checks shared by the prefill stages.  Fills Hr, Kr, R on success.
// Shapes of B sequences of at most T tokens holding `tokens` tokens in all (B*T, or the
// total of a ragged batch): R = tokens * Kr packed rows.
int check_dims(int B, int T, long long tokens, int H, int K, int d_head, int group, int* Hr, int* Kr, long long* R) {
  if (B < 1 || T < 1 || group < 1 || H < 1 || K < 1 || K > H || H % group || K % group) return NAMOH_ERR_INVALID_ARG;
  if (H / group > NAMOH_MAX_HEADS) return NAMOH_ERR_INVALID_ARG;
  if (d_head >= 0 && !supported_dims(d_head, group)) return NAMOH_ERR_UNSUPPORTED;
  if (T > kMaxPrefillT) return NAMOH_ERR_UNSUPPORTED;
  *Hr = H / group;
  *Kr = K / group;
  *R = tokens * *Kr;
  if (*R * group >= (1ll << 31)) return NAMOH_ERR_INVALID_ARG;
  if ((long long)B * *Hr > kMaxPrefillSegments) return NAMOH_ERR_UNSUPPORTED;
  return NAMOH_OK;
}

int check_shape(int B, int T, int H, int K, int d_head, int group, int* Hr, int* Kr, long long* R) {
  return check_dims(B, T, (long long)B * T, H, K, d_head, group, Hr, Kr, R);
}

// plan bytes for R packed rows in nseg segments: at most ceil(R/128) + nseg query tiles, g items each
size_t plan_bytes_rows(long long R, int nseg, int g) {
  const long long max_items = ((R + attn::kItemRows - 1) / attn::kItemRows + nseg) * g;
  return 16 + (size_t)max_items * sizeof(int4);
}

size_t plan_bytes_for(int B, int T, int Hr, int Kr, int g) { return plan_bytes_rows((long long)B * T * Kr, B * Hr, g); }

int plan_qtiles_for(int T) { return (T + kPlanTileRows - 1) / kPlanTileRows; }  // query tiles per segment, at most

// The RoPE launch builds the plan in one extra block when the plan's shared memory is small
// enough not to cut the RoPE blocks' occupancy.
constexpr int kFusedPlanSmemMax = 32 * 1024;

int launch_plan(const int32_t* seg_offsets, int nseg, int T, int g, const int32_t* seg_cap, void* plan,
                cudaStream_t stream) {
  const int max_qtiles = plan_qtiles_for(T);
  const int smem = plan_smem_ints(max_qtiles, nseg) * (int)sizeof(int);
  if (smem > 200 * 1024) return NAMOH_ERR_UNSUPPORTED;
  if (smem > 48 * 1024) {
    const cudaError_t e = cudaFuncSetAttribute(attn::plan_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "plan_kernel shared memory attribute");
  }
  int* header = static_cast<int*>(plan);
  int4* items = reinterpret_cast<int4*>(static_cast<char*>(plan) + 16);
  attn::plan_kernel<<<1, 1024, smem, stream>>>(seg_offsets, nseg, seg_cap, g, max_qtiles, header, items);
  return cuda_check_launch("plan_kernel launch");
}

// RoPE + cache pack; with a plan buffer also the attention plan (in the same launch when
// the plan's shared memory is small, else as a second kernel).
// rope_flags: NAMOH_ROPE_GLOBAL takes the positions from row_src: t = (row_src[r] / Kr) % T,
// or row_src[r] / Kr - cu_seqlens[b] in a ragged batch (T is then the longest sequence).
int launch_rope_and_plan(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int Hr, int Kr, int R,
                         int d_head, int group, float rope_base, unsigned rope_flags, const int32_t* cu_seqlens,
                         const int32_t* seg_offsets, const int32_t* row_src, uint16_t* q_rot, uint16_t* k_cache,
                         uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap, long long cache_rows,
                         uint32_t* dev_status, void* plan, const DeviceInfo& info, cudaStream_t stream,
                         const RopePool* pool = nullptr) {
  RopeTable tab;
  fill_rope_table(&tab, d_head, (double)rope_base);
  const int nseg = B * Hr;
  const int qtiles = plan_qtiles_for(T);
  const int32_t* plan_cap = seg_base ? seg_cap : nullptr;
  const bool fuse_plan = plan && plan_smem_ints(qtiles, nseg) * (int)sizeof(int) <= kFusedPlanSmemMax;
  const cudaError_t e = launch_rope_pack(d_head, q, k, v, R, group, seg_offsets, nseg, seg_base, seg_cap, cache_rows,
                                         q_rot, k_cache, v_cache, v_cache != v, tab, dev_status, info.sm_count, stream,
                                         fuse_plan ? plan : nullptr, qtiles, plan_cap,
                                         (rope_flags & NAMOH_ROPE_GLOBAL) ? row_src : nullptr, Kr, T, cu_seqlens,
                                         Hr, (rope_flags & NAMOH_ROPE_INTERLEAVED) != 0, pool);
  if (e != cudaSuccess) return cuda_fail(e, "rope_pack_kernel launch");
  if (plan && !fuse_plan) return launch_plan(seg_offsets, nseg, T, group, plan_cap, plan, stream);
  return NAMOH_OK;
}

int launch_attention(const uint16_t* q_rot, const uint16_t* k_cache, const uint16_t* v_cache, long long R, int D,
                     int g, const int32_t* seg_offsets, const int32_t* row_src, const float* gate,
                     const int64_t* seg_base, long long cache_rows, void* plan, uint16_t* y, uint32_t* dev_status,
                     const DeviceInfo& info, cudaStream_t stream, int window = 0,
                     const uint32_t* sa_mask = nullptr, int sa_words = 0, int sa_lg = 0,
                     uint64_t mma_wait_ns = kWaitLimitNs, bool withhold_q = false) {
  CUtensorMap tq, tk, tv;
  if (!attn::encode_rows_map(&tq, q_rot, R, g * D) || !attn::encode_rows_map(&tk, k_cache, cache_rows, D) ||
      !attn::encode_rows_map(&tv, v_cache, cache_rows, D))
    return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled");
  attn::Params p;
  p.seg_offsets = seg_offsets;
  p.seg_base = seg_base;
  p.row_src = row_src;
  p.gate = gate;
  p.sched = static_cast<int*>(plan);
  p.nitems = static_cast<int*>(plan) + 2;
  p.items = reinterpret_cast<const int4*>(static_cast<char*>(plan) + 16);
  p.y = y;
  p.rows = (int)R;
  p.window = window;
  p.g = g;
  p.y_sector_aligned = (reinterpret_cast<uintptr_t>(y) & 31u) == 0;
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  p.status = dev_status;
  p.sa_mask = sa_mask;
  p.sa_words = sa_words;
  p.sa_lg = sa_lg;
  p.mma_wait_ns = mma_wait_ns;
  p.withhold_q = withhold_q ? 1 : 0;
  cudaError_t e;
  if (sa_mask)
    e = (D == 128) ? attn::launch_attn<128, true>(tq, tk, tv, p, info.sm_count, stream)
                   : attn::launch_attn<64, true>(tq, tk, tv, p, info.sm_count, stream);
  else
    e = (D == 128) ? attn::launch_attn<128, false>(tq, tk, tv, p, info.sm_count, stream)
                   : attn::launch_attn<64, false>(tq, tk, tv, p, info.sm_count, stream);
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, "attn_fwd_kernel launch");
}

bool device_ok(DeviceInfo* info) {  // a Blackwell datacenter part with the shared memory the kernel needs
  return current_device_info(info) && info->major == 10 &&
         (size_t)attn::Smem<128>::kAlloc <= info->max_smem_optin;
}
}  // namespace

}  // namespace namoh

using namespace namoh;

extern "C" int namoh_rope_pack_ex(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H,
                                  int K, int d_head, int group, float rope_base, unsigned rope_flags,
                                  const int32_t* seg_offsets, const int32_t* row_src, uint16_t* q_rot,
                                  uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base,
                                  const int32_t* seg_cap, int64_t cache_rows, uint32_t* dev_status, void* plan,
                                  size_t plan_bytes, void* stream_v) {
  if (!q || !k || !v || !seg_offsets || !q_rot || !k_cache || !v_cache || !dev_status) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (!(rope_base > 1.0f) || !isfinite(rope_base)) return NAMOH_ERR_INVALID_ARG;
  if (!rope_flags_ok(rope_flags) || ((rope_flags & NAMOH_ROPE_GLOBAL) && !row_src)) return NAMOH_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(q_rot) || !aligned16(k_cache) ||
      !aligned16(v_cache))
    return NAMOH_ERR_INVALID_ARG;
  if (k_cache == k) return NAMOH_ERR_INVALID_ARG;
  if (seg_base) {
    if (!seg_cap || cache_rows < 1 || cache_rows >= (1ll << 31) || v_cache == v) return NAMOH_ERR_INVALID_ARG;
  } else {
    cache_rows = R;
  }
  if (plan && ((reinterpret_cast<uintptr_t>(plan) & 15u) || plan_bytes < plan_bytes_for(B, T, Hr, Kr, group)))
    return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!current_device_info(&info)) return cuda_fail(cudaGetLastError(), "device query");
  return launch_rope_and_plan(q, k, v, B, T, Hr, Kr, (int)R, d_head, group, rope_base, rope_flags, nullptr,
                              seg_offsets, row_src, q_rot, k_cache, v_cache, seg_base, seg_cap, cache_rows, dev_status,
                              plan, info, reinterpret_cast<cudaStream_t>(stream_v));
}

extern "C" int namoh_rope_pack(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H, int K,
                               int d_head, int group, float rope_base, const int32_t* seg_offsets, uint16_t* q_rot,
                               uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap,
                               int64_t cache_rows, uint32_t* dev_status, void* plan, size_t plan_bytes,
                               void* stream_v) {
  return namoh_rope_pack_ex(q, k, v, B, T, H, K, d_head, group, rope_base, 0u, seg_offsets, nullptr, q_rot, k_cache,
                            v_cache, seg_base, seg_cap, cache_rows, dev_status, plan, plan_bytes, stream_v);
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
  return launch_attention(q_rot, k_cache, v_cache, R, d_head, group, seg_offsets, row_src, gate, seg_base, cache_rows,
                          plan, y, dev_status, info, reinterpret_cast<cudaStream_t>(stream_v));
}

extern "C" int namoh_attention_timeout_probe(const uint16_t* q_rot, const uint16_t* k_cache, const uint16_t* v_cache,
                                             int B, int T, int H, int K, int d_head, int group,
                                             const int32_t* seg_offsets, const int32_t* row_src, const float* gate,
                                             void* plan, size_t plan_bytes, uint16_t* y, uint64_t wait_limit_ns,
                                             uint32_t* dev_status, void* stream_v) {
  if (!q_rot || !k_cache || !v_cache || !seg_offsets || !row_src || !gate || !y || !dev_status)
    return NAMOH_ERR_INVALID_ARG;
  if (wait_limit_ns < 1000ull || wait_limit_ns > kWaitLimitNs) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (!aligned16(q_rot) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(y)) return NAMOH_ERR_INVALID_ARG;
  if (!plan || (reinterpret_cast<uintptr_t>(plan) & 15u) || plan_bytes < plan_bytes_for(B, T, Hr, Kr, group))
    return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!device_ok(&info)) return NAMOH_ERR_UNSUPPORTED;
  return launch_attention(q_rot, k_cache, v_cache, R, d_head, group, seg_offsets, row_src, gate, nullptr, R, plan, y,
                          dev_status, info, reinterpret_cast<cudaStream_t>(stream_v), 0, nullptr, 0, 0,
                          wait_limit_ns, true);
}

namespace namoh {
namespace {
// Shared body of namoh_prefill_ex and namoh_prefill_varlen: R packed rows in B*Hr segments
// of at most T rows; cu_seqlens (ragged batch) only enters the global RoPE positions.
int prefill_impl(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int Hr, int Kr, long long R,
                 int d_head, int group, float rope_base, unsigned rope_flags, const int32_t* cu_seqlens,
                 const int32_t* seg_offsets, const int32_t* row_src, const float* gate, uint16_t* y, uint16_t* k_cache,
                 uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap, int64_t cache_rows,
                 int32_t* seg_len, void* workspace, size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!q || !k || !v || !seg_offsets || !row_src || !gate || !y || !k_cache || !v_cache || !dev_status)
    return NAMOH_ERR_INVALID_ARG;
  if (!(rope_base > 1.0f) || !isfinite(rope_base)) return NAMOH_ERR_INVALID_ARG;
  if (!rope_flags_ok(rope_flags)) return NAMOH_ERR_INVALID_ARG;
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
  void* plan = ws.take<char>(plan_bytes_rows(R, B * Hr, group));
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!device_ok(&info)) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);

  int st = launch_rope_and_plan(q, k, v, B, T, Hr, Kr, (int)R, d_head, group, rope_base, rope_flags, cu_seqlens,
                                seg_offsets, row_src, q_rot, k_cache, v_cache, seg_base, seg_cap, cache_rows,
                                dev_status, plan, info, stream);
  if (st != NAMOH_OK) return st;
  if (seg_len) {
    seg_len_kernel<<<(B * Hr + 255) / 256, 256, 0, stream>>>(seg_offsets, B * Hr, seg_len);
    if (const int st2 = cuda_check_launch("seg_len_kernel launch")) return st2;
  }
  return launch_attention(q_rot, k_cache, v_cache, R, d_head, group, seg_offsets, row_src, gate, seg_base, cache_rows,
                          plan, y, dev_status, info, stream);
}

size_t prefill_workspace_rows(long long R, int nseg, int d_head, int group) {
  WorkspaceCarver ws{nullptr, 0, 0};
  ws.take<uint16_t>((size_t)R * group * d_head);
  ws.take<char>(plan_bytes_rows(R, nseg, group));
  return align_up(ws.used, 256);
}

// shapes of a ragged batch: T = max_seqlen <= total_tokens, R = total_tokens * Kr
int check_varlen(int B, int total_tokens, int max_seqlen, int H, int K, int d_head, int group, int* Hr, int* Kr,
                 long long* R) {
  if (max_seqlen < 1 || total_tokens < max_seqlen) return NAMOH_ERR_INVALID_ARG;
  return check_dims(B, max_seqlen, total_tokens, H, K, d_head, group, Hr, Kr, R);
}
}  // namespace
}  // namespace namoh

extern "C" size_t namoh_prefill_workspace_size(int B, int T, int H, int K, int d_head, int group) {
  int Hr, Kr;
  long long R;
  if (check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R) != NAMOH_OK) return 0;
  return prefill_workspace_rows(R, B * Hr, d_head, group);
}

extern "C" int namoh_prefill_ex(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H, int K,
                                int d_head, int group, float rope_base, unsigned rope_flags,
                                const int32_t* seg_offsets, const int32_t* row_src, const float* gate, uint16_t* y,
                                uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base,
                                const int32_t* seg_cap, int64_t cache_rows, int32_t* seg_len, void* workspace,
                                size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  return prefill_impl(q, k, v, B, T, Hr, Kr, R, d_head, group, rope_base, rope_flags, nullptr, seg_offsets, row_src,
                      gate, y, k_cache, v_cache, seg_base, seg_cap, cache_rows, seg_len, workspace, workspace_bytes,
                      dev_status, stream_v);
}

extern "C" size_t namoh_prefill_varlen_workspace_size(int B, int total_tokens, int max_seqlen, int H, int K,
                                                      int d_head, int group) {
  int Hr, Kr;
  long long R;
  if (check_varlen(B, total_tokens, max_seqlen, H, K, d_head, group, &Hr, &Kr, &R) != NAMOH_OK) return 0;
  return prefill_workspace_rows(R, B * Hr, d_head, group);
}

extern "C" int namoh_prefill_varlen(const uint16_t* q, const uint16_t* k, const uint16_t* v,
                                    const int32_t* cu_seqlens, int B, int total_tokens, int max_seqlen, int H, int K,
                                    int d_head, int group, float rope_base, unsigned rope_flags,
                                    const int32_t* seg_offsets, const int32_t* row_src, const float* gate,
                                    uint16_t* y, uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base,
                                    const int32_t* seg_cap, int64_t cache_rows, int32_t* seg_len, void* workspace,
                                    size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!cu_seqlens) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  const int st = check_varlen(B, total_tokens, max_seqlen, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  return prefill_impl(q, k, v, B, max_seqlen, Hr, Kr, R, d_head, group, rope_base, rope_flags, cu_seqlens,
                      seg_offsets, row_src, gate, y, k_cache, v_cache, seg_base, seg_cap, cache_rows, seg_len,
                      workspace, workspace_bytes, dev_status, stream_v);
}

extern "C" int namoh_prefill(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H, int K,
                             int d_head, int group, float rope_base, const int32_t* seg_offsets,
                             const int32_t* row_src, const float* gate, uint16_t* y, uint16_t* k_cache,
                             uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap, int64_t cache_rows,
                             int32_t* seg_len, void* workspace, size_t workspace_bytes, uint32_t* dev_status,
                             void* stream_v) {
  return namoh_prefill_ex(q, k, v, B, T, H, K, d_head, group, rope_base, 0u, seg_offsets, row_src, gate, y, k_cache,
                          v_cache, seg_base, seg_cap, cache_rows, seg_len, workspace, workspace_bytes, dev_status,
                          stream_v);
}

// ---------------------------------------------------------------------------
// SA + NAMOH (App. B.8, selection model of App. B.3): block selection inside each routed history,
// then the routed attention over the kept blocks and the query's current block.
// ---------------------------------------------------------------------------
namespace namoh {
namespace {
constexpr int kSaMaxBlocks = 1024;  // blocks per history the selector holds

int sa_block_lg(int block) {
  return block == 32 ? 5 : block == 64 ? 6 : block == 128 ? 7 : -1;
}

int sa_words_for(int T, int block) { return ((T + block - 1) / block + 31) / 32; }

size_t sa_workspace_rows(long long R, int nseg, int d_head, int group, int block) {
  WorkspaceCarver ws{nullptr, 0, 0};
  ws.take<uint16_t>((size_t)R * group * d_head);
  ws.take<char>(plan_bytes_rows(R, nseg, group));
  ws.take<uint16_t>((size_t)(R / block + nseg) * d_head);
  return align_up(ws.used, 256);
}
}  // namespace
}  // namespace namoh

extern "C" int namoh_sa_mask_words(int T, int block) {
  if (T < 1 || sa_block_lg(block) < 0) return 0;
  return sa_words_for(T, block);
}

extern "C" size_t namoh_sa_prefill_workspace_size(int B, int T, int H, int K, int d_head, int group, int block) {
  int Hr, Kr;
  long long R;
  if (sa_block_lg(block) < 0 || check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R) != NAMOH_OK) return 0;
  return sa_workspace_rows(R, B * Hr, d_head, group, block);
}

extern "C" int namoh_sa_prefill(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int H, int K,
                                int d_head, int group, float rope_base, unsigned rope_flags,
                                const int32_t* seg_offsets, const int32_t* row_src, const float* gate, int block,
                                int alpha_num, int alpha_den, uint32_t* sa_mask, uint16_t* y, uint16_t* k_cache,
                                uint16_t* v_cache, const int64_t* seg_base, const int32_t* seg_cap,
                                int64_t cache_rows, int32_t* seg_len, void* workspace, size_t workspace_bytes,
                                uint32_t* dev_status, void* stream_v) {
  int Hr, Kr;
  long long R;
  const int st = check_shape(B, T, H, K, d_head, group, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  const int lg = sa_block_lg(block);
  if (lg < 0 || alpha_num < 1 || alpha_den < alpha_num || !sa_mask) return NAMOH_ERR_INVALID_ARG;
  if ((T + block - 1) / block > kSaMaxBlocks) return NAMOH_ERR_INVALID_ARG;
  if (!q || !k || !v || !seg_offsets || !row_src || !gate || !y || !k_cache || !v_cache || !dev_status)
    return NAMOH_ERR_INVALID_ARG;
  if (!(rope_base > 1.0f) || !isfinite(rope_base) || !rope_flags_ok(rope_flags)) return NAMOH_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(y) || !aligned16(k_cache) || !aligned16(v_cache) ||
      (reinterpret_cast<uintptr_t>(sa_mask) & 3u))
    return NAMOH_ERR_INVALID_ARG;
  if (k_cache == k) return NAMOH_ERR_INVALID_ARG;
  if (seg_base) {
    if (!seg_cap || cache_rows < 1 || cache_rows >= (1ll << 31) || v_cache == v) return NAMOH_ERR_INVALID_ARG;
  } else {
    cache_rows = R;
  }
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  const int nseg = B * Hr;
  WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
  uint16_t* q_rot = ws.take<uint16_t>((size_t)R * group * d_head);
  void* plan = ws.take<char>(plan_bytes_rows(R, nseg, group));
  const long long kbar_rows = R / block + nseg;
  uint16_t* kbar = ws.take<uint16_t>((size_t)kbar_rows * d_head);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!device_ok(&info)) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  const int words = sa_words_for(T, block);
  // blocks no taller than the RoPE pass's chunks are pooled by that pass, the others by their own kernel
  const bool pool_in_rope = block <= rope_chunk_rows(d_head, group);
  const RopePool pool{kbar, sa_mask, lg, words};
  int rc = launch_rope_and_plan(q, k, v, B, T, Hr, Kr, (int)R, d_head, group, rope_base, rope_flags, nullptr,
                                seg_offsets, row_src, q_rot, k_cache, v_cache, seg_base, seg_cap, cache_rows,
                                dev_status, plan, info, stream, pool_in_rope ? &pool : nullptr);
  if (rc != NAMOH_OK) return rc;
  if (seg_len) {
    seg_len_kernel<<<(nseg + 255) / 256, 256, 0, stream>>>(seg_offsets, nseg, seg_len);
    if (const int st2 = cuda_check_launch("seg_len_kernel launch")) return st2;
  }
  CUtensorMap tq;
  if (!attn::encode_rows_map(&tq, q_rot, R, group * d_head)) return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled");
  const long long max_items = ((R + attn::kItemRows - 1) / attn::kItemRows + nseg) * group;
  rc = launch_sa_select(tq, q_rot, k_cache, seg_offsets, seg_base, seg_base ? seg_cap : nullptr, cache_rows, nseg, T,
                        R, d_head, group, lg, alpha_num, alpha_den, kbar, kbar_rows, sa_mask, words, plan,
                        (int)max_items, dev_status, stream, pool_in_rope);
  if (rc != NAMOH_OK) return rc;
  return launch_attention(q_rot, k_cache, v_cache, R, d_head, group, seg_offsets, row_src, gate, seg_base, cache_rows,
                          plan, y, dev_status, info, stream, 0, sa_mask, words, lg);
}

// ---------------------------------------------------------------------------
// Shared heads (the paper's shared-head variant): every token of each always-active head,
// full causal or sliding window, global RoPE (the rank in a segment holding every token is
// t), no gate.  The layout is the identity one: segment (b, j) = rows (b Hs + j) T .. + T.
// ---------------------------------------------------------------------------
namespace namoh {
namespace {
// rows = false: seg_offsets only (the band kernel computes y's rows itself)
__global__ void shared_layout_kernel(int B, int T, int Hs, int32_t* __restrict__ seg_offsets,
                                     int32_t* __restrict__ row_src, float* __restrict__ gate, bool rows) {
  const long long R = (long long)B * Hs * T;
  if (!rows) {
    for (int s = blockIdx.x * blockDim.x + threadIdx.x; s <= B * Hs; s += gridDim.x * blockDim.x)
      seg_offsets[s] = (int32_t)((long long)s * T);
    return;
  }
  for (long long r = blockIdx.x * (long long)blockDim.x + threadIdx.x; r < R; r += (long long)gridDim.x * blockDim.x) {
    const long long bj = r / T, t = r - bj * T;
    const long long b = bj / Hs, j = bj - b * Hs;
    row_src[r] = (int32_t)((b * T + t) * Hs + j);  // y is [B, T, Hs, d]
    gate[r] = 1.f;
    if (t == 0) seg_offsets[bj] = (int32_t)r;
    if (r == R - 1) seg_offsets[B * Hs] = (int32_t)R;
  }
}

struct SharedWs {
  int32_t *seg_offsets, *row_src;
  float* gate;
  uint16_t* q_rot;
  void* plan;
};
void carve_shared(WorkspaceCarver& ws, SharedWs* o, int B, int T, int Hs, int d_head) {
  const long long R = (long long)B * Hs * T;
  o->seg_offsets = ws.take<int32_t>((size_t)B * Hs + 1);
  o->row_src = ws.take<int32_t>((size_t)R);
  o->gate = ws.take<float>((size_t)R);
  o->q_rot = ws.take<uint16_t>((size_t)R * d_head);
  o->plan = ws.take<char>(plan_bytes_rows(R, B * Hs, 1));
}
}  // namespace
}  // namespace namoh

extern "C" size_t namoh_shared_workspace_size(int B, int T, int Hs, int d_head) {
  int Hr, Kr;
  long long R;
  if (check_shape(B, T, Hs, Hs, d_head, 1, &Hr, &Kr, &R) != NAMOH_OK) return 0;
  WorkspaceCarver ws{nullptr, 0, 0};
  SharedWs o;
  carve_shared(ws, &o, B, T, Hs, d_head);
  return align_up(ws.used, 256);
}

extern "C" int namoh_shared_prefill(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int T, int Hs,
                                    int d_head, int window, float rope_base, unsigned rope_flags, uint16_t* y,
                                    uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base,
                                    const int32_t* seg_cap, int64_t cache_rows, int32_t* seg_len, void* workspace,
                                    size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!q || !k || !v || !y || !k_cache || !v_cache || !dev_status) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  long long R;
  int st = check_shape(B, T, Hs, Hs, d_head, 1, &Hr, &Kr, &R);
  if (st != NAMOH_OK) return st;
  if (window < 0 || !(rope_base > 1.0f) || !isfinite(rope_base) || !rope_flags_ok(rope_flags))
    return NAMOH_ERR_INVALID_ARG;
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
  SharedWs o;
  carve_shared(ws, &o, B, T, Hs, d_head);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!device_ok(&info)) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  // a window of at most one key tile: the band kernel (no plan, no per-row layout)
  const bool band = window > 0 && window <= kMaxBandWindow;
  if (band)
    shared_layout_kernel<<<(B * Hs + 256) / 256, 256, 0, stream>>>(B, T, Hs, o.seg_offsets, nullptr, nullptr, false);
  else
    shared_layout_kernel<<<info.sm_count * 4, 256, 0, stream>>>(B, T, Hs, o.seg_offsets, o.row_src, o.gate, true);
  if (const int e = cuda_check_launch("shared_layout_kernel launch")) return e;
  // global positions: the rank in a segment holding every token is t (the global flag is redundant)
  st = launch_rope_and_plan(q, k, v, B, T, Hs, Hs, (int)R, d_head, 1, rope_base, rope_flags & NAMOH_ROPE_INTERLEAVED,
                            nullptr, o.seg_offsets, o.row_src, o.q_rot, k_cache, v_cache, seg_base, seg_cap,
                            cache_rows, dev_status, band ? nullptr : o.plan, info, stream);
  if (st != NAMOH_OK) return st;
  if (seg_len) {
    seg_len_kernel<<<(B * Hs + 255) / 256, 256, 0, stream>>>(o.seg_offsets, B * Hs, seg_len);
    if (const int e = cuda_check_launch("seg_len_kernel launch")) return e;
  }
  if (band)
    return launch_window_attention(o.q_rot, k_cache, v_cache, B, T, Hs, d_head, window, seg_base, cache_rows, y,
                                   dev_status, info.sm_count, stream);
  return launch_attention(o.q_rot, k_cache, v_cache, R, d_head, 1, o.seg_offsets, o.row_src, o.gate, seg_base,
                          cache_rows, o.plan, y, dev_status, info, stream, window);
}
