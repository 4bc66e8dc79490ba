// window_attn.cu -- the shared heads' sliding-window attention (Sec. 4.4, shared heads for local
// context): every token of an always-active head attends to the last w <= 128 tokens of its
// sequence, itself included, with RoPE at the token's global position (already applied to q~
// and k~ by the RoPE pass) and no gate.
//
// A query tile of 128 rows t0 .. t0 + 127 sees keys t0 - w + 1 .. t0 + 127: at most the key
// tile before it ("prev") and its own ("diag").  One S tile of 256 columns covers both,
// S = q~ [k~_prev | k~_diag]^T, and row i keeps columns i + 129 - w .. i + 128 of it (a band of
// w keys).  The softmax of a band is exact in one pass (no running max, no rescale), and
// P V = P_prev V_prev + P_diag V_diag is one accumulation over 256 keys.
//
// CTA (192 threads, one per SM); CTA c takes the contiguous run of query tiles
// [c N / G, (c + 1) N / G) of the N tiles of all segments, so that the diagonal key tile of one
// query tile is the previous key tile of the next and is loaded once:
//   warps 0-3  softmax / epilogue: thread i owns row i (TMEM lane i).  The rows of warp w see
//              columns 32 w + 1 .. 32 w + 159 only, so the warp reads the five 32-column chunks
//              w .. w + 4 of S and writes P for all 256 keys (zeros outside its columns).
//   warp 4     TMA producer: per query tile its Q tile, then K and V of its diagonal key tile
//              (and of the previous one when the tile starts a run mid-sequence), through a
//              6-slot ring of 128B-swizzled tiles.
//   warp 5     MMA issuer and TMEM owner.
// TMEM: two 256-column buffers, query tiles alternating between them.  In a buffer S_prev sits
// at [0, 128) and S_diag at [128, 256); P (bf16 pairs, 256 keys) then overwrites [0, 128) and O
// accumulates at [128, 128 + D).  The issuer puts S of tile i + 1 (two accumulators) ahead of PV
// of tile i, so that the softmax of tile i + 1 runs while PV(i) does, and the epilogue of tile i
// follows it.
// Every wait is bounded (NAMOH_DEV_TIMEOUT, then all roles drain and exit).
#include <algorithm>

#include "common.cuh"

namespace namoh {
namespace attn {
bool encode_rows_map(CUtensorMap* map, const void* base, long long rows, int row_elems);
}

namespace win {

constexpr int BM = 128;  // query rows per tile
constexpr int BN = 128;  // keys per key tile
constexpr int kMaxWindow = BN;
constexpr int kThreads = 192;
constexpr int kWarpLoad = 4;
constexpr int kWarpMma = 5;
constexpr int kRing = 6;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kBufCols = 256;  // one query tile's S, then P and O
constexpr uint32_t kOCol = 128;     // O within a buffer

template <int D>
struct Smem {
  static constexpr int kAtoms = D / 64;          // 64-column (128-byte) swizzle atoms per row
  static constexpr int kTileBytes = BM * D * 2;  // one Q / K / V tile
  static constexpr int kAtomBytes = BM * 128;    // 16 KB: 128 rows x 128 bytes
  static constexpr int kQ = 0;
  static constexpr int kRing0 = kTileBytes;
  static constexpr int kBar = kRing0 + kRing * kTileBytes;
  static constexpr int kBytes = kBar + 256;
  static constexpr int kAlloc = kBytes + 1024;  // slack for 1024-byte alignment
};

struct Bars {
  uint64_t q_full, q_empty;
  uint64_t ring_full[kRing], ring_empty[kRing];
  uint64_t s_full[2];  // S of the buffer's query tile written
  uint64_t p_full[2];  // P of it written (the four softmax warps)
  uint64_t o_full[2];  // its PV completed
  uint64_t o_free[2];  // its O read by the epilogue: the buffer may take the next S
  uint64_t drain;
  uint32_t tmem_base;
  int abort_flag;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

struct Params {
  int nseg;                 // segments (b, j) = shared head j of sequence b, T rows each
  int T, Hs;
  int window;               // 1 .. kMaxWindow
  int nq;                   // query tiles per segment: ceil(T / BM)
  long long ntiles;         // nseg * nq
  const int64_t* seg_base;  // [nseg] cache row of each segment's token 0, or null (s T)
  uint16_t* y;              // [B, T, Hs, D]: row (b T + t) Hs + j
  int y_sector_aligned;
  float scale_log2;         // log2(e) / sqrt(D)
  uint32_t* status;
};

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                          uint32_t* status) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status);
  return __all_sync(0xffffffffu, ok);
}

// The query tiles of CTA c: [lo, hi) of the ntiles tiles (segment-major).
__device__ __forceinline__ void cta_range(const Params& p, long long* lo, long long* hi) {
  const long long G = gridDim.x, c = blockIdx.x;
  *lo = p.ntiles * c / G;
  *hi = p.ntiles * (c + 1) / G;
}

// Tile li of the CTA's run: its segment, query tile, whether it reads a previous key tile and
// whether that tile is the previous query tile's diagonal one (already in the ring).
struct Tile {
  int s, qt;
  bool has_prev, chained;
};
__device__ __forceinline__ Tile tile_of(const Params& p, long long lo, long long li) {
  Tile t;
  const long long i = lo + li;
  t.s = (int)(i / p.nq);
  t.qt = (int)(i - (long long)t.s * p.nq);
  t.has_prev = t.qt >= 1 && p.window >= 2;
  t.chained = li >= 1 && t.qt >= 1;
  return t;
}

// Ring entries of one tile (in load order: [K_prev], K_diag, [V_prev], V_diag), given the ring
// counter at its start and the previous tile's diagonal entries.
struct Entries {
  uint32_t kp, kd, vp, vd;
  uint32_t next;  // ring counter after the tile's loads
};
__device__ __forceinline__ Entries entries_of(const Tile& t, uint32_t ring, uint32_t prev_kd, uint32_t prev_vd) {
  Entries e;
  if (t.has_prev && !t.chained) {
    e.kp = ring;
    e.kd = ring + 1;
    e.vp = ring + 2;
    e.vd = ring + 3;
    e.next = ring + 4;
  } else {
    e.kd = ring;
    e.vd = ring + 1;
    e.kp = prev_kd;
    e.vp = prev_vd;
    e.next = ring + 2;
  }
  return e;
}

// Softmax of one band tile for the rows of warp w: S columns 32 w .. 32 w + 159 from TMEM, the
// band and sequence-start masks, the exact row max and sum, and P = exp2(S * scale - m) as bf16
// pairs over the buffer's first 128 columns: the warp's 80 packed columns at 16 w .. 16 w + 79,
// zeros in the other 48.  One code path for the four warps (the column offsets are runtime
// TMEM addresses).  Returns the row sum.
__device__ __forceinline__ float band_softmax(uint32_t buf, int w, int lane, int qt, int window, float scale_log2) {
  constexpr int kCols = 160;
  float sv[kCols];
#pragma unroll
  for (int c = 0; c < 5; ++c) {
    uint32_t r[32];
    tmem_ld32(buf + (uint32_t)(32 * (w + c)), r);
#pragma unroll
    for (int i = 0; i < 32; ++i) sv[c * 32 + i] = __uint_as_float(r[i]);
  }
  tmem_wait_ld();
  // column 32 w + j holds key rank t0 - 128 + 32 w + j, the row's query rank is t0 + 32 w + lane:
  // in the band iff lane + 129 - window <= j <= lane + 128, and a key rank below 0 is no key
  int lo = lane + BN + 1 - window;
  if (qt == 0) lo = max(lo, BN - 32 * w);
  const int hi = lane + BN;
#pragma unroll
  for (int j = 0; j < kCols; ++j)
    if (j < lo || j > hi) sv[j] = -INFINITY;
  float m8[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) m8[i] = fmax3(sv[i], sv[8 + i], sv[16 + i]);
#pragma unroll
  for (int c = 24; c < kCols - 8; c += 16) {
#pragma unroll
    for (int i = 0; i < 8; ++i) m8[i] = fmax3(m8[i], sv[c + i], sv[c + 8 + i]);
  }
#pragma unroll
  for (int i = 0; i < 8; ++i) m8[i] = fmaxf(m8[i], sv[kCols - 8 + i]);
  const float mx = fmax3(fmax3(m8[0], m8[1], m8[2]), fmax3(m8[3], m8[4], m8[5]), fmaxf(m8[6], m8[7]));
  const float m = mx * scale_log2;  // finite: every row keeps at least its own key
  uint64_t sum2[4] = {0ull, 0ull, 0ull, 0ull};
  const uint64_t sc2 = f2_pack(scale_log2, scale_log2), nm2 = f2_pack(-m, -m);
  // P: packed column c holds keys 2c, 2c + 1 of the 256; written 16 columns at a time
#pragma unroll
  for (int q = 0; q < 5; ++q) {
    uint32_t r[16];
#pragma unroll
    for (int e = 0; e < 16; ++e) {
      const int j = 32 * q + 2 * e;
      float x0, x1;
      f2_unpack(f2_fma(f2_pack(sv[j], sv[j + 1]), sc2, nm2), x0, x1);
      const float e0 = fast_exp2(x0), e1 = fast_exp2(x1);
      sum2[e & 3] = f2_add(sum2[e & 3], f2_pack(e0, e1));
      r[e] = pack_bf16x2(e0, e1);
    }
    tmem_st16(buf + (uint32_t)(16 * (w + q)), r);
  }
  uint32_t z[16];
#pragma unroll
  for (int e = 0; e < 16; ++e) z[e] = 0u;
  for (int b = 0; b < 8; ++b)
    if (b < w || b >= w + 5) tmem_st16(buf + (uint32_t)(16 * b), z);
  float sa, sb;
  f2_unpack(f2_add(f2_add(sum2[0], sum2[1]), f2_add(sum2[2], sum2[3])), sa, sb);
  return sa + sb;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    window_attn_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                       const __grid_constant__ CUtensorMap tm_v, Params p) {
  using L = Smem<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + L::kBar);
  volatile int* abort_flag = &bars->abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    mbar_init(&bars->q_full, 1);
    mbar_init(&bars->q_empty, 1);
    for (int i = 0; i < kRing; ++i) {
      mbar_init(&bars->ring_full[i], 1);
      mbar_init(&bars->ring_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->p_full[i], 4);
      mbar_init(&bars->o_full[i], 1);
      mbar_init(&bars->o_free[i], 4);
    }
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
  pdl_launch_dependents();
  pdl_wait();  // q~ and the caches come from the RoPE pass before this kernel
  long long lo, hi;
  cta_range(p, &lo, &hi);
  const int n = (int)(hi - lo);

  if (warp == kWarpLoad) {
    // ------------------------------------------------------------------ TMA producer
    if (lane == 0) {
      uint32_t ring = 0;
      bool ok = true;
      auto load_tile = [&](const CUtensorMap* tm, long long row) {
        const int slot = ring % kRing;
        const uint32_t use = ring / kRing;
        if (use > 0 && !mbar_wait(&bars->ring_empty[slot], (use - 1) & 1, abort_flag, p.status)) return false;
        mbar_arrive_expect_tx(&bars->ring_full[slot], L::kTileBytes);
        for (int a = 0; a < L::kAtoms; ++a)
          tma_load_2d(smem + L::kRing0 + slot * L::kTileBytes + a * L::kAtomBytes, tm, a * 64, (int32_t)row,
                      &bars->ring_full[slot]);
        ++ring;
        return true;
      };
      for (int li = 0; li < n && ok; ++li) {
        const Tile t = tile_of(p, lo, li);
        if (li > 0) ok = mbar_wait(&bars->q_empty, (li - 1) & 1, abort_flag, p.status);
        if (!ok) break;
        mbar_arrive_expect_tx(&bars->q_full, L::kTileBytes);
        for (int a = 0; a < L::kAtoms; ++a)
          tma_load_2d(smem + L::kQ + a * L::kAtomBytes, &tm_q, a * 64, (int32_t)((long long)t.s * p.T + t.qt * BM),
                      &bars->q_full);
        const long long kb = (p.seg_base ? p.seg_base[t.s] : (long long)t.s * p.T) + (long long)t.qt * BN;
        const bool load_prev = t.has_prev && !t.chained;
        if (load_prev) ok = load_tile(&tm_k, kb - BN);
        if (ok) ok = load_tile(&tm_k, kb);
        if (ok && load_prev) ok = load_tile(&tm_v, kb - BN);
        if (ok) ok = load_tile(&tm_v, kb);
      }
      if (!ok) {
        const uint64_t t0 = global_timer_ns();
        while (global_timer_ns() - t0 < 1000000ull) {
        }
      }
    }
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_qk = make_idesc_bf16(BM, BN, false, false);
    constexpr uint32_t idesc_pv = make_idesc_bf16(BM, D, false, true);
    const uint64_t q_desc = make_smem_desc_sw128(smem_u32(smem + L::kQ), 16, 1024);
    auto qk_off = [](int kk) -> uint64_t { return (uint64_t)(((kk >> 2) * L::kAtomBytes + (kk & 3) * 32) >> 4); };
    auto pv_off = [](int kk) -> uint64_t { return (uint64_t)((kk * 2048) >> 4); };
    auto slot_addr = [&](uint32_t r) { return smem_u32(smem + L::kRing0 + (r % kRing) * L::kTileBytes); };
    auto ring_ready = [&](uint32_t r) {
      return warp_wait(&bars->ring_full[r % kRing], (r / kRing) & 1, abort_flag, p.status);
    };
    // rows of a V tile past the sequence end hold other data: zero them, so that the 0 weights
    // of P there cannot meet a NaN
    auto zero_v_tail = [&](uint32_t r, int valid_keys) {
      uint8_t* vtile = smem + L::kRing0 + (r % kRing) * L::kTileBytes;
      for (int a = 0; a < L::kAtoms; ++a) {
        uint4* vb = reinterpret_cast<uint4*>(vtile + a * L::kAtomBytes);
        for (int i = valid_keys * 8 + lane; i < BN * 8; i += 32) vb[i] = make_uint4(0, 0, 0, 0);
      }
      fence_proxy_async_smem();
      __syncwarp();
    };
    // whether tile li's diagonal key tile is read again by tile li + 1
    auto reused = [&](int li) {
      if (li + 1 >= n) return false;
      const Tile nx = tile_of(p, lo, li + 1);
      return nx.chained && nx.has_prev;
    };
    // S of tile li into buffer li & 1: S_prev and S_diag interleaved instruction by instruction
    auto issue_s = [&](int li, const Tile& t, const Entries& e) {
      const uint32_t sbuf = tmem + kBufCols * (uint32_t)(li & 1);
      const uint64_t kp = make_smem_desc_sw128(slot_addr(e.kp), 16, 1024);
      const uint64_t kd = make_smem_desc_sw128(slot_addr(e.kd), 16, 1024);
#pragma unroll
      for (int ks = 0; ks < D / 16; ++ks) {
        if (t.has_prev) mma_bf16_ss(sbuf, q_desc + qk_off(ks), kp + qk_off(ks), idesc_qk, ks > 0 ? 1u : 0u);
        mma_bf16_ss(sbuf + BN, q_desc + qk_off(ks), kd + qk_off(ks), idesc_qk, ks > 0 ? 1u : 0u);
      }
      mma_commit(&bars->s_full[li & 1]);
      mma_commit(&bars->q_empty);
      if (t.has_prev) mma_commit(&bars->ring_empty[e.kp % kRing]);
      if (!reused(li)) mma_commit(&bars->ring_empty[e.kd % kRing]);
    };
    // PV of tile li: O = P_prev V_prev + P_diag V_diag, 16 (or 8) instructions into one accumulator
    auto issue_pv = [&](int li, const Tile& t, const Entries& e) {
      const uint32_t pbuf = tmem + kBufCols * (uint32_t)(li & 1);
      const uint64_t vp = make_smem_desc_sw128(slot_addr(e.vp), L::kAtomBytes, 1024);
      const uint64_t vd = make_smem_desc_sw128(slot_addr(e.vd), L::kAtomBytes, 1024);
      if (t.has_prev) {
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          mma_bf16_ts(pbuf + kOCol, pbuf + (uint32_t)(kk * 8), vp + pv_off(kk), idesc_pv, kk > 0 ? 1u : 0u);
      }
#pragma unroll
      for (int kk = 0; kk < 8; ++kk)
        mma_bf16_ts(pbuf + kOCol, pbuf + (uint32_t)(64 + kk * 8), vd + pv_off(kk), idesc_pv,
                    (kk > 0 || t.has_prev) ? 1u : 0u);
      mma_commit(&bars->o_full[li & 1]);
      if (t.has_prev) mma_commit(&bars->ring_empty[e.vp % kRing]);
      if (!reused(li)) mma_commit(&bars->ring_empty[e.vd % kRing]);
    };
    // the waits S of tile li needs: its buffer free, its Q tile and its K tiles
    auto s_ready = [&](int li, const Tile& t, const Entries& e) {
      if (li >= 2 && !warp_wait(&bars->o_free[li & 1], ((li >> 1) - 1) & 1, abort_flag, p.status)) return false;
      if (!warp_wait(&bars->q_full, li & 1, abort_flag, p.status)) return false;
      if (t.has_prev && !ring_ready(e.kp)) return false;
      return ring_ready(e.kd);
    };
    // the waits PV of tile li needs: its P and its V tiles (a partial last one zeroed past the end)
    auto pv_ready = [&](int li, const Tile& t, const Entries& e) {
      if (!warp_wait(&bars->p_full[li & 1], (li >> 1) & 1, abort_flag, p.status)) return false;
      if (t.has_prev && !ring_ready(e.vp)) return false;
      if (!ring_ready(e.vd)) return false;
      const int valid = p.T - t.qt * BN;
      if (valid < BN) zero_v_tail(e.vd, valid);
      return true;
    };
    // Order: S(0); then for each tile li, S(li + 1) as soon as its buffer is free (the softmax
    // of tile li + 1 then overlaps PV(li)), then PV(li)
    bool ok = true;
    uint32_t ring = 0;
    Tile tc{}, tn{};
    Entries cur{}, nxt{};
    if (n > 0) {
      tc = tile_of(p, lo, 0);
      cur = entries_of(tc, ring, 0, 0);
      ring = cur.next;
      ok = s_ready(0, tc, cur);
      if (ok) {
        tc_fence_after();
        issue_s(0, tc, cur);
      }
    }
    for (int li = 0; li < n && ok; ++li) {
      if (li + 1 < n) {
        tn = tile_of(p, lo, li + 1);
        nxt = entries_of(tn, ring, cur.kd, cur.vd);
        ring = nxt.next;
        ok = s_ready(li + 1, tn, nxt);
        if (!ok) break;
        tc_fence_after();
        issue_s(li + 1, tn, nxt);
      }
      ok = pv_ready(li, tc, cur);
      if (!ok) break;
      tc_fence_after();
      issue_pv(li, tc, cur);
      tc = tn;
      cur = nxt;
    }
    if (!ok) {
      mma_commit(&bars->drain);
      const uint64_t t0 = global_timer_ns();
      while (!mbar_try_wait(&bars->drain, 0) && global_timer_ns() - t0 < 100000000ull) {
      }
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------------------ softmax / epilogue
    // Order: softmax(0); then for each tile li, the softmax of tile li + 1 (its S comes before
    // PV(li)) and then the epilogue of tile li.
    const int row = warp * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    bool ok = true;
    auto softmax = [&](int li, float* l) {
      const Tile t = tile_of(p, lo, li);
      const uint32_t buf = tmem + lane_addr + kBufCols * (uint32_t)(li & 1);
      if (!warp_wait(&bars->s_full[li & 1], (li >> 1) & 1, abort_flag, p.status)) return false;
      tc_fence_after();
      *l = band_softmax(buf, warp, lane, t.qt, p.window, p.scale_log2);
      tmem_wait_st();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->p_full[li & 1]);
      return true;
    };
    float l_cur = 0.f, l_next = 0.f;
    if (n > 0) ok = softmax(0, &l_cur);
    for (int li = 0; li < n && ok; ++li) {
      if (li + 1 < n) {
        ok = softmax(li + 1, &l_next);
        if (!ok) break;
      }
      // epilogue: O out of TMEM (the buffer is then free), O / l as bf16 to y
      const Tile t = tile_of(p, lo, li);
      const uint32_t buf = tmem + lane_addr + kBufCols * (uint32_t)(li & 1);
      ok = warp_wait(&bars->o_full[li & 1], (li >> 1) & 1, abort_flag, p.status);
      if (!ok) break;
      tc_fence_after();
      uint32_t o[D / 32][32];
#pragma unroll
      for (int c = 0; c < D / 32; ++c) tmem_ld32(buf + kOCol + (uint32_t)(c * 32), o[c]);
      tmem_wait_ld();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->o_free[li & 1]);
      const int tq = t.qt * BM + row;
      if (tq < p.T) {
        const float inv = 1.0f / l_cur;
        uint32_t w[D / 2];
#pragma unroll
        for (int e = 0; e < D / 2; ++e)
          w[e] = pack_bf16x2(__uint_as_float(o[e / 16][(e % 16) * 2]) * inv,
                             __uint_as_float(o[e / 16][(e % 16) * 2 + 1]) * inv);
        const int b = t.s / p.Hs, j = t.s - b * p.Hs;
        uint16_t* dst = p.y + (((long long)b * p.T + tq) * p.Hs + j) * D;
        if (p.y_sector_aligned) {
#pragma unroll
          for (int c = 0; c < D / 16; ++c) st_global_v8(dst + c * 16, w + c * 8);
        } else {
#pragma unroll
          for (int c = 0; c < D / 8; ++c)
            *reinterpret_cast<uint4*>(dst + c * 8) = make_uint4(w[4 * c], w[4 * c + 1], w[4 * c + 2], w[4 * c + 3]);
        }
      }
      l_cur = l_next;
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kWarpMma) tmem_dealloc(tmem, kTmemCols);
}

template <int D>
cudaError_t launch_d(const CUtensorMap& tq, const CUtensorMap& tk, const CUtensorMap& tv, const Params& p, int grid,
                     cudaStream_t stream) {
  const int smem = Smem<D>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(window_attn_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  e = launch_pdl(window_attn_kernel<D>, dim3(grid), dim3(kThreads), (size_t)smem, stream, tq, tk, tv, p);
  return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace win

// The shared heads' attention under a sliding window of 1 .. 128 keys: q_rot holds segment
// s = b Hs + j at rows s T .. s T + T - 1, its keys and values sit in the caches at rows
// seg_base[s] + t (s T + t without seg_base), y is [B, T, Hs, D].
int launch_window_attention(const uint16_t* q_rot, const uint16_t* k_cache, const uint16_t* v_cache, int B, int T,
                            int Hs, int D, int window, const int64_t* seg_base, long long cache_rows, uint16_t* y,
                            uint32_t* dev_status, int sm_count, cudaStream_t stream) {
  if (window < 1 || window > win::kMaxWindow || (D != 64 && D != 128)) return NAMOH_ERR_INVALID_ARG;
  const long long nseg = (long long)B * Hs, R = nseg * T;
  CUtensorMap tq, tk, tv;
  if (!attn::encode_rows_map(&tq, q_rot, R, D) || !attn::encode_rows_map(&tk, k_cache, cache_rows, D) ||
      !attn::encode_rows_map(&tv, v_cache, cache_rows, D))
    return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled");
  win::Params p;
  p.nseg = (int)nseg;
  p.T = T;
  p.Hs = Hs;
  p.window = window;
  p.nq = (T + win::BM - 1) / win::BM;
  p.ntiles = nseg * p.nq;
  p.seg_base = seg_base;
  p.y = y;
  p.y_sector_aligned = (reinterpret_cast<uintptr_t>(y) & 31u) == 0;
  p.scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  p.status = dev_status;
  const int grid = (int)std::min<long long>(sm_count, p.ntiles);
  const cudaError_t e = D == 128 ? win::launch_d<128>(tq, tk, tv, p, grid, stream)
                                 : win::launch_d<64>(tq, tk, tv, p, grid, stream);
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, "window_attn_kernel launch");
}

}  // namespace namoh
