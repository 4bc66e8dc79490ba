// proj.cu -- the projections around the routed-attention path (Sec. 3.1).
//
// One grouped GEMM over the packed rows of the routing (one group per KV-group head i, App. B.7),
// the A rows gathered from the token axis, in two modes:
//   QKV   (Eq. namoh-qkv): row r of segment (b, i) computes x_t [W_Q^(ig..ig+g-1) | W_K^(i) |
//         W_V^(i)] for t = row_src[r] / Kr, written as g query rows, one key row and one value
//         row in packed order -- the inputs of namoh_prefill.
//   OUT_P (Eq. namoh-attention): row r computes P_r = y_r [W_O^(ig); ...; W_O^(ig+g-1)] from
//         the combine's per-slot terms y = g h (A row = y[row_src[r]]), written (bf16) at the
//         token-slot row row_src[r]; combine_kernel then sums each token's K adjacent P rows
//         into o in fp32.
// Only active token-head pairs are computed (Sec. 3.1: inactive pairs generate nothing).
//
// One persistent CTA per SM, 288 threads:
//   warps 0-3  epilogue: TMEM lane = tile row; fp32 accumulators -> bf16 q, k, v rows
//   warps 4-7  loads: per 64-wide slice of the contraction the 128 gathered A rows arrive by
//              16-byte cp.async copies (a warp moves four whole 128-byte rows per instruction)
//              into the 128-byte-swizzled layout, and one TMA tile copy brings the group's
//              BN x 64 weight tile.  A thread retires stage j once its copies of it have
//              landed (wait_group, kLag stages later), fences them into the async proxy and
//              arrives on the stage's barrier.  (TMA gather4 moves only 512 bytes per
//              instruction and measured 7x slower here.)
//   warp 8     TMEM owner and MMA issue: tcgen05.mma kind::f16, M = 128, N = BN, K = 16
// QKV with exactly two column tiles (e.g. g = 1, d = 128: 384 columns as 2 x 192) computes both in
// one pass over the contraction: a stage holds the A slice once and both weight slices, and the
// two accumulators' MMAs alternate instruction by instruction (two chains in the tensor pipe
// instead of one; one TMEM buffer of 384 columns, so the epilogue does not overlap the next tile).
// The row-tile list comes from range_table_kernel + tile_list_kernel, or, for one token chunk of
// at most kListSeg segments, from each CTA itself: it reads the segment offsets and derives the
// entries it will run (no list kernels between the routing and the GEMM).
// Work items are (128-row tile of a segment, BN-column tile) from a list ordered by sequence,
// then position in the segment, then head: CTAs running at the same time work on the same
// stretch of tokens across heads, so x rows are reused from L2, and
// the N tiles of one row tile are adjacent items.  A static round robin hands out the items;
// the loaders fetch the next item's row indices during the current one.
// Two TMEM accumulators let the epilogue of one item overlap the main loop of the next.
// Every wait is bounded (NAMOH_DEV_TIMEOUT).
#include <algorithm>

#include "common.cuh"

namespace namoh {
namespace proj {

constexpr int BM = 128;  // packed rows per tile
constexpr int BK = 64;   // contraction elements per stage: one 128-byte swizzle row
constexpr int kThreads = 288;
constexpr int kSmemBudget = 208 * 1024;
constexpr int kMaxTileListBytes = 200 * 1024;  // shared memory of the tile-list builder
// A layout of at most kListSeg segments in one token chunk, with at most kListTiles row tiles per
// CTA, has its tile list computed by each CTA itself (no list kernels before the GEMM).
constexpr int kListSeg = 1024;
constexpr int kListTiles = 288;
constexpr int kListBytes = kListTiles * 16 + (2 * kListSeg + 1) * 4;


// pipeline stages that fit the shared-memory budget (at most 6)
constexpr int stages_for(int BN, int NT) {
  return kSmemBudget / (BM * 128 + NT * BN * 128) > 6 ? 6 : kSmemBudget / (BM * 128 + NT * BN * 128);
}

// NT column tiles of BN columns are computed together (NT accumulators, their MMAs interleaved
// per k-block, the stage holding the A slice once and NT weight slices).
template <int BN, int NT>
struct Layout {
  static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256, "UMMA N and the 32-column epilogue chunks");
  static_assert(NT >= 1 && NT * BN <= 512, "the accumulators fit in TMEM");
  static constexpr int kA = BM * 128;
  static constexpr int kB = NT * BN * 128;
  static constexpr int kBSlice = BN * 128;  // one column tile's weight slice (1024-byte multiple)
  // TMEM accumulator buffers: two (the epilogue of one group overlaps the next) when a group
  // takes at most 256 columns, else one
  static constexpr int kBufs = NT * BN <= 256 ? 2 : 1;
  static constexpr int kStage = kA + kB;
  static constexpr int kStages = kSmemBudget / kStage > 6 ? 6 : kSmemBudget / kStage;
  static constexpr int kLag = kStages - 2;  // stages of copies a loader keeps in flight before retiring one
  static_assert(kLag >= 1, "pipeline depth");
  static constexpr int kBar = kStages * kStage;
  static constexpr int kList = kBar + 256;          // the CTA's own tile list (when built in-kernel)
  static constexpr int kAlloc = kList + kListBytes + 1024;  // plus slack for 1024-byte alignment
};

struct Params {
  const int4* tiles;           // {first row, rows, segment, 0}: the 128-row tiles, in work order;
                               // null: each CTA derives its own tiles from seg_offsets
  const int32_t* seg_offsets;  // [nseg + 1] (the in-kernel list)
  const int32_t* tile_off;     // the list's first entry for this launch
  const int32_t* ntiles;       // the number of entries for this launch
  const int32_t* row_src;      // [R]
  int R;                       // packed rows: a tile row at or past R (an inconsistent layout) is skipped
  int nseg, Hr, Kr;
  int a_rows;                  // tokens (rows of x)
  int kdim;                    // contraction length: d_model
  int ncols;                   // output columns per group: (g + 2) d
  int g, d;
  const void* a;               // x [a_rows, kdim] (QKV), y [a_rows = N*Kr, g d] (OUT_P)
  uint16_t *q, *k, *v;         // outputs (OUT_P: q = P [a_rows, ncols])
  int out_aligned32;           // q, k, v 32-byte aligned: whole-sector stores
  long long p_row0;            // OUT_P: P row of token-slot row t Kr + k is t Kr + k - p_row0
  long long p_rows;            // OUT_P: rows of P
  uint32_t* status;
};

struct Bars {
  uint64_t full[6], empty[6];
  uint64_t acc_full[2], acc_empty[2];
  uint32_t tmem_base;
  int abort_flag;
};

struct Tile {
  int seg, row0, rows, hr, nt;
};

__device__ __forceinline__ Tile decode_tile(const Params& p, int4 e) {
  Tile t;
  t.row0 = e.x;
  t.rows = e.y;
  t.seg = e.z;
  t.hr = e.z % p.Hr;
  t.nt = 0;
  return t;
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, uint32_t* status) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status);
  return __all_sync(0xffffffffu, ok);
}

// 16 bytes global -> shared through the L1 path (no registers), completed by wait_group.
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gmem_src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Row ranges of the segments per token chunk: lo[c][s] = the first row of segment s whose token
// is >= c * chunk (rows ascend in token inside a segment); lo[nchunk][s] = the segment's end.
// With one chunk these are the segments' bounds.
__global__ void range_table_kernel(const int32_t* __restrict__ seg_offsets, const int32_t* __restrict__ row_src,
                                   int nseg, int nchunk, long long chunk, int Kr, int32_t* __restrict__ lo_tab) {
  const long long n = (long long)(nchunk + 1) * nseg;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const int c = (int)(i / nseg), s = (int)(i - (long long)c * nseg);
    const int a = __ldg(seg_offsets + s), e = max(a, __ldg(seg_offsets + s + 1));
    int lo = a, hi = e;
    if (c == nchunk) {
      lo = e;
    } else if (c > 0) {
      const long long target = (long long)c * chunk;
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if ((long long)(__ldg(row_src + mid) / Kr) < target) lo = mid + 1; else hi = mid;
      }
    }
    lo_tab[i] = lo;
  }
}

// The row-tile list (one block), chunk by chunk.  Inside a chunk: sequence b's tiles before
// b + 1's; tile p of every head before tile p + 1 of any, heads in order.  Tile (b, p, h) lands at
//   (tiles of sequences before b) + sum_h' min(p, n_tiles(b, h')) + #{h' < h : n_tiles(b, h') > p}.
// chunk_off[c] / chunk_cnt[c]: the chunk's first entry and its number of entries.
__global__ void __launch_bounds__(1024) tile_list_kernel(const int32_t* __restrict__ lo_tab, int nseg, int Hr,
                                                         int nchunk, int4* __restrict__ tiles,
                                                         int32_t* __restrict__ chunk_off,
                                                         int32_t* __restrict__ chunk_cnt) {
  extern __shared__ int s_nt[];  // [nseg] tiles per segment, then [nseg / Hr] per-sequence bases
  int* s_base = s_nt + nseg;
  __shared__ int s_total;
  const int B = nseg / Hr;
  const int tid = threadIdx.x;
  int done = 0;
  for (int c = 0; c < nchunk; ++c) {
    const int32_t* lo = lo_tab + (long long)c * nseg;
    const int32_t* hi = lo + nseg;
    for (int s = tid; s < nseg; s += blockDim.x) {
      const int n = __ldg(hi + s) - __ldg(lo + s);
      s_nt[s] = n > 0 ? (n + BM - 1) / BM : 0;
    }
    __syncthreads();
    if (tid == 0) {
      int run = 0;
      for (int b = 0; b < B; ++b) {
        s_base[b] = run;
        for (int h = 0; h < Hr; ++h) run += s_nt[b * Hr + h];
      }
      chunk_off[c] = done;
      chunk_cnt[c] = run;
      s_total = run;
    }
    __syncthreads();
    for (int s = tid; s < nseg; s += blockDim.x) {
      const int b = s / Hr, h = s - b * Hr;
      const int* nt = s_nt + b * Hr;
      const int r0 = __ldg(lo + s), r1 = __ldg(hi + s);
      for (int q = 0; q < nt[h]; ++q) {
        int pos = s_base[b];
        for (int h2 = 0; h2 < Hr; ++h2) pos += min(q, nt[h2]) + (h2 < h && nt[h2] > q ? 1 : 0);
        const int row0 = r0 + q * BM;
        tiles[done + pos] = make_int4(row0, min(BM, r1 - row0), s, 0);
      }
    }
    done += s_total;
    __syncthreads();
  }
}

enum Mode { kQKV = 0, kOutP = 1 };

template <int BN, int kMode, int NT>
__global__ void __launch_bounds__(kThreads, 1) proj_kernel(const __grid_constant__ CUtensorMap tm_b, Params p) {
  using L = Layout<BN, NT>;
  constexpr int NB = L::kBufs;
  constexpr int S = L::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + L::kBar);
  volatile int* abort_flag = &bars->abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&bars->full[i], 129);  // 128 loader threads + the weight tile's expect_tx
      mbar_init(&bars->empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->acc_full[i], 1);
      mbar_init(&bars->acc_empty[i], 4);
    }
    bars->abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 4 && lane == 0) tma_prefetch_desc(&tm_b);
  if (warp == 8) {
    tmem_alloc(&bars->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  pdl_wait();  // the routing layout, the tile list and the inputs are visible from here

  // A CTA takes row tiles mt = blockIdx.x, + gridDim.x, ... and runs every column tile of each
  // before the next (the tile's rows are decoded once and re-gathered from L2), NT at a time.
  const int nt_count = p.ncols / BN;
  const int ngroups = nt_count / NT;
  const int nk = p.kdim / BK;
  const int G = gridDim.x;
  const bool local_list = p.tiles == nullptr;
  int4* s_tiles = reinterpret_cast<int4*>(smem + L::kList);
  __shared__ int s_ntiles;
  int ntiles = 0;
  const int4* tiles = nullptr;
  if (!local_list) {
    ntiles = __ldg(p.ntiles);
    tiles = p.tiles + __ldg(p.tile_off);
  } else {
    // The list in the order tile_list_kernel writes: sequence b's tiles before b + 1's, tile q of
    // every head before tile q + 1 of any, heads in order.  Tile (b, q, h) is entry
    //   base(b) + cnt_b(q) + #{h' < h : nt(b, h') > q},  cnt_b(q) = sum_h' min(q, nt(b, h')),
    // so entry mt is found by the last b with base(b) <= mt, then the last q with
    // cnt_b(q) <= mt - base(b) (cnt_b grows with q), then the head.
    int* s_nt = reinterpret_cast<int*>(s_tiles + kListTiles);  // [nseg] row tiles per segment
    int* s_base = s_nt + kListSeg;                             // [B + 1] first entry per sequence
    const int B = p.nseg / p.Hr, Hr = p.Hr;
    for (int i = threadIdx.x; i < p.nseg; i += blockDim.x) {
      const int n = __ldg(p.seg_offsets + i + 1) - __ldg(p.seg_offsets + i);
      s_nt[i] = n > 0 ? (n + BM - 1) / BM : 0;
    }
    __syncthreads();
    for (int b = threadIdx.x; b < B; b += blockDim.x) {
      int tot = 0;
      for (int h = 0; h < Hr; ++h) tot += s_nt[b * Hr + h];
      s_base[b + 1] = tot;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      s_base[0] = 0;
      for (int b = 0; b < B; ++b) s_base[b + 1] += s_base[b];
      s_ntiles = s_base[B];
    }
    __syncthreads();
    ntiles = s_ntiles;
    for (int k = threadIdx.x; (int)blockIdx.x + k * G < ntiles && k < kListTiles; k += blockDim.x) {
      const int mt = (int)blockIdx.x + k * G;
      int lo = 0, hi = B;
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (s_base[mid] <= mt) lo = mid; else hi = mid;
      }
      const int b = lo, local = mt - s_base[b];
      const int* nt = s_nt + b * Hr;
      int qmax = 0;
      for (int h = 0; h < Hr; ++h) qmax = max(qmax, nt[h]);
      auto cnt = [&](int q) {
        int c = 0;
        for (int h = 0; h < Hr; ++h) c += min(q, nt[h]);
        return c;
      };
      int qlo = 0, qhi = qmax;  // cnt(qlo) <= local < cnt(qhi)
      while (qhi - qlo > 1) {
        const int mid = (qlo + qhi) >> 1;
        if (cnt(mid) <= local) qlo = mid; else qhi = mid;
      }
      int idx = local - cnt(qlo), h = 0;
      for (; h < Hr; ++h)
        if (nt[h] > qlo) {
          if (idx == 0) break;
          --idx;
        }
      const int sg = b * Hr + h;
      const int o0 = __ldg(p.seg_offsets + sg), n = __ldg(p.seg_offsets + sg + 1) - o0;
      s_tiles[k] = make_int4(o0 + qlo * BM, min(BM, n - qlo * BM), sg, 0);
    }
    __syncthreads();
  }
  // entry mt of the list (mt one of this CTA's: blockIdx.x + k G)
  auto tile_at = [&](int mt) -> int4 { return local_list ? s_tiles[(mt - (int)blockIdx.x) / G] : __ldg(tiles + mt); };

  if (warp >= 4 && warp < 8) {
    // ---- loads: thread lt moves 16-byte chunk (lt & 7) of rows (lt >> 3) + 16 w, w = 0..7
    constexpr int kLag = L::kLag;
    const int lt = threadIdx.x - 128;
    const int rq = lt >> 3, ch = lt & 7;
    const uint16_t* a_base = static_cast<const uint16_t*>(p.a);
    // routing row_src value -> the gathered A row, clamped into the tensor (rows past the
    // segment's end load row 0 and are not stored)
    auto in_rows = [&](const Tile& tt, int r) { return r < tt.rows && tt.row0 + r >= 0 && tt.row0 + r < p.R; };
    auto a_row_of = [&](int src) -> int {
      const int row = kMode == kQKV ? src / p.Kr : src;
      return min(max(row, 0), p.a_rows - 1);
    };
    uint32_t it = 0;
    bool ok = true;
    int mt = blockIdx.x;
    Tile t{};
    int rows_a[8];
    if (mt < ntiles) {
      t = decode_tile(p, tile_at(mt));
#pragma unroll
      for (int w = 0; w < 8; ++w) {
        const int r = rq + 16 * w;
        rows_a[w] = a_row_of(in_rows(t, r) ? ld_issue_s32(p.row_src + t.row0 + r) : 0);
      }
    }
    // the next row tile's entry, offsets and row indices are fetched during this one's k-blocks
    // (kq counts them across its column tiles), each load issued four k-blocks before its use
    const bool prefetch = ngroups * nk >= 12;
    for (; mt < ntiles && ok; mt += gridDim.x) {
      const int next = mt + gridDim.x;
      int nx_row0 = 0, nx_rows = 0, nx_seg = 0;
      Tile nx{};
      int nx_src[8];
      const uint16_t* src[8];
#pragma unroll
      for (int w = 0; w < 8; ++w) src[w] = a_base + (size_t)rows_a[w] * p.kdim + ch * 8;
      int kq = 0;
      for (int gi = 0; gi < ngroups && ok; ++gi) {
        const int b_row = t.hr * p.ncols + gi * NT * BN;
        for (int kb = 0; kb < nk; ++kb, ++it, ++kq) {
          if (prefetch && next < ntiles) {
            if (kq == 0) {
              if (local_list) {
                const int4 e = tile_at(next);
                nx_row0 = e.x;
                nx_rows = e.y;
                nx_seg = e.z;
              } else {
                const int32_t* e = reinterpret_cast<const int32_t*>(tiles + next);
                nx_row0 = ld_issue_s32(e);
                nx_rows = ld_issue_s32(e + 1);
                nx_seg = ld_issue_s32(e + 2);
              }
            } else if (kq == 4) {
              nx = decode_tile(p, make_int4(nx_row0, nx_rows, nx_seg, 0));
#pragma unroll
              for (int w = 0; w < 8; ++w) {
                const int r = rq + 16 * w;
                nx_src[w] = in_rows(nx, r) ? ld_issue_s32(p.row_src + nx.row0 + r) : 0;
              }
            }
          }
          const int slot = it % S;
          if (it >= (uint32_t)S && !warp_wait(&bars->empty[slot], ((it / S) - 1) & 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          uint8_t* a = smem + slot * L::kStage;
          if (lt == 0) {
            mbar_arrive_expect_tx(&bars->full[slot], L::kB);
#pragma unroll
            for (int j = 0; j < NT; ++j)
              tma_load_2d(a + L::kA + j * L::kBSlice, &tm_b, kb * BK, b_row + j * BN, &bars->full[slot]);
          }
#pragma unroll
          for (int w = 0; w < 8; ++w) {
            const int r = rq + 16 * w;
            cp_async16(a + r * 128 + ((ch ^ (r & 7)) << 4), src[w] + kb * BK);
          }
          cp_async_commit();
          if (it >= (uint32_t)kLag) {
            cp_async_wait<kLag>();
            fence_proxy_async_smem();
            mbar_arrive(&bars->full[(it - kLag) % S]);
          }
        }
      }
      if (!ok || next >= ntiles) break;
      if (prefetch) {
        t = nx;
#pragma unroll
        for (int w = 0; w < 8; ++w) rows_a[w] = a_row_of(nx_src[w]);
      } else {
        t = decode_tile(p, tile_at(next));
#pragma unroll
        for (int w = 0; w < 8; ++w) {
          const int r = rq + 16 * w;
          rows_a[w] = a_row_of(in_rows(t, r) ? ld_issue_s32(p.row_src + t.row0 + r) : 0);
        }
      }
    }
    if (ok) {  // retire the last stages
      cp_async_wait<0>();
      fence_proxy_async_smem();
      for (uint32_t j = it > (uint32_t)kLag ? it - kLag : 0; j < it; ++j) mbar_arrive(&bars->full[j % S]);
    }
  } else if (warp == 8) {
    // ---- MMA issue
    constexpr uint32_t idesc = make_idesc_bf16(BM, BN, false, false);
    uint32_t it = 0;
    bool ok = true;
    int li = 0;
    for (int mt = blockIdx.x; mt < ntiles && ok; mt += gridDim.x) {
      for (int gi = 0; gi < ngroups && ok; ++gi, ++li) {
        const int buf = li % NB;
        if (li >= NB && !warp_wait(&bars->acc_empty[buf], ((li / NB) - 1) & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + buf * 256;
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const int slot = it % S;
          if (!warp_wait(&bars->full[slot], (it / S) & 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t a_desc = make_smem_desc_sw128(smem_u32(smem + slot * L::kStage), 16, 1024);
          const uint64_t b_desc = make_smem_desc_sw128(smem_u32(smem + slot * L::kStage + L::kA), 16, 1024);
          // the NT accumulators' MMAs interleaved: independent chains overlap in the tensor pipe
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
#pragma unroll
            for (int j = 0; j < NT; ++j)
              mma_bf16_ss(d_tmem + j * BN, a_desc + (uint64_t)(kk * 2),
                          b_desc + (uint64_t)((j * L::kBSlice) >> 4) + (uint64_t)(kk * 2), idesc, (kb | kk) ? 1u : 0u);
          mma_commit(&bars->empty[slot]);
        }
        if (ok) mma_commit(&bars->acc_full[buf]);
      }
    }
  } else {
    // ---- epilogue: thread = tile row = TMEM lane
    const int row = warp * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    int li = 0;
    bool ok = true;
    for (int mt = blockIdx.x; mt < ntiles && ok; mt += gridDim.x) {
      const Tile t = decode_tile(p, tile_at(mt));
      const int r = t.row0 + row;
      const bool valid = row < t.rows && r >= 0 && r < p.R;
      // OUT_P writes row r's partial product at its token-slot row row_src[r]
      const long long dst_row = kMode == kOutP && valid ? ld_issue_s32(p.row_src + r) - p.p_row0 : r;
      for (int gi = 0; gi < ngroups; ++gi, ++li) {
        const int buf = li % NB;
        if (!warp_wait(&bars->acc_full[buf], (li / NB) & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < NT * BN / 32; ++c) {
          uint32_t v[32];
          tmem_ld32(tmem + lane_addr + buf * 256 + c * 32, v);
          tmem_wait_ld();
          if (!valid) continue;
          const int n = gi * NT * BN + c * 32;  // first output column of the chunk
          uint16_t* dst;
          if constexpr (kMode == kQKV) {
            const int gd = p.g * p.d;
            if (n < gd) dst = p.q + ((long long)r * p.g + n / p.d) * p.d + n % p.d;
            else if (n < gd + p.d) dst = p.k + (long long)r * p.d + (n - gd);
            else dst = p.v + (long long)r * p.d + (n - gd - p.d);
          } else {
            if (dst_row < 0 || dst_row >= p.p_rows) continue;  // an inconsistent layout
            dst = p.q + (long long)dst_row * p.ncols + n;
          }
          uint32_t w[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) w[e] = pack_bf16x2(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
          if (p.out_aligned32) {
            st_global_v8(dst, w);
            st_global_v8(dst + 16, w + 8);
          } else {
            uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
            for (int e = 0; e < 4; ++e) d4[e] = make_uint4(w[4 * e], w[4 * e + 1], w[4 * e + 2], w[4 * e + 3]);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->acc_empty[buf]);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) {
    // a wait gave up: let copies and MMAs still in flight finish before TMEM and the block go
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 1000000ull) {
    }
  }
  __syncthreads();
  if (warp == 8) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// o[t] (+)= sum_k P[t Kr + k] in fp32: a token's Kr slot rows are adjacent in P.
__global__ void combine_kernel(const uint16_t* __restrict__ P, long long ntok, int Kr, int d_model,
                               float* __restrict__ o, int accumulate) {
  const int v8 = d_model / 8;  // 16-byte vectors of P per row
  const long long n = ntok * v8;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const long long t = i / v8;
    const int c = (int)(i - t * v8);
    float a[8];
    if (accumulate) {
      const float4 o0 = reinterpret_cast<const float4*>(o + t * d_model)[2 * c];
      const float4 o1 = reinterpret_cast<const float4*>(o + t * d_model)[2 * c + 1];
      a[0] = o0.x; a[1] = o0.y; a[2] = o0.z; a[3] = o0.w;
      a[4] = o1.x; a[5] = o1.y; a[6] = o1.z; a[7] = o1.w;
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) a[e] = 0.f;
    }
    for (int k = 0; k < Kr; ++k) {
      const uint4 w = __ldg(reinterpret_cast<const uint4*>(P + (t * Kr + k) * d_model) + c);
      const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        a[2 * e] += bf16_lo(ws[e]);
        a[2 * e + 1] += bf16_hi(ws[e]);
      }
    }
    reinterpret_cast<float4*>(o + t * d_model)[2 * c] = make_float4(a[0], a[1], a[2], a[3]);
    reinterpret_cast<float4*>(o + t * d_model)[2 * c + 1] = make_float4(a[4], a[5], a[6], a[7]);
  }
}

bool encode_map(CUtensorMap* map, const void* base, long long rows, int cols, int box_rows) {
  EncodeTiledFn enc = tensor_map_encoder();
  if (!enc) return false;
  cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  cuuint32_t box[2] = {(cuuint32_t)BK, (cuuint32_t)box_rows};
  cuuint32_t estr[2] = {1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN, int kMode, int NT>
cudaError_t launch_bn_nt(const Params& p, const void* b, long long b_rows, int grid, cudaStream_t stream) {
  CUtensorMap tb;
  if (!encode_map(&tb, b, b_rows, p.kdim, BN)) return cudaErrorInvalidValue;
  const int smem = Layout<BN, NT>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(proj_kernel<BN, kMode, NT>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(proj_kernel<BN, kMode, NT>, dim3(grid), dim3(kThreads), (size_t)smem, stream, tb, p);
}

// Two column tiles per group when the QKV projection has exactly two and the group's stages
// still leave a 3-deep pipeline (A gathered once for both, two interleaved accumulators).
template <int BN, int kMode>
cudaError_t launch_bn(const Params& p, const void* b, long long b_rows, int grid, cudaStream_t stream) {
  if constexpr (kMode == kQKV && 2 * BN <= 512 && stages_for(BN, 2) >= 3) {
    if (p.ncols == 2 * BN) return launch_bn_nt<BN, kMode, 2>(p, b, b_rows, grid, stream);
  }
  return launch_bn_nt<BN, kMode, 1>(p, b, b_rows, grid, stream);
}

// The widest column tile (multiple of 32, at most 256) that divides the output columns.
int pick_bn(int ncols) {
  for (int bn : {256, 192, 160, 128, 96, 64})
    if (ncols % bn == 0) return bn;
  return 0;
}

template <int kMode>
cudaError_t launch(int bn, const Params& p, const void* b, long long b_rows, int grid, cudaStream_t stream) {
  switch (bn) {
    case 256: return launch_bn<256, kMode>(p, b, b_rows, grid, stream);
    case 192: return launch_bn<192, kMode>(p, b, b_rows, grid, stream);
    case 160: return launch_bn<160, kMode>(p, b, b_rows, grid, stream);
    case 128: return launch_bn<128, kMode>(p, b, b_rows, grid, stream);
    case 96: return launch_bn<96, kMode>(p, b, b_rows, grid, stream);
    default: return launch_bn<64, kMode>(p, b, b_rows, grid, stream);
  }
}

// Shapes shared by both projections: R = total_tokens * Kr packed rows in B * Hr segments.
int check_common(int B, int total_tokens, int d_model, int H, int K, int d_head, int group, int* Hr, int* Kr) {
  if (B < 1 || total_tokens < 1 || group < 1 || H < 1 || K < 1 || K > H || H % group || K % group)
    return NAMOH_ERR_INVALID_ARG;
  if (H / group > NAMOH_MAX_HEADS || (long long)B * (H / group) >= (1ll << 24)) return NAMOH_ERR_INVALID_ARG;
  if ((d_head != 64 && d_head != 128) || (group & (group - 1)) || group > 8) return NAMOH_ERR_UNSUPPORTED;
  // the list builder keeps B*Hr + B ints in shared memory
  if (((long long)B * (H / group) + B) * 4 > kMaxTileListBytes) return NAMOH_ERR_UNSUPPORTED;
  if (d_model < BK || d_model % BK || d_model > (1 << 16)) return NAMOH_ERR_UNSUPPORTED;
  *Hr = H / group;
  *Kr = K / group;
  const long long R = (long long)total_tokens * *Kr;
  if (R * group >= (1ll << 31) || (long long)total_tokens * d_model >= (1ll << 40)) return NAMOH_ERR_INVALID_ARG;
  return NAMOH_OK;
}

}  // namespace proj
}  // namespace namoh

using namespace namoh;


namespace {
// Workspace of the tile list for nchunk token chunks: the row-range table, the tiles (at most
// ceil(R / 128) + nchunk * nseg of them) and each chunk's offset and count.
struct TileList {
  int32_t* lo_tab;
  int4* tiles;
  int32_t *off, *cnt;
};
void carve_tiles(WorkspaceCarver& ws, TileList* t, long long R, int nseg, int nchunk) {
  t->lo_tab = ws.take<int32_t>((size_t)(nchunk + 1) * nseg);
  t->tiles = ws.take<int4>((size_t)((R + proj::BM - 1) / proj::BM + (long long)nchunk * nseg));
  t->off = ws.take<int32_t>((size_t)nchunk);
  t->cnt = ws.take<int32_t>((size_t)nchunk);
}

int build_tiles(const int32_t* seg_offsets, const int32_t* row_src, int nseg, int Hr, int Kr, int nchunk,
                long long chunk, const TileList& t, int sm_count, cudaStream_t stream) {
  const long long n = (long long)(nchunk + 1) * nseg;
  proj::range_table_kernel<<<(unsigned)std::min<long long>((n + 255) / 256, sm_count * 8LL), 256, 0, stream>>>(
      seg_offsets, row_src, nseg, nchunk, chunk, Kr, t.lo_tab);
  if (const int st = cuda_check_launch("range_table_kernel launch")) return st;
  const int smem = (nseg + nseg / Hr) * (int)sizeof(int);
  if (smem > 48 * 1024) {
    const cudaError_t e =
        cudaFuncSetAttribute(proj::tile_list_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return cuda_fail(e, "tile_list_kernel shared memory attribute");
  }
  proj::tile_list_kernel<<<1, 1024, smem, stream>>>(t.lo_tab, nseg, Hr, nchunk, t.tiles, t.off, t.cnt);
  return cuda_check_launch("tile_list_kernel launch");
}

// Whether each CTA can derive its own row tiles (one token chunk): the segment counts fit its
// shared-memory table and the CTA's share of the at most ceil(R / 128) + nseg tiles fits its list.
bool list_in_kernel(long long R, int nseg, int grid) {
  const long long max_tiles = (R + proj::BM - 1) / proj::BM + nseg;
  return nseg <= proj::kListSeg && (max_tiles + grid - 1) / grid <= proj::kListTiles;
}

// The output projection's token chunks bound the per-slot products kept at once (chunk Kr d_model
// bf16) to kOutChunkBytes of workspace.  (Chunks small enough for the products to stay in L2,
// 64 MB, measured slower: 184 against 147 us on the balanced layer, from the tail of each chunk's
// smaller launch.)
constexpr size_t kOutChunkBytes = 1ull << 30;
long long out_chunk_tokens(long long total_tokens, int Kr, int d_model) {
  long long c = (long long)(kOutChunkBytes / ((size_t)Kr * d_model * sizeof(uint16_t)));
  c = c < 128 ? 128 : c;
  return c < total_tokens ? c : total_tokens;
}

size_t qkv_workspace(long long total_tokens, int Kr, int nseg) {
  WorkspaceCarver ws{nullptr, 0, 0};
  TileList t;
  carve_tiles(ws, &t, total_tokens * Kr, nseg, 1);
  return align_up(ws.used, 256);
}

size_t out_workspace(long long total_tokens, int Kr, int nseg, int d_model) {
  const long long chunk = out_chunk_tokens(total_tokens, Kr, d_model);
  const int nchunk = (int)((total_tokens + chunk - 1) / chunk);
  WorkspaceCarver ws{nullptr, 0, 0};
  TileList t;
  carve_tiles(ws, &t, total_tokens * Kr, nseg, nchunk);
  ws.take<uint16_t>((size_t)chunk * Kr * d_model);
  return align_up(ws.used, 256);
}
}  // namespace

extern "C" size_t namoh_proj_workspace_size(int B, int total_tokens, int d_model, int H, int K, int group) {
  if (B < 1 || total_tokens < 1 || d_model < 1 || group < 1 || H < 1 || K < 1 || H % group || K % group) return 0;
  const int Hr = H / group, Kr = K / group;
  const size_t a = qkv_workspace(total_tokens, Kr, B * Hr), b = out_workspace(total_tokens, Kr, B * Hr, d_model);
  return a > b ? a : b;  // one size serves both calls
}

extern "C" int namoh_proj_qkv(const uint16_t* x, int total_tokens, int d_model, const uint16_t* w_qkv, int B, int H,
                              int K, int d_head, int group, const int32_t* seg_offsets, const int32_t* row_src,
                              uint16_t* q, uint16_t* k, uint16_t* v, void* workspace, size_t workspace_bytes,
                              uint32_t* dev_status, void* stream_v) {
  if (!x || !w_qkv || !seg_offsets || !row_src || !q || !k || !v || !dev_status) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  int st = proj::check_common(B, total_tokens, d_model, H, K, d_head, group, &Hr, &Kr);
  if (st != NAMOH_OK) return st;
  if (!aligned16(x) || !aligned16(w_qkv) || !aligned16(q) || !aligned16(k) || !aligned16(v))
    return NAMOH_ERR_INVALID_ARG;
  const int ncols = (group + 2) * d_head;
  const int bn = proj::pick_bn(ncols);
  DeviceInfo info;
  if (!current_device_info(&info) || info.major != 10) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  const int nseg = B * Hr;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
  TileList tl;
  carve_tiles(ws, &tl, (long long)total_tokens * Kr, nseg, 1);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  const bool local_list = list_in_kernel((long long)total_tokens * Kr, nseg, info.sm_count);
  if (!local_list) {
    st = build_tiles(seg_offsets, row_src, nseg, Hr, Kr, 1, total_tokens, tl, info.sm_count, stream);
    if (st != NAMOH_OK) return st;
  }
  proj::Params p{};
  p.tiles = local_list ? nullptr : tl.tiles;
  p.seg_offsets = seg_offsets;
  p.tile_off = tl.off;
  p.ntiles = tl.cnt;
  p.row_src = row_src;
  p.R = (int)((long long)total_tokens * Kr);
  p.nseg = nseg;
  p.Hr = Hr;
  p.Kr = Kr;
  p.a = x;
  p.a_rows = total_tokens;
  p.kdim = d_model;
  p.ncols = ncols;
  p.g = group;
  p.d = d_head;
  p.q = q;
  p.k = k;
  p.v = v;
  p.out_aligned32 = ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k) |
                      reinterpret_cast<uintptr_t>(v)) & 31u) == 0;
  p.status = dev_status;
  const cudaError_t e = proj::launch<proj::kQKV>(bn, p, w_qkv, (long long)Hr * ncols, info.sm_count, stream);
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, "proj_kernel (qkv) launch");
}

extern "C" int namoh_proj_out(const uint16_t* y, int total_tokens, int d_model, const uint16_t* w_o, int B, int H,
                              int K, int d_head, int group, const int32_t* seg_offsets, const int32_t* row_src,
                              float* o, int accumulate, void* workspace, size_t workspace_bytes, uint32_t* dev_status,
                              void* stream_v) {
  if (!y || !w_o || !seg_offsets || !row_src || !o || !dev_status) return NAMOH_ERR_INVALID_ARG;
  int Hr, Kr;
  int st = proj::check_common(B, total_tokens, d_model, H, K, d_head, group, &Hr, &Kr);
  if (st != NAMOH_OK) return st;
  if (!aligned16(y) || !aligned16(w_o) || !aligned16(o)) return NAMOH_ERR_INVALID_ARG;
  const int bn = proj::pick_bn(d_model);
  DeviceInfo info;
  if (!current_device_info(&info) || info.major != 10) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  const int nseg = B * Hr;
  const long long R = (long long)total_tokens * Kr;
  // token chunks whose per-slot products stay in L2 until the combine reads them
  const long long chunk = out_chunk_tokens(total_tokens, Kr, d_model);
  const int nchunk = (int)((total_tokens + chunk - 1) / chunk);
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
  TileList tl;
  carve_tiles(ws, &tl, R, nseg, nchunk);
  uint16_t* P = ws.take<uint16_t>((size_t)chunk * Kr * d_model);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  const bool local_list = nchunk == 1 && list_in_kernel(R, nseg, info.sm_count);
  if (!local_list) {
    st = build_tiles(seg_offsets, row_src, nseg, Hr, Kr, nchunk, chunk, tl, info.sm_count, stream);
    if (st != NAMOH_OK) return st;
  }
  proj::Params p{};
  p.tiles = local_list ? nullptr : tl.tiles;
  p.seg_offsets = seg_offsets;
  p.row_src = row_src;
  p.R = (int)R;
  p.nseg = nseg;
  p.Hr = Hr;
  p.Kr = Kr;
  p.a = y;
  p.a_rows = (int)R;
  p.kdim = group * d_head;
  p.ncols = d_model;
  p.g = group;
  p.d = d_head;
  p.q = P;
  p.out_aligned32 = 1;  // P starts 256-byte aligned and its rows are multiples of 128 bytes
  p.status = dev_status;
  for (int c = 0; c < nchunk; ++c) {
    const long long t0 = (long long)c * chunk, nt = std::min<long long>(chunk, total_tokens - t0);
    p.tile_off = tl.off + c;
    p.ntiles = tl.cnt + c;
    p.p_row0 = t0 * Kr;
    p.p_rows = nt * Kr;
    const cudaError_t e = proj::launch<proj::kOutP>(bn, p, w_o, (long long)Hr * d_model, info.sm_count, stream);
    if (e != cudaSuccess) return cuda_fail(e, "proj_kernel (out) launch");
    proj::combine_kernel<<<info.sm_count * 8, 256, 0, stream>>>(P, nt, Kr, d_model, o + t0 * d_model,
                                                                 accumulate ? 1 : 0);
    if (const int e2 = cuda_check_launch("combine_kernel launch")) return e2;
  }
  return NAMOH_OK;
}
