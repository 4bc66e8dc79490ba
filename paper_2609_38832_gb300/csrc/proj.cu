// proj.cu -- the projections around the routed-attention path (Sec. 3.1).
//
// Both are grouped GEMMs over the packed rows of the routing (one group per KV-group head i,
// App. C), with the A rows gathered from the token axis:
//   QKV (Eq. namoh-qkv):  row r of segment (b, i) computes x_t [W_Q^(ig..ig+g-1) | W_K^(i) | W_V^(i)]
//                         for t = row_src[r] / Kr, written as g query rows, one key row and one
//                         value row in packed order -- the inputs of namoh_prefill.
//   OUT (Eq. namoh-attention, o_t = sum_i g h W_O^(i)): row r computes y_r [W_O^(ig); ...;
//                         W_O^(ig+g-1)] from the combine's per-slot terms y = g h and adds it
//                         into o[t] (fp32): the token's K slots sum there.
// Only active token-head pairs are computed (Sec. 3.1: inactive pairs generate nothing).
//
// One persistent CTA per SM, 192 threads:
//   warps 0-3  epilogue: TMEM lane = tile row; fp32 accumulators -> bf16 rows (QKV) or fp32
//              reductions into o (OUT)
//   warp 4     loads: per 64-wide slice of the contraction, 32 TMA gather4 copies (one per lane,
//              four token rows each) fill the 128-row A tile in the 128-byte-swizzled layout,
//              and one TMA tile copy brings the group's BN x 64 weight tile
//   warp 5     TMEM owner and MMA issue: tcgen05.mma kind::f16, M = 128, N = BN, K = 16
// Work items are (128-row tile of a segment, BN-column tile), taken in a static round robin;
// the N tiles of one row tile are adjacent items, so the gathered rows are reused from L2.
// Two TMEM accumulators let the epilogue of one item overlap the main loop of the next.
// Every wait is bounded (NAMOH_DEV_TIMEOUT).
#include "common.cuh"

namespace namoh {
namespace proj {

constexpr int BM = 128;  // packed rows per tile
constexpr int BK = 64;   // contraction elements per stage: one 128-byte swizzle row
constexpr int kThreads = 192;
constexpr int kSmemBudget = 212 * 1024;

enum Mode { kQKV = 0, kOut = 1 };

template <int BN>
struct Layout {
  static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256, "UMMA N and the 32-column epilogue chunks");
  static constexpr int kA = BM * 128;
  static constexpr int kB = BN * 128;
  static constexpr int kStage = kA + kB;
  static constexpr int kStages = kSmemBudget / kStage > 6 ? 6 : kSmemBudget / kStage;
  static constexpr int kBar = kStages * kStage;
  static constexpr int kAlloc = kBar + 256 + 1024;  // barriers, plus slack for 1024-byte alignment
};

struct Params {
  const int32_t* seg_offsets;  // [nseg + 1]
  const int32_t* tile_prefix;  // [nseg + 1]: 128-row tiles of the segments before s; [nseg] = all
  const int32_t* row_src;      // [R]
  int nseg, Hr, Kr;
  int a_rows;                  // rows of the gathered tensor (tokens for QKV, token slots for OUT)
  int kdim;                    // contraction length: d_model (QKV) or g d (OUT)
  int ncols;                   // output columns per group: (g + 2) d (QKV) or d_model (OUT)
  int g, d;
  uint16_t *q, *k, *v;         // QKV outputs
  float* o;                    // OUT output [ntok, d_model]
  int ntok;
  int out_aligned32;           // q, k, v 32-byte aligned: whole-sector stores
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

// Item -> (segment, rows, column tile).  The segment is the last s with tile_prefix[s] <= the
// item's row tile (empty segments have no tiles, so the search passes over them).
__device__ __forceinline__ Tile decode_item(const Params& p, int item, int nt_count) {
  Tile t;
  const int mtg = item / nt_count;
  t.nt = item - mtg * nt_count;
  int lo = 0, hi = p.nseg;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (__ldg(p.tile_prefix + mid) <= mtg) lo = mid; else hi = mid;
  }
  t.seg = lo;
  t.row0 = __ldg(p.seg_offsets + lo) + (mtg - __ldg(p.tile_prefix + lo)) * BM;
  t.rows = min(BM, __ldg(p.seg_offsets + lo + 1) - t.row0);
  t.hr = lo % p.Hr;
  return t;
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, uint32_t* status) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status);
  return __all_sync(0xffffffffu, ok);
}

// Four rows (y0..y3) x 64 columns from x into shared memory, 128-byte swizzled like a 4-row
// box of the same tensor map (its box is one row high).
__device__ __forceinline__ void tma_gather4(void* smem_dst, const CUtensorMap* map, int32_t x, int32_t y0, int32_t y1,
                                            int32_t y2, int32_t y3, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile::gather4.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5, %6}], [%7];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y0), "r"(y1), "r"(y2), "r"(y3), "r"(smem_u32(bar))
      : "memory");
}

// 128-row tiles of each segment, scanned: one block.
__global__ void __launch_bounds__(1024) tile_prefix_kernel(const int32_t* __restrict__ seg_offsets, int nseg,
                                                           int32_t* __restrict__ tile_prefix) {
  __shared__ int s_sum[1024];
  const int tid = threadIdx.x, nthr = blockDim.x;
  const int per = (nseg + nthr - 1) / nthr;
  const int s0 = min(nseg, tid * per), s1 = min(nseg, s0 + per);
  auto tiles = [&](int s) {
    const int n = __ldg(seg_offsets + s + 1) - __ldg(seg_offsets + s);
    return n > 0 ? (n + BM - 1) / BM : 0;
  };
  int sum = 0;
  for (int s = s0; s < s1; ++s) sum += tiles(s);
  s_sum[tid] = sum;
  __syncthreads();
  for (int off = 1; off < nthr; off <<= 1) {
    const int add = tid >= off ? s_sum[tid - off] : 0;
    __syncthreads();
    s_sum[tid] += add;
    __syncthreads();
  }
  int run = s_sum[tid] - sum;
  for (int s = s0; s < s1; ++s) {
    tile_prefix[s] = run;
    run += tiles(s);
  }
  if (tid == nthr - 1) tile_prefix[nseg] = s_sum[nthr - 1];
}

template <int BN, int kMode>
__global__ void __launch_bounds__(kThreads, 1) proj_kernel(const __grid_constant__ CUtensorMap tm_a,
                                                           const __grid_constant__ CUtensorMap tm_b, Params p) {
  using L = Layout<BN>;
  constexpr int S = L::kStages;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + L::kBar);
  volatile int* abort_flag = &bars->abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&bars->full[i], 1);
      mbar_init(&bars->empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->acc_full[i], 1);
      mbar_init(&bars->acc_empty[i], 4);
    }
    bars->abort_flag = 0;
    mbar_fence_init();
  }
  if (warp == 4 && lane == 0) {
    tma_prefetch_desc(&tm_a);
    tma_prefetch_desc(&tm_b);
  }
  if (warp == 5) {
    tmem_alloc(&bars->tmem_base, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  pdl_wait();  // the routing layout, the tile prefix and the inputs are visible from here

  const int nt_count = p.ncols / BN;
  const int nitems = __ldg(p.tile_prefix + p.nseg) * nt_count;
  const int nk = p.kdim / BK;

  if (warp == 4) {
    // ---- loads
    uint32_t it = 0;
    bool ok = true;
    for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
      const Tile t = decode_item(p, item, nt_count);
      int c[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int r = 4 * lane + e;
        int row = 0;  // rows past the segment's end load row 0; their outputs are not stored
        if (r < t.rows) {
          const int src = __ldg(p.row_src + t.row0 + r);
          row = kMode == kQKV ? src / p.Kr : src;
        }
        c[e] = min(max(row, 0), p.a_rows - 1);
      }
      const int b_row = t.hr * p.ncols + t.nt * BN;
      for (int kb = 0; kb < nk; ++kb, ++it) {
        const int slot = it % S;
        if (it >= (uint32_t)S && !warp_wait(&bars->empty[slot], ((it / S) - 1) & 1, abort_flag, p.status)) {
          ok = false;
          break;
        }
        uint8_t* a = smem + slot * L::kStage;
        if (lane == 0) mbar_arrive_expect_tx(&bars->full[slot], L::kStage);
        __syncwarp();
        tma_gather4(a + lane * 512, &tm_a, kb * BK, c[0], c[1], c[2], c[3], &bars->full[slot]);
        if (lane == 0) tma_load_2d(a + L::kA, &tm_b, kb * BK, b_row, &bars->full[slot]);
      }
    }
  } else if (warp == 5) {
    // ---- MMA issue
    constexpr uint32_t idesc = make_idesc_bf16(BM, BN, false, false);
    uint32_t it = 0;
    bool ok = true;
    int li = 0;
    for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x, ++li) {
      const int buf = li & 1;
      if (li >= 2 && !warp_wait(&bars->acc_empty[buf], ((li >> 1) - 1) & 1, abort_flag, p.status)) break;
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
#pragma unroll
        for (int kk = 0; kk < BK / 16; ++kk)
          mma_bf16_ss(d_tmem, a_desc + (uint64_t)(kk * 2), b_desc + (uint64_t)(kk * 2), idesc,
                      (kb | kk) ? 1u : 0u);
        mma_commit(&bars->empty[slot]);
      }
      if (ok) mma_commit(&bars->acc_full[buf]);
    }
  } else {
    // ---- epilogue: thread = tile row = TMEM lane
    const int row = warp * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    int li = 0;
    for (int item = blockIdx.x; item < nitems; item += gridDim.x, ++li) {
      const Tile t = decode_item(p, item, nt_count);
      const int buf = li & 1;
      const bool valid = row < t.rows;
      const int r = t.row0 + row;
      int src = valid ? __ldg(p.row_src + r) : 0;
      if (!warp_wait(&bars->acc_full[buf], (li >> 1) & 1, abort_flag, p.status)) break;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < BN / 32; ++c) {
        uint32_t v[32];
        tmem_ld32(tmem + lane_addr + buf * 256 + c * 32, v);
        tmem_wait_ld();
        if (!valid) continue;
        const int n = t.nt * BN + c * 32;  // first output column of the chunk
        if constexpr (kMode == kQKV) {
          uint16_t* dst;
          const int gd = p.g * p.d;
          if (n < gd) dst = p.q + ((long long)r * p.g + n / p.d) * p.d + n % p.d;
          else if (n < gd + p.d) dst = p.k + (long long)r * p.d + (n - gd);
          else dst = p.v + (long long)r * p.d + (n - gd - p.d);
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
        } else {
          const int tok = src / p.Kr;
          if (tok < 0 || tok >= p.ntok) continue;  // an inconsistent layout: nothing outside o
          float4* dst = reinterpret_cast<float4*>(p.o + (long long)tok * p.ncols + n);
#pragma unroll
          for (int e = 0; e < 8; ++e)
            atomicAdd(dst + e, make_float4(__uint_as_float(v[4 * e]), __uint_as_float(v[4 * e + 1]),
                                           __uint_as_float(v[4 * e + 2]), __uint_as_float(v[4 * e + 3])));
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->acc_empty[buf]);
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
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
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

template <int BN, int kMode>
cudaError_t launch_bn(const Params& p, const void* a, long long a_rows, const void* b, long long b_rows, int grid,
                      cudaStream_t stream) {
  CUtensorMap ta, tb;
  if (!encode_map(&ta, a, a_rows, p.kdim, 1) || !encode_map(&tb, b, b_rows, p.kdim, BN)) return cudaErrorInvalidValue;
  const int smem = Layout<BN>::kAlloc;
  cudaError_t e = cudaFuncSetAttribute(proj_kernel<BN, kMode>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(proj_kernel<BN, kMode>, dim3(grid), dim3(kThreads), (size_t)smem, stream, ta, tb, p);
}

// The widest column tile (multiple of 32, at most 256) that divides the output columns.
int pick_bn(int ncols) {
  for (int bn : {256, 192, 160, 128, 96, 64})
    if (ncols % bn == 0) return bn;
  return 0;
}

template <int kMode>
cudaError_t launch(int bn, const Params& p, const void* a, long long a_rows, const void* b, long long b_rows,
                   int grid, cudaStream_t stream) {
  switch (bn) {
    case 256: return launch_bn<256, kMode>(p, a, a_rows, b, b_rows, grid, stream);
    case 192: return launch_bn<192, kMode>(p, a, a_rows, b, b_rows, grid, stream);
    case 160: return launch_bn<160, kMode>(p, a, a_rows, b, b_rows, grid, stream);
    case 128: return launch_bn<128, kMode>(p, a, a_rows, b, b_rows, grid, stream);
    case 96: return launch_bn<96, kMode>(p, a, a_rows, b, b_rows, grid, stream);
    default: return launch_bn<64, kMode>(p, a, a_rows, b, b_rows, grid, stream);
  }
}

// Shapes shared by both projections: R = total_tokens * Kr packed rows in B * Hr segments.
int check_common(int B, int total_tokens, int d_model, int H, int K, int d_head, int group, int* Hr, int* Kr) {
  if (B < 1 || total_tokens < 1 || group < 1 || H < 1 || K < 1 || K > H || H % group || K % group)
    return NAMOH_ERR_INVALID_ARG;
  if (H / group > NAMOH_MAX_HEADS || (long long)B * (H / group) >= (1ll << 24)) return NAMOH_ERR_INVALID_ARG;
  if ((d_head != 64 && d_head != 128) || (group & (group - 1)) || group > 8) return NAMOH_ERR_UNSUPPORTED;
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

extern "C" size_t namoh_proj_workspace_size(int B, int H, int K, int group) {
  if (B < 1 || group < 1 || H < 1 || K < 1 || H % group) return 0;
  return align_up((size_t)(B * (H / group) + 1) * sizeof(int32_t), 256);
}

namespace {
int proj_prologue(const int32_t* seg_offsets, int nseg, void* workspace, size_t workspace_bytes, int32_t** prefix,
                  cudaStream_t stream) {
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  if (workspace_bytes < (size_t)(nseg + 1) * sizeof(int32_t)) return NAMOH_ERR_WORKSPACE;
  *prefix = static_cast<int32_t*>(workspace);
  proj::tile_prefix_kernel<<<1, 1024, 0, stream>>>(seg_offsets, nseg, *prefix);
  return cuda_check_launch("tile_prefix_kernel launch");
}
}  // namespace

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
  int32_t* prefix = nullptr;
  st = proj_prologue(seg_offsets, nseg, workspace, workspace_bytes, &prefix, stream);
  if (st != NAMOH_OK) return st;
  proj::Params p{};
  p.seg_offsets = seg_offsets;
  p.tile_prefix = prefix;
  p.row_src = row_src;
  p.nseg = nseg;
  p.Hr = Hr;
  p.Kr = Kr;
  p.a_rows = total_tokens;
  p.kdim = d_model;
  p.ncols = ncols;
  p.g = group;
  p.d = d_head;
  p.q = q;
  p.k = k;
  p.v = v;
  p.ntok = total_tokens;
  p.out_aligned32 = ((reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k) |
                      reinterpret_cast<uintptr_t>(v)) & 31u) == 0;
  p.status = dev_status;
  const cudaError_t e = proj::launch<proj::kQKV>(bn, p, x, total_tokens, w_qkv, (long long)Hr * ncols,
                                                 info.sm_count, stream);
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
  if (bn == 0) return NAMOH_ERR_UNSUPPORTED;
  DeviceInfo info;
  if (!current_device_info(&info) || info.major != 10) return NAMOH_ERR_UNSUPPORTED;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  if (!accumulate) {
    const cudaError_t e = cudaMemsetAsync(o, 0, (size_t)total_tokens * d_model * sizeof(float), stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaMemsetAsync of o");
  }
  const int nseg = B * Hr;
  int32_t* prefix = nullptr;
  st = proj_prologue(seg_offsets, nseg, workspace, workspace_bytes, &prefix, stream);
  if (st != NAMOH_OK) return st;
  proj::Params p{};
  p.seg_offsets = seg_offsets;
  p.tile_prefix = prefix;
  p.row_src = row_src;
  p.nseg = nseg;
  p.Hr = Hr;
  p.Kr = Kr;
  p.a_rows = total_tokens * Kr;
  p.kdim = group * d_head;
  p.ncols = d_model;
  p.g = group;
  p.d = d_head;
  p.o = o;
  p.ntok = total_tokens;
  p.status = dev_status;
  const cudaError_t e = proj::launch<proj::kOut>(bn, p, y, (long long)total_tokens * Kr, w_o, (long long)Hr * d_model,
                                                 info.sm_count, stream);
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, "proj_kernel (out) launch");
}
