// rope_pack.cu -- head-relative RoPE at the packed rank (Sec. 3.2, Eq. namoh-head-rope).
//
// One group of D/16 threads per packed row r: the row's segment s is found by binary
// search over seg_offsets, rho = r - seg_offsets[s].  Each thread owns 8 rotation pairs
// (j, j + D/2) and moves them with 16-byte loads/stores.  The angle is computed once per
// row and applied to K and to all g query heads of the row (KV-group routing shares the
// rank, App. C).  Outputs: Q~ (bf16 scratch for the attention kernel), K~ into the key
// cache, and V copied into the value cache unless the caller passed v_cache == v.  When
// given a plan buffer, one extra block builds the attention work list in the same launch.
#include "common.cuh"
#include "plan.cuh"

namespace namoh {

constexpr int kRopeStageMax = 8192;  // seg_offsets entries staged in shared memory (32 KB)

// With a plan header given, block 0 builds the attention work list (it depends only on
// seg_offsets) while the other blocks rotate rows; it goes first so that it is resident in
// the first wave.
template <int D, int G>
__global__ void __launch_bounds__(256) rope_pack_kernel(const uint16_t* __restrict__ q, const uint16_t* __restrict__ k,
                                                        const uint16_t* __restrict__ v, int R,
                                                        const int32_t* __restrict__ seg_offsets, int nseg,
                                                        const int64_t* __restrict__ seg_base,
                                                        const int32_t* __restrict__ seg_cap, long long cache_rows,
                                                        uint16_t* __restrict__ q_rot, uint16_t* __restrict__ k_cache,
                                                        uint16_t* __restrict__ v_cache, int copy_v, RopeTable tab,
                                                        uint32_t* __restrict__ status, int* __restrict__ plan_header,
                                                        int2* __restrict__ plan_items, const int32_t* __restrict__ plan_cap,
                                                        int plan_qtiles) {
  constexpr int LPR = D / 16;  // threads per row
  constexpr int HALF = D / 2;
  extern __shared__ int32_t s_dyn[];
  const int first = plan_header ? 1 : 0;
  if ((int)blockIdx.x < first) {
    build_plan(seg_offsets, nseg, plan_cap, G, plan_qtiles, plan_header, plan_items, s_dyn);
    return;
  }
  const int rope_blocks = gridDim.x - first;
  const int block = blockIdx.x - first;
  const bool staged = (nseg + 1) <= kRopeStageMax;
  if (staged) {
    for (int i = threadIdx.x; i <= nseg; i += blockDim.x) s_dyn[i] = __ldg(seg_offsets + i);
    __syncthreads();
  }
  const int32_t* offs = staged ? s_dyn : seg_offsets;
  const int lane_in_row = threadIdx.x % LPR;
  const int j0 = lane_in_row * 8;
  const long long groups = (long long)rope_blocks * (blockDim.x / LPR);
  float th_hi[8], th_lo[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    th_hi[i] = tab.theta_hi[j0 + i];
    th_lo[i] = tab.theta_lo[j0 + i];
  }
  for (long long r = (long long)block * (blockDim.x / LPR) + threadIdx.x / LPR; r < R; r += groups) {
    // every load of this row first, so their latencies overlap
    const uint4 ka = __ldg(reinterpret_cast<const uint4*>(k + (size_t)r * D + j0));
    const uint4 kb = __ldg(reinterpret_cast<const uint4*>(k + (size_t)r * D + HALF + j0));
    uint4 qa[G], qb[G];
#pragma unroll
    for (int j = 0; j < G; ++j) {
      qa[j] = __ldg(reinterpret_cast<const uint4*>(q + ((size_t)r * G + j) * D + j0));
      qb[j] = __ldg(reinterpret_cast<const uint4*>(q + ((size_t)r * G + j) * D + HALF + j0));
    }
    uint4 va = make_uint4(0, 0, 0, 0), vb = va;
    if (copy_v) {
      va = __ldg(reinterpret_cast<const uint4*>(v + (size_t)r * D) + lane_in_row);
      vb = __ldg(reinterpret_cast<const uint4*>(v + (size_t)r * D) + lane_in_row + LPR);
    }
    // segment of row r: last s with seg_offsets[s] <= r
    int lo = 0, hi = nseg;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (offs[mid] <= r) lo = mid; else hi = mid;
    }
    const int rho = (int)(r - offs[lo]);
    long long dst = r;
    bool write_cache = true;
    if (seg_base) {
      dst = __ldg(seg_base + lo) + rho;
      if (rho >= __ldg(seg_cap + lo) || dst < 0 || dst >= cache_rows) {
        write_cache = false;
        if (lane_in_row == 0) report(status, NAMOH_DEV_CAPACITY);
      }
    }
    float sn[8], cs[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) rope_sincos((float)rho, th_hi[i], th_lo[i], tab, &sn[i], &cs[i]);

    // x'_j = x_j cos - x_{j+D/2} sin ;  x'_{j+D/2} = x_{j+D/2} cos + x_j sin
    auto rotate = [&](const uint4& a, const uint4& b, uint16_t* dst_row) {
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
    };
#pragma unroll
    for (int j = 0; j < G; ++j) rotate(qa[j], qb[j], q_rot + ((size_t)r * G + j) * D);
    if (write_cache) {
      rotate(ka, kb, k_cache + (size_t)dst * D);
      if (copy_v) {
        uint4* vd = reinterpret_cast<uint4*>(v_cache + (size_t)dst * D);
        vd[lane_in_row] = va;
        vd[lane_in_row + LPR] = vb;
      }
    }
  }
}

template <int D>
cudaError_t launch_rope_pack_d(int g, dim3 grid, size_t smem, cudaStream_t stream, const uint16_t* q,
                               const uint16_t* k, const uint16_t* v, int R, const int32_t* seg_offsets, int nseg,
                               const int64_t* seg_base, const int32_t* seg_cap, long long cache_rows, uint16_t* q_rot,
                               uint16_t* k_cache, uint16_t* v_cache, int copy_v, const RopeTable& tab,
                               uint32_t* status, int* plan_header, int2* plan_items, const int32_t* plan_cap,
                               int plan_qtiles) {
  switch (g) {
#define NAMOH_ROPE_CASE(GG)                                                                                     \
  case GG:                                                                                                      \
    if (smem > 48 * 1024) {                                                                                     \
      cudaError_t e = cudaFuncSetAttribute(rope_pack_kernel<D, GG>, cudaFuncAttributeMaxDynamicSharedMemorySize, \
                                           (int)smem);                                                          \
      if (e != cudaSuccess) return e;                                                                           \
    }                                                                                                           \
    rope_pack_kernel<D, GG><<<grid, 256, smem, stream>>>(q, k, v, R, seg_offsets, nseg, seg_base, seg_cap,       \
                                                         cache_rows, q_rot, k_cache, v_cache, copy_v, tab, status, \
                                                         plan_header, plan_items, plan_cap, plan_qtiles);        \
    break;
    NAMOH_ROPE_CASE(1)
    NAMOH_ROPE_CASE(2)
    NAMOH_ROPE_CASE(4)
    NAMOH_ROPE_CASE(8)
#undef NAMOH_ROPE_CASE
    default:
      return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

cudaError_t launch_rope_pack(int D, const uint16_t* q, const uint16_t* k, const uint16_t* v, int R, int g,
                             const int32_t* seg_offsets, int nseg, const int64_t* seg_base, const int32_t* seg_cap,
                             long long cache_rows, uint16_t* q_rot, uint16_t* k_cache, uint16_t* v_cache, bool copy_v,
                             const RopeTable& tab, uint32_t* status, int sm_count, cudaStream_t stream,
                             void* plan, int plan_qtiles, const int32_t* plan_cap) {
  const int threads = 256;
  const int rows_per_block = threads / (D / 16);
  long long blocks = ((long long)R + rows_per_block - 1) / rows_per_block;
  const long long cap = (long long)sm_count * 8;
  if (blocks > cap) blocks = cap;
  int* plan_header = static_cast<int*>(plan);
  int2* plan_items = plan ? reinterpret_cast<int2*>(static_cast<char*>(plan) + 16) : nullptr;
  const long long grid = blocks + (plan ? 1 : 0);
  if (grid == 0) return cudaSuccess;
  size_t smem = (nseg + 1 <= kRopeStageMax) ? (size_t)(nseg + 1) * sizeof(int32_t) : 0;
  if (plan) {
    const size_t ps = (size_t)plan_smem_ints(plan_qtiles, nseg) * sizeof(int);
    if (ps > smem) smem = ps;
  }
  if (D == 128)
    return launch_rope_pack_d<128>(g, dim3((unsigned)grid), smem, stream, q, k, v, R, seg_offsets, nseg, seg_base,
                                   seg_cap, cache_rows, q_rot, k_cache, v_cache, copy_v ? 1 : 0, tab, status,
                                   plan_header, plan_items, plan_cap, plan_qtiles);
  return launch_rope_pack_d<64>(g, dim3((unsigned)grid), smem, stream, q, k, v, R, seg_offsets, nseg, seg_base,
                                seg_cap, cache_rows, q_rot, k_cache, v_cache, copy_v ? 1 : 0, tab, status,
                                plan_header, plan_items, plan_cap, plan_qtiles);
}

}  // namespace namoh
