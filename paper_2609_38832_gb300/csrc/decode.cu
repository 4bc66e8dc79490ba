// decode.cu -- one decode step over routed KV histories (Sec. 3.1 last paragraph; Sec. 3.2
// "Efficient execution": only the active heads' queries run and only their caches are read
// or updated; App. B.7 "Adopted KV-group routing" for g > 1).
//
// Three launches:
//   1. decode_append_kernel  one warp per (sequence, slot): rho = seg_len[s]; k~ = k R(p)
//                            and v are written at cache row seg_base[s] + rho; the g queries
//                            are rotated to p (kept in fp32 in the workspace).  p is rho, or
//                            the token's index in its sequence under global RoPE (Sec. 3.2);
//                            pairs (j, j + D/2), or (2j, 2j + 1) when interleaved.
//   2. decode_split_kernel   grid (splits, pairs): each CTA streams a contiguous range of the
//                            pair's rho + 1 cache rows.  A half-warp owns one row at a time
//                            (16 lanes x 16-byte loads = 256 bytes = one bf16 row of d = 128)
//                            and keeps 4 rows of K~ and V in flight; online softmax in fp32.
//                            Half-warp partials are merged in shared memory and the CTA writes
//                            (max, sum, acc[d]) per query head.
//   3. decode_merge_kernel   merges the splits, writes y = gate * h (bf16) and sets
//                            seg_len[s] = rho + 1.
// A full segment (or one whose next row would fall outside the cache) sets
// NAMOH_DEV_CAPACITY; its y is zero and its length is unchanged.
#include <float.h>

#include "common.cuh"

namespace namoh {
namespace {

constexpr int kMaxSplits = 64;
constexpr int kSplitThreads = 256;
constexpr int kRowsInFlight = 4;

struct PairInfo {
  long long base;  // first cache row attended over
  int len;         // rows to attend over (rho + 1, or the last `window` of them), 0 if the append was refused
  int seg;
  int new_len;     // the segment's length after the append (rho + 1)
};

template <int D>
__global__ void decode_append_kernel(const int32_t* __restrict__ topk_head, const uint16_t* __restrict__ q,
                                     const uint16_t* __restrict__ k, const uint16_t* __restrict__ v, int Hr, int Kr,
                                     int g, uint16_t* __restrict__ k_cache, uint16_t* __restrict__ v_cache,
                                     const int64_t* __restrict__ seg_base, const int32_t* __restrict__ seg_len,
                                     const int32_t* __restrict__ seg_cap, long long cache_rows, RopeTable tab,
                                     float* __restrict__ q_rot, PairInfo* __restrict__ info,
                                     uint32_t* __restrict__ status, const int64_t* __restrict__ token_pos,
                                     int interleaved, int window) {
  constexpr int HALF = D / 2;
  const int pair = blockIdx.x;  // b * Kr + slot
  const int b = pair / Kr;
  const int lane = threadIdx.x;
  const int h = topk_head[pair];
  const int s = b * Hr + h;
  const int rho = seg_len[s];
  const long long base = seg_base[s];
  const bool room = rho >= 0 && rho < seg_cap[s] && base + rho < cache_rows && base >= 0;
  if (lane == 0) {
    // a sliding window attends over the last `window` rows, the new one included
    const int first = (window > 0 && rho + 1 > window) ? rho + 1 - window : 0;
    PairInfo pi;
    pi.base = base + first;
    pi.len = room ? rho + 1 - first : 0;
    pi.seg = s;
    pi.new_len = rho + 1;
    info[pair] = pi;
    if (!room) report(status, NAMOH_DEV_CAPACITY);
  }
  if (!room) return;
  const long long dst = base + rho;
  const float p = token_pos ? (float)token_pos[b] : (float)rho;
  for (int jj = lane; jj < HALF; jj += 32) {
    float sn, cs;
    rope_sincos(p, tab.theta_hi[jj], tab.theta_lo[jj], tab, &sn, &cs);
    const int i0 = interleaved ? 2 * jj : jj, i1 = interleaved ? 2 * jj + 1 : jj + HALF;
    {
      const uint16_t* kr = k + (size_t)pair * D;
      const float x0 = __uint_as_float((uint32_t)kr[i0] << 16);
      const float x1 = __uint_as_float((uint32_t)kr[i1] << 16);
      const __nv_bfloat16 o0 = __float2bfloat16_rn(fmaf(x0, cs, -x1 * sn));
      const __nv_bfloat16 o1 = __float2bfloat16_rn(fmaf(x1, cs, x0 * sn));
      k_cache[dst * D + i0] = *reinterpret_cast<const uint16_t*>(&o0);
      k_cache[dst * D + i1] = *reinterpret_cast<const uint16_t*>(&o1);
      v_cache[dst * D + i0] = v[(size_t)pair * D + i0];
      v_cache[dst * D + i1] = v[(size_t)pair * D + i1];
    }
    for (int j = 0; j < g; ++j) {
      const uint16_t* qr = q + ((size_t)pair * g + j) * D;
      const float x0 = __uint_as_float((uint32_t)qr[i0] << 16);
      const float x1 = __uint_as_float((uint32_t)qr[i1] << 16);
      float* out = q_rot + ((size_t)pair * g + j) * D;
      out[i0] = fmaf(x0, cs, -x1 * sn);
      out[i1] = fmaf(x1, cs, x0 * sn);
    }
  }
}

// Partials layout: [pair][split][j][D + 2] = acc[D], max, sum  (max in log2 units)
template <int D, int G>
__global__ void __launch_bounds__(kSplitThreads) decode_split_kernel(const uint16_t* __restrict__ k_cache,
                                                                     const uint16_t* __restrict__ v_cache,
                                                                     const float* __restrict__ q_rot,
                                                                     const PairInfo* __restrict__ info, int splits,
                                                                     float scale_log2, float* __restrict__ part) {
  constexpr int LPR = D / 8;              // lanes per row: 8 bf16 (16 bytes) per lane
  constexpr int NGROUPS = kSplitThreads / LPR;
  constexpr int NWARPS = kSplitThreads / 32;
  __shared__ float s_m[NWARPS][G];
  __shared__ float s_l[NWARPS][G];
  __shared__ float s_acc[NWARPS][G][D];

  const int z = blockIdx.x;
  const int pair = blockIdx.y;
  const PairInfo pi = info[pair];
  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int grp = tid / LPR;       // row group (half-warp for D = 128)
  const int li = tid % LPR;        // lane within the row group
  const int e0 = li * 8;           // first element owned

  const int len = pi.len;
  const int per = (len + splits - 1) / splits;
  const int r0 = min(len, z * per), r1 = min(len, r0 + per);

  float qv[G][8];
#pragma unroll
  for (int j = 0; j < G; ++j)
#pragma unroll
    for (int e = 0; e < 8; ++e) qv[j][e] = q_rot[((size_t)pair * G + j) * D + e0 + e] * scale_log2;

  float m[G], l[G], acc[G][8];
#pragma unroll
  for (int j = 0; j < G; ++j) {
    m[j] = -INFINITY;
    l[j] = 0.f;
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[j][e] = 0.f;
  }

  const uint4* kc = reinterpret_cast<const uint4*>(k_cache + (size_t)pi.base * D) + li;
  const uint4* vc = reinterpret_cast<const uint4*>(v_cache + (size_t)pi.base * D) + li;
  constexpr int STEP = NGROUPS * kRowsInFlight;
  for (int rb = r0; rb < r1; rb += STEP) {
    uint4 kr[kRowsInFlight], vr[kRowsInFlight];
    bool have[kRowsInFlight];
#pragma unroll
    for (int u = 0; u < kRowsInFlight; ++u) {
      const int r = rb + u * NGROUPS + grp;
      have[u] = r < r1;
      if (have[u]) {
        kr[u] = __ldg(kc + (size_t)r * (D / 8));
        vr[u] = __ldg(vc + (size_t)r * (D / 8));
      } else {
        kr[u] = make_uint4(0, 0, 0, 0);
        vr[u] = make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int j = 0; j < G; ++j) {
      float sc[kRowsInFlight];
#pragma unroll
      for (int u = 0; u < kRowsInFlight; ++u) {
        const uint32_t w[4] = {kr[u].x, kr[u].y, kr[u].z, kr[u].w};
        float d0 = 0.f;
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          d0 = fmaf(qv[j][2 * p], bf16_lo(w[p]), d0);
          d0 = fmaf(qv[j][2 * p + 1], bf16_hi(w[p]), d0);
        }
#pragma unroll
        for (int o = LPR / 2; o >= 1; o >>= 1) d0 += __shfl_xor_sync(0xffffffffu, d0, o);
        sc[u] = have[u] ? d0 : -INFINITY;
      }
      float mn = m[j];
#pragma unroll
      for (int u = 0; u < kRowsInFlight; ++u) mn = fmaxf(mn, sc[u]);
      const bool any = mn != -INFINITY;  // false when this group had no rows in the step
      const float corr = any ? fast_exp2(m[j] - mn) : 1.f;
      m[j] = mn;
      l[j] *= corr;
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[j][e] *= corr;
#pragma unroll
      for (int u = 0; u < kRowsInFlight; ++u) {
        const float pu = any ? fast_exp2(sc[u] - mn) : 0.f;
        l[j] += pu;
        const uint32_t w[4] = {vr[u].x, vr[u].y, vr[u].z, vr[u].w};
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          acc[j][2 * p] = fmaf(pu, bf16_lo(w[p]), acc[j][2 * p]);
          acc[j][2 * p + 1] = fmaf(pu, bf16_hi(w[p]), acc[j][2 * p + 1]);
        }
      }
    }
  }

  // merge the row groups of each warp (lanes li, li + LPR, ... own the same elements)
#pragma unroll
  for (int j = 0; j < G; ++j) {
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1) {
      const float mo = __shfl_xor_sync(0xffffffffu, m[j], o);
      const float lo = __shfl_xor_sync(0xffffffffu, l[j], o);
      const float M = fmaxf(m[j], mo);
      const float wa = (M == -INFINITY) ? 0.f : fast_exp2(m[j] - M);
      const float wb = (M == -INFINITY) ? 0.f : fast_exp2(mo - M);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const float ao = __shfl_xor_sync(0xffffffffu, acc[j][e], o);
        acc[j][e] = acc[j][e] * wa + ao * wb;
      }
      l[j] = l[j] * wa + lo * wb;
      m[j] = M;
    }
  }
  if (lane < LPR) {
#pragma unroll
    for (int j = 0; j < G; ++j) {
      if (lane == 0) {
        s_m[warp][j] = m[j];
        s_l[warp][j] = l[j];
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) s_acc[warp][j][e0 + e] = acc[j][e];
    }
  }
  __syncthreads();
  float* out = part + ((size_t)pair * kMaxSplits + z) * G * (D + 2);
  for (int idx = tid; idx < G * D; idx += kSplitThreads) {
    const int j = idx / D, d = idx % D;
    float M = -INFINITY;
    for (int w2 = 0; w2 < NWARPS; ++w2) M = fmaxf(M, s_m[w2][j]);
    float a = 0.f, ls = 0.f;
    if (M != -INFINITY) {
      for (int w2 = 0; w2 < NWARPS; ++w2) {
        const float w = fast_exp2(s_m[w2][j] - M);
        a = fmaf(w, s_acc[w2][j][d], a);
        ls = fmaf(w, s_l[w2][j], ls);
      }
    }
    out[j * (D + 2) + d] = a;
    if (d == 0) {
      out[j * (D + 2) + D] = M;
      out[j * (D + 2) + D + 1] = ls;
    }
  }
}

template <int D>
__global__ void decode_merge_kernel(const PairInfo* __restrict__ info, const float* __restrict__ gate,
                                    const float* __restrict__ part, int splits, int g, uint16_t* __restrict__ y,
                                    int32_t* __restrict__ seg_len) {
  const int pair = blockIdx.x;
  const PairInfo pi = info[pair];
  const float gt = gate[pair];
  for (int idx = threadIdx.x; idx < g * D; idx += blockDim.x) {
    const int j = idx / D, d = idx % D;
    float out = 0.f;
    if (pi.len > 0) {
      float M = -INFINITY;
      for (int z = 0; z < splits; ++z)
        M = fmaxf(M, part[(((size_t)pair * kMaxSplits + z) * g + j) * (D + 2) + D]);
      float a = 0.f, ls = 0.f;
      for (int z = 0; z < splits; ++z) {
        const float* pz = part + (((size_t)pair * kMaxSplits + z) * g + j) * (D + 2);
        const float mz = pz[D];
        if (mz == -INFINITY) continue;
        const float w = fast_exp2(mz - M);
        a = fmaf(w, pz[d], a);
        ls = fmaf(w, pz[D + 1], ls);
      }
      out = gt * a / ls;
    }
    const __nv_bfloat16 o = __float2bfloat16_rn(out);
    y[((size_t)pair * g + j) * D + d] = *reinterpret_cast<const uint16_t*>(&o);
  }
  if (threadIdx.x == 0 && pi.len > 0) seg_len[pi.seg] = pi.new_len;
}

struct DecodeWs {
  float* q_rot;
  PairInfo* info;
  float* part;
};
void carve_decode(WorkspaceCarver& ws, DecodeWs* out, int pairs, int g, int D) {
  out->q_rot = ws.take<float>((size_t)pairs * g * D);
  out->info = ws.take<PairInfo>((size_t)pairs);
  out->part = ws.take<float>((size_t)pairs * kMaxSplits * g * (D + 2));
}

template <int D, int G>
cudaError_t launch_split(const uint16_t* kc, const uint16_t* vc, const float* qr, const PairInfo* info, int pairs,
                         int sm_count, float scale_log2, float* part, cudaStream_t stream, int* splits_out) {
  int occ = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, decode_split_kernel<D, G>, kSplitThreads, 0);
  if (e != cudaSuccess) return e;
  if (occ < 1) occ = 1;
  int splits = (sm_count * occ) / pairs;
  splits = splits < 1 ? 1 : (splits > kMaxSplits ? kMaxSplits : splits);
  *splits_out = splits;
  decode_split_kernel<D, G><<<dim3(splits, pairs), kSplitThreads, 0, stream>>>(kc, vc, qr, info, splits, scale_log2,
                                                                               part);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_split_g(int g, const uint16_t* kc, const uint16_t* vc, const float* qr, const PairInfo* info,
                           int pairs, int sm_count, float scale_log2, float* part, cudaStream_t stream, int* splits) {
  switch (g) {
    case 1:
      return launch_split<D, 1>(kc, vc, qr, info, pairs, sm_count, scale_log2, part, stream, splits);
    case 2:
      return launch_split<D, 2>(kc, vc, qr, info, pairs, sm_count, scale_log2, part, stream, splits);
    case 4:
      return launch_split<D, 4>(kc, vc, qr, info, pairs, sm_count, scale_log2, part, stream, splits);
    default:
      return launch_split<D, 8>(kc, vc, qr, info, pairs, sm_count, scale_log2, part, stream, splits);
  }
}

bool decode_dims_ok(int d_head, int g) {
  return (d_head == 64 || d_head == 128) && (g == 1 || g == 2 || g == 4 || g == 8);
}

}  // namespace
}  // namespace namoh

using namespace namoh;

extern "C" size_t namoh_decode_workspace_size(int B, int H, int K, int d_head, int group) {
  if (B < 1 || group < 1 || H % group || K % group || !decode_dims_ok(d_head, group)) return 0;
  WorkspaceCarver ws{nullptr, 0, 0};
  DecodeWs dw;
  carve_decode(ws, &dw, B * (K / group), group, d_head);
  return align_up(ws.used, 256);
}

namespace namoh {
namespace {
// The body of namoh_decode_ex and namoh_shared_decode; window 0 attends over every row.
int decode_impl(const int32_t* topk_head, const float* gate, const uint16_t* q, const uint16_t* k, const uint16_t* v,
                int B, int H, int K, int d_head, int group, float rope_base, unsigned rope_flags,
                const int64_t* token_pos, int window, uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base,
                int32_t* seg_len, const int32_t* seg_cap, int64_t cache_rows, uint16_t* y, void* workspace,
                size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!topk_head || !gate || !q || !k || !v || !k_cache || !v_cache || !seg_base || !seg_len || !seg_cap || !y ||
      !dev_status)
    return NAMOH_ERR_INVALID_ARG;
  if (B < 1 || group < 1 || H < 1 || K < 1 || K > H || H % group || K % group) return NAMOH_ERR_INVALID_ARG;
  if (H / group > NAMOH_MAX_HEADS || cache_rows < 1 || cache_rows >= (1ll << 40)) return NAMOH_ERR_INVALID_ARG;
  if (!(rope_base > 1.0f) || !isfinite(rope_base)) return NAMOH_ERR_INVALID_ARG;
  if (!rope_flags_ok(rope_flags) || ((rope_flags & NAMOH_ROPE_GLOBAL) != 0) != (token_pos != nullptr))
    return NAMOH_ERR_INVALID_ARG;
  if (!decode_dims_ok(d_head, group)) return NAMOH_ERR_UNSUPPORTED;
  if (!aligned16(k_cache) || !aligned16(v_cache) || !aligned16(q) || !aligned16(y)) return NAMOH_ERR_INVALID_ARG;
  const int D = d_head, g = group, Hr = H / g, Kr = K / g;
  const int pairs = B * Kr;
  if ((long long)B * Kr >= (1 << 30)) return NAMOH_ERR_INVALID_ARG;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
  DecodeWs dw;
  carve_decode(ws, &dw, pairs, g, D);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  DeviceInfo info;
  if (!current_device_info(&info)) return cuda_fail(cudaGetLastError(), "device query");
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);

  RopeTable tab;
  fill_rope_table(&tab, D, (double)rope_base);
  const int interleaved = (rope_flags & NAMOH_ROPE_INTERLEAVED) ? 1 : 0;
  if (D == 128)
    decode_append_kernel<128><<<pairs, 32, 0, stream>>>(topk_head, q, k, v, Hr, Kr, g, k_cache, v_cache, seg_base,
                                                        seg_len, seg_cap, cache_rows, tab, dw.q_rot, dw.info,
                                                        dev_status, token_pos, interleaved, window);
  else
    decode_append_kernel<64><<<pairs, 32, 0, stream>>>(topk_head, q, k, v, Hr, Kr, g, k_cache, v_cache, seg_base,
                                                       seg_len, seg_cap, cache_rows, tab, dw.q_rot, dw.info,
                                                       dev_status, token_pos, interleaved, window);
  if (const int st = cuda_check_launch("decode_append_kernel launch")) return st;

  const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)D));
  int splits = 1;
  cudaError_t e = (D == 128) ? launch_split_g<128>(g, k_cache, v_cache, dw.q_rot, dw.info, pairs, info.sm_count,
                                                   scale_log2, dw.part, stream, &splits)
                             : launch_split_g<64>(g, k_cache, v_cache, dw.q_rot, dw.info, pairs, info.sm_count,
                                                  scale_log2, dw.part, stream, &splits);
  if (e != cudaSuccess) return cuda_fail(e, "decode_split_kernel launch");
  const int mthreads = g * D < 1024 ? g * D : 1024;
  if (D == 128)
    decode_merge_kernel<128><<<pairs, mthreads, 0, stream>>>(dw.info, gate, dw.part, splits, g, y, seg_len);
  else
    decode_merge_kernel<64><<<pairs, mthreads, 0, stream>>>(dw.info, gate, dw.part, splits, g, y, seg_len);
  if (const int st = cuda_check_launch("decode_merge_kernel launch")) return st;
  return NAMOH_OK;
}

__global__ void all_heads_kernel(int B, int Hs, int32_t* __restrict__ topk_head, float* __restrict__ gate) {
  for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < B * Hs; i += gridDim.x * blockDim.x) {
    topk_head[i] = i % Hs;
    gate[i] = 1.f;
  }
}
}  // namespace
}  // namespace namoh

extern "C" int namoh_decode_ex(const int32_t* topk_head, const float* gate, const uint16_t* q, const uint16_t* k,
                               const uint16_t* v, int B, int H, int K, int d_head, int group, float rope_base,
                               unsigned rope_flags, const int64_t* token_pos, uint16_t* k_cache, uint16_t* v_cache,
                               const int64_t* seg_base, int32_t* seg_len, const int32_t* seg_cap, int64_t cache_rows,
                               uint16_t* y, void* workspace, size_t workspace_bytes, uint32_t* dev_status,
                               void* stream_v) {
  return decode_impl(topk_head, gate, q, k, v, B, H, K, d_head, group, rope_base, rope_flags, token_pos, 0, k_cache,
                     v_cache, seg_base, seg_len, seg_cap, cache_rows, y, workspace, workspace_bytes, dev_status,
                     stream_v);
}

extern "C" size_t namoh_shared_decode_workspace_size(int B, int Hs, int d_head) {
  const size_t base = namoh_decode_workspace_size(B, Hs, Hs, d_head, 1);
  if (base == 0) return 0;
  return base + align_up((size_t)B * Hs * sizeof(int32_t), 256) + align_up((size_t)B * Hs * sizeof(float), 256);
}

extern "C" int namoh_shared_decode(const uint16_t* q, const uint16_t* k, const uint16_t* v, int B, int Hs, int d_head,
                                   int window, float rope_base, unsigned rope_flags, uint16_t* k_cache,
                                   uint16_t* v_cache, const int64_t* seg_base, int32_t* seg_len,
                                   const int32_t* seg_cap, int64_t cache_rows, uint16_t* y, void* workspace,
                                   size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (window < 0 || (rope_flags & NAMOH_ROPE_GLOBAL)) return NAMOH_ERR_INVALID_ARG;
  const size_t need = namoh_shared_decode_workspace_size(B, Hs, d_head);
  if (need == 0) return NAMOH_ERR_INVALID_ARG;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u) || workspace_bytes < need)
    return NAMOH_ERR_WORKSPACE;
  const size_t base = namoh_decode_workspace_size(B, Hs, Hs, d_head, 1);
  int32_t* topk = reinterpret_cast<int32_t*>(static_cast<char*>(workspace) + base);
  float* gate = reinterpret_cast<float*>(static_cast<char*>(workspace) + base +
                                         align_up((size_t)B * Hs * sizeof(int32_t), 256));
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  all_heads_kernel<<<(B * Hs + 255) / 256, 256, 0, stream>>>(B, Hs, topk, gate);
  if (const int st = cuda_check_launch("all_heads_kernel launch")) return st;
  // positions: the rank (every token of a shared head is in its segment, so the rank is t)
  return decode_impl(topk, gate, q, k, v, B, Hs, Hs, d_head, 1, rope_base, rope_flags, nullptr, window, k_cache,
                     v_cache, seg_base, seg_len, seg_cap, cache_rows, y, workspace, base, dev_status, stream_v);
}

extern "C" int namoh_decode(const int32_t* topk_head, const float* gate, const uint16_t* q, const uint16_t* k,
                            const uint16_t* v, int B, int H, int K, int d_head, int group, float rope_base,
                            uint16_t* k_cache, uint16_t* v_cache, const int64_t* seg_base, int32_t* seg_len,
                            const int32_t* seg_cap, int64_t cache_rows, uint16_t* y, void* workspace,
                            size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  return namoh_decode_ex(topk_head, gate, q, k, v, B, H, K, d_head, group, rope_base, 0u, nullptr, k_cache, v_cache,
                         seg_base, seg_len, seg_cap, cache_rows, y, workspace, workspace_bytes, dev_status, stream_v);
}
