// route.cu -- routing and dispatch (Sec. 3.1 Eq. namoh-gates; Sec. 3.2 Eq. namoh-head-rope).
//
// Three launches, all stream-ordered, no host synchronisation:
//   1. route_topk_kernel   one thread per token: TopK of the fp32 logits (descending,
//                          ties to the lower head index), fp32 softmax gates over all H,
//                          and per-chunk head counts (one block = one 256-token chunk).
//   2. route_scan_kernel   one block per sequence: exclusive scan of the chunk counts over
//                          chunks for every head -> chunk base ranks and totals n[b, h];
//                          the last block to finish scans n over (b, h) -> seg_offsets.
//   3. route_rank_kernel   per chunk: warp ballots give each (token, slot) its rank among
//                          the chunk's earlier tokens for that head; adds the chunk base
//                          -> rank, row and row_src.
// All integer work is exact, so the packed layout is deterministic and bit-identical to
// a sequential append in token order.
#include <float.h>

#include "common.cuh"

namespace namoh {
namespace {

constexpr int kChunk = 256;  // tokens per block in the top-K and rank kernels

template <int HMAX>
__global__ void __launch_bounds__(kChunk) route_topk_kernel(const float* __restrict__ scores, int T, int H, int K,
                                                            int nchunks, int32_t* __restrict__ topk_head,
                                                            float* __restrict__ gate,
                                                            int32_t* __restrict__ chunk_count,
                                                            int* __restrict__ scan_ticket,
                                                            uint32_t* __restrict__ status) {
  __shared__ int s_cnt[NAMOH_MAX_HEADS];
  __shared__ int s_bad;
  const int c = blockIdx.x;
  const int b = blockIdx.y;
  const int tid = threadIdx.x;
  const int t = c * kChunk + tid;
  if (tid < NAMOH_MAX_HEADS) s_cnt[tid] = 0;
  if (tid == 0) s_bad = 0;
  if (scan_ticket && b == 0 && c == 0 && tid == 0) *scan_ticket = 0;  // consumed by route_scan_kernel
  __syncthreads();

  if (t < T) {
    // this token's H logits: independent loads, all in flight together
    const size_t tok = (size_t)b * T + t;
    const float* src = scores + tok * H;
    float sc[HMAX];
    if ((H & 3) == 0 && (reinterpret_cast<uintptr_t>(src) & 15u) == 0) {
#pragma unroll
      for (int h4 = 0; h4 < HMAX / 4; ++h4) {
        float4 x = make_float4(0.f, 0.f, 0.f, 0.f);
        if (h4 * 4 < H) x = __ldg(reinterpret_cast<const float4*>(src) + h4);
        sc[4 * h4 + 0] = x.x;
        sc[4 * h4 + 1] = x.y;
        sc[4 * h4 + 2] = x.z;
        sc[4 * h4 + 3] = x.w;
      }
    } else {
#pragma unroll
      for (int h = 0; h < HMAX; ++h) sc[h] = (h < H) ? __ldg(src + h) : 0.f;
    }
    bool bad = false;
#pragma unroll
    for (int h = 0; h < HMAX; ++h) {
      if (h < H && !isfinite(sc[h])) {
        bad = true;
        sc[h] = -FLT_MAX;
      }
    }
    // softmax denominator over all H logits (fp32); pairwise partial maxima / sums
    float mx = -FLT_MAX;
#pragma unroll
    for (int h = 0; h < HMAX; ++h)
      if (h < H) mx = fmaxf(mx, sc[h]);
    float z0 = 0.f, z1 = 0.f;
#pragma unroll
    for (int h = 0; h < HMAX; h += 2) {
      if (h < H) z0 += expf(sc[h] - mx);
      if (h + 1 < H) z1 += expf(sc[h + 1] - mx);
    }
    const float inv_z = 1.0f / (z0 + z1);

    // K passes; pass k picks the best head strictly after the previous pick in the
    // total order (score desc, index asc).
    float pv = 0.f;
    int pi = -1;
    const size_t base = tok * K;
    for (int k = 0; k < K; ++k) {
      float bv = 0.f;
      int bi = -1;
#pragma unroll
      for (int h = 0; h < HMAX; ++h) {
        const float x = sc[h];
        const bool elig = (h < H) && (pi < 0 || x < pv || (x == pv && h > pi));
        const bool better = elig && (bi < 0 || x > bv);
        bv = better ? x : bv;
        bi = better ? h : bi;
      }
      topk_head[base + k] = bi;
      gate[base + k] = expf(bv - mx) * inv_z;
      if (chunk_count) atomicAdd(&s_cnt[bi], 1);
      pv = bv;
      pi = bi;
    }
    if (bad) s_bad = 1;
  }
  __syncthreads();
  if (chunk_count && tid < H) chunk_count[((size_t)b * nchunks + c) * H + tid] = s_cnt[tid];
  if (tid == 0 && s_bad) report(status, NAMOH_DEV_NONFINITE_SCORE);
}

// One block per sequence b: for every head, exclusive scan of the chunk counts over chunks
// (thread (h, p) owns the chunk range [p*per, (p+1)*per)) -> chunk bases and n[b, h].
// The last block to finish (ticket) scans n over (b, h) order into seg_offsets.
__global__ void __launch_bounds__(1024) route_scan_kernel(const int32_t* __restrict__ chunk_count, int B, int H,
                                                          int nchunks, int32_t* __restrict__ chunk_base,
                                                          int32_t* __restrict__ n_out, int* __restrict__ ticket,
                                                          int32_t* __restrict__ seg_offsets) {
  __shared__ int s_part[1024];
  __shared__ int s_last;
  const int b = blockIdx.x;
  const int tid = threadIdx.x;
  const int P = blockDim.x / H;  // parts per head (blockDim is a multiple of H)
  const int h = tid % H, p = tid / H;
  const int per = (nchunks + P - 1) / P;
  const int c0 = min(nchunks, p * per), c1 = min(nchunks, c0 + per);
  const int32_t* cc = chunk_count + (size_t)b * nchunks * H;
  int sum = 0;
  for (int c = c0; c < c1; ++c) sum += __ldg(cc + (size_t)c * H + h);
  s_part[tid] = sum;
  __syncthreads();
  int before = 0;
  for (int q = 0; q < p; ++q) before += s_part[q * H + h];
  int run = before;
  int32_t* out = chunk_base + (size_t)b * nchunks * H;
  for (int c = c0; c < c1; ++c) {
    out[(size_t)c * H + h] = run;
    run += __ldg(cc + (size_t)c * H + h);
  }
  if (p == P - 1) n_out[(size_t)b * H + h] = run;

  // the last sequence block to finish builds seg_offsets
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(ticket, 1) == B - 1);
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const int nseg = B * H;
  const volatile int32_t* nv = n_out;
  const int per2 = (nseg + blockDim.x - 1) / blockDim.x;
  const int i0 = min(nseg, tid * per2), i1 = min(nseg, i0 + per2);
  int s2 = 0;
  for (int i = i0; i < i1; ++i) s2 += nv[i];
  __syncthreads();
  s_part[tid] = s2;
  __syncthreads();
  for (int off = 1; off < (int)blockDim.x; off <<= 1) {  // Hillis-Steele inclusive scan
    const int v = (tid >= off) ? s_part[tid - off] : 0;
    __syncthreads();
    s_part[tid] += v;
    __syncthreads();
  }
  int r2 = s_part[tid] - s2;
  for (int i = i0; i < i1; ++i) {
    seg_offsets[i] = r2;
    r2 += nv[i];
  }
  if (tid == blockDim.x - 1) seg_offsets[nseg] = s_part[tid];
}

// Per chunk: rank = chunk base + rank among this chunk's earlier tokens for the head.
__global__ void __launch_bounds__(kChunk) route_rank_kernel(const int32_t* __restrict__ topk_head, int T, int H,
                                                            int K, int nchunks,
                                                            const int32_t* __restrict__ chunk_base,
                                                            const int32_t* __restrict__ seg_offsets,
                                                            int32_t* __restrict__ rank, int32_t* __restrict__ row,
                                                            int32_t* __restrict__ row_src) {
  __shared__ uint32_t s_bal[kChunk / 32][NAMOH_MAX_HEADS];
  __shared__ int s_wbase[kChunk / 32][NAMOH_MAX_HEADS];
  __shared__ int s_cbase[NAMOH_MAX_HEADS];  // rank of the chunk's first token for each head
  __shared__ int s_soff[NAMOH_MAX_HEADS];   // segment offset of each head in this sequence
  const int c = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int t = c * kChunk + tid;
  const bool valid = t < T;
  const size_t tok = (size_t)b * T + t;
  if (tid < H) {
    s_cbase[tid] = chunk_base[((size_t)b * nchunks + c) * H + tid];
    s_soff[tid] = seg_offsets[(size_t)b * H + tid];
  }
  uint64_t mask = 0;
  if (valid)
    for (int k = 0; k < K; ++k) mask |= 1ull << topk_head[tok * K + k];
  for (int h = 0; h < H; ++h) {
    const uint32_t bal = __ballot_sync(0xffffffffu, (mask >> h) & 1ull);
    if (lane == 0) s_bal[warp][h] = bal;
  }
  __syncthreads();
  for (int i = tid; i < (kChunk / 32) * H; i += kChunk) {
    const int w = i / H, h = i % H;
    int before = 0;
    for (int q = 0; q < w; ++q) before += __popc(s_bal[q][h]);
    s_wbase[w][h] = before;
  }
  __syncthreads();
  if (!valid) return;
  const uint32_t lt = (1u << lane) - 1u;
  for (int k = 0; k < K; ++k) {
    const int h = topk_head[tok * K + k];
    const int rho = s_cbase[h] + s_wbase[warp][h] + __popc(s_bal[warp][h] & lt);
    const int r = s_soff[h] + rho;
    rank[tok * K + k] = rho;
    row[tok * K + k] = r;
    row_src[r] = (int32_t)(tok * K + k);
  }
}

template <int HMAX>
cudaError_t launch_topk(const float* scores, int B, int T, int H, int K, int nchunks, int32_t* topk, float* gate,
                        int32_t* chunk_count, int* ticket, uint32_t* status, cudaStream_t stream) {
  dim3 grid(nchunks, B);
  route_topk_kernel<HMAX><<<grid, kChunk, 0, stream>>>(scores, T, H, K, nchunks, topk, gate, chunk_count, ticket,
                                                       status);
  return cudaGetLastError();
}

}  // namespace
}  // namespace namoh

using namespace namoh;

extern "C" size_t namoh_route_workspace_size(int B, int T, int H, int K) {
  if (B < 1 || T < 1 || H < 1 || K < 1) return 0;
  const size_t nchunks = ((size_t)T + kChunk - 1) / kChunk;
  WorkspaceCarver ws{nullptr, 0, 0};
  ws.take<int32_t>((size_t)B * nchunks * H);  // chunk counts
  ws.take<int32_t>((size_t)B * nchunks * H);  // chunk bases
  ws.take<int32_t>((size_t)B * H);            // n
  ws.take<int>(1);                            // scan ticket
  return align_up(ws.used, 256);
}

extern "C" int namoh_route(const float* scores, int B, int T, int H, int K, int32_t* topk_head, float* gate,
                           int32_t* rank, int32_t* row, int32_t* seg_offsets, int32_t* row_src, void* workspace,
                           size_t workspace_bytes, uint32_t* dev_status, void* stream_v) {
  if (!scores || !topk_head || !gate || !dev_status) return NAMOH_ERR_INVALID_ARG;
  if (B < 1 || T < 1 || H < 1 || K < 1 || K > H || H > NAMOH_MAX_HEADS) return NAMOH_ERR_INVALID_ARG;
  if ((long long)B * T * K >= (1ll << 31) || (long long)B * H >= (1ll << 20)) return NAMOH_ERR_INVALID_ARG;
  const bool compact = seg_offsets != nullptr;
  if (compact != (rank != nullptr) || compact != (row != nullptr) || compact != (row_src != nullptr))
    return NAMOH_ERR_INVALID_ARG;
  cudaStream_t stream = reinterpret_cast<cudaStream_t>(stream_v);
  const int nchunks = (T + kChunk - 1) / kChunk;

  int32_t* chunk_count = nullptr;
  int32_t* chunk_base = nullptr;
  int32_t* n = nullptr;
  int* ticket = nullptr;
  if (compact) {
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
    WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
    chunk_count = ws.take<int32_t>((size_t)B * nchunks * H);
    chunk_base = ws.take<int32_t>((size_t)B * nchunks * H);
    n = ws.take<int32_t>((size_t)B * H);
    ticket = ws.take<int>(1);
    if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  }

  cudaError_t e;
  if (H <= 8)
    e = launch_topk<8>(scores, B, T, H, K, nchunks, topk_head, gate, chunk_count, ticket, dev_status, stream);
  else if (H <= 16)
    e = launch_topk<16>(scores, B, T, H, K, nchunks, topk_head, gate, chunk_count, ticket, dev_status, stream);
  else if (H <= 32)
    e = launch_topk<32>(scores, B, T, H, K, nchunks, topk_head, gate, chunk_count, ticket, dev_status, stream);
  else
    e = launch_topk<64>(scores, B, T, H, K, nchunks, topk_head, gate, chunk_count, ticket, dev_status, stream);
  if (e != cudaSuccess) return cuda_fail(e, "route_topk_kernel launch");
  if (!compact) return NAMOH_OK;

  const int scan_threads = 1024 - (1024 % H);
  route_scan_kernel<<<B, scan_threads, 0, stream>>>(chunk_count, B, H, nchunks, chunk_base, n, ticket, seg_offsets);
  if (const int st = cuda_check_launch("route_scan_kernel launch")) return st;
  route_rank_kernel<<<dim3(nchunks, B), kChunk, 0, stream>>>(topk_head, T, H, K, nchunks, chunk_base, seg_offsets,
                                                             rank, row, row_src);
  if (const int st = cuda_check_launch("route_rank_kernel launch")) return st;
  return NAMOH_OK;
}

// ---------------------------------------------------------------------------
// Routing with built-in scratch (no caller workspace, no allocation).
// The scratch is a file-scope device array; host code only ever passes the
// device address obtained from cudaGetSymbolAddress, never the array's name.
// ---------------------------------------------------------------------------
#include <mutex>

namespace namoh {
namespace {
constexpr size_t kRouteStaticScratchBytes = 4u << 20;  // 4 MiB on every device that loads the library
static __device__ __align__(256) unsigned char g_route_scratch[kRouteStaticScratchBytes];

constexpr int kMaxScratchDevices = 64;
std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxScratchDevices] = {};

// Device address of g_route_scratch on the current device (resolved once per device).
void* route_scratch_address() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxScratchDevices) return nullptr;
  std::lock_guard<std::mutex> lock(g_scratch_mutex);
  if (!g_scratch_addr[dev]) {
    void* ptr = nullptr;
    if (cudaGetSymbolAddress(&ptr, g_route_scratch) != cudaSuccess) return nullptr;
    g_scratch_addr[dev] = ptr;
  }
  return g_scratch_addr[dev];
}
}  // namespace
}  // namespace namoh

extern "C" int namoh_route_noalloc(const float* scores, int B, int T, int H, int K, int32_t* topk_head, float* gate,
                                   int32_t* rank, int32_t* row, int32_t* seg_offsets, int32_t* row_src,
                                   uint32_t* dev_status, void* stream) {
  if (!scores || !topk_head || !gate || !dev_status) return NAMOH_ERR_INVALID_ARG;
  if (B < 1 || T < 1 || H < 1 || K < 1 || K > H || H > NAMOH_MAX_HEADS) return NAMOH_ERR_INVALID_ARG;
  if (seg_offsets && namoh_route_workspace_size(B, T, H, K) > kRouteStaticScratchBytes) return NAMOH_ERR_WORKSPACE;
  void* scratch = route_scratch_address();
  if (!scratch) return cuda_fail(cudaErrorInvalidSymbol, "cudaGetSymbolAddress of the routing scratch");
  return namoh_route(scores, B, T, H, K, topk_head, gate, rank, row, seg_offsets, row_src, scratch,
                     kRouteStaticScratchBytes, dev_status, stream);
}
