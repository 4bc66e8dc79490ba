// route.cu -- routing and dispatch (Sec. 3.1 Eq. namoh-gates; Sec. 3.2 Eq. namoh-head-rope).
//
// Every token selects exactly K heads, so sequence b's rows start at b*T*K and each
// sequence's segment offsets depend only on that sequence's own head counts.
//
// One cooperative launch when the chunks of all sequences fit on the GPU at once:
//   route_fused_kernel     per 256-token chunk: TopK + gates and chunk head counts; one
//                          bounded grid barrier; then every chunk sums its sequence's count
//                          table itself (chunk bases, n, segment offsets) and ranks its
//                          tokens with warp ballots.
// Otherwise three stream-ordered launches:
//   1. route_topk_kernel   one thread per token: TopK of the fp32 logits (descending,
//                          ties to the lower head index), fp32 softmax gates over all H,
//                          and per-chunk head counts (one block = one 256-token chunk).
//   2. route_scan_kernel   one block per sequence: exclusive scan of the chunk counts over
//                          chunks for every head -> chunk base ranks, n[b, h] and the
//                          sequence's segment offsets.
//   3. route_rank_kernel   per chunk: warp ballots give each (token, slot) its rank among
//                          the chunk's earlier tokens for that head; adds the chunk base
//                          -> rank, row and row_src.
// All integer work is exact, so the packed layout is deterministic and bit-identical to
// a sequential append in token order, on either path.
#include <float.h>

#include <mutex>

#include "common.cuh"

namespace namoh {
namespace {

constexpr int kChunk = 256;  // tokens per block in the top-K and rank kernels

// TopK and gates of token `tok` (Sec. 3.1 Eq. namoh-gates).  Writes topk_head and gate,
// adds the picks to s_cnt (when given) and returns the picked heads as a bit mask.
template <int HMAX>
__device__ __forceinline__ uint64_t topk_token(const float* __restrict__ scores, size_t tok, int H, int K,
                                               int32_t* __restrict__ topk_head, float* __restrict__ gate, int* s_cnt,
                                               int* s_bad) {
  // this token's H logits: independent loads, all in flight together
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
  uint64_t mask = 0;
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
    if (s_cnt) atomicAdd(&s_cnt[bi], 1);
    mask |= 1ull << bi;
    pv = bv;
    pi = bi;
  }
  if (bad) *s_bad = 1;
  return mask;
}

template <int HMAX>
__global__ void __launch_bounds__(kChunk) route_topk_kernel(const float* __restrict__ scores, int T, int H, int K,
                                                            int nchunks, int32_t* __restrict__ topk_head,
                                                            float* __restrict__ gate,
                                                            int32_t* __restrict__ chunk_count,
                                                            uint32_t* __restrict__ status) {
  __shared__ int s_cnt[NAMOH_MAX_HEADS];
  __shared__ int s_bad;
  const int c = blockIdx.x;
  const int b = blockIdx.y;
  const int tid = threadIdx.x;
  const int t = c * kChunk + tid;
  if (tid < NAMOH_MAX_HEADS) s_cnt[tid] = 0;
  if (tid == 0) s_bad = 0;
  __syncthreads();
  if (t < T) topk_token<HMAX>(scores, (size_t)b * T + t, H, K, topk_head, gate, chunk_count ? s_cnt : nullptr, &s_bad);
  __syncthreads();
  if (chunk_count && tid < H) chunk_count[((size_t)b * nchunks + c) * H + tid] = s_cnt[tid];
  if (tid == 0 && s_bad) report(status, NAMOH_DEV_NONFINITE_SCORE);
}

// One block per sequence b: for every head, exclusive scan of the chunk counts over chunks
// (thread (h, p) owns the chunk range [p*per, (p+1)*per)) -> chunk bases and n[b, h]; then
// seg_offsets[b*H + h] = b*T*K + sum of n[b, h'] over h' < h.
__global__ void __launch_bounds__(1024) route_scan_kernel(const int32_t* __restrict__ chunk_count, int B, int T,
                                                          int H, int K, int nchunks, int32_t* __restrict__ chunk_base,
                                                          int32_t* __restrict__ seg_offsets) {
  __shared__ int s_part[1024];
  __shared__ int s_n[NAMOH_MAX_HEADS];
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
  if (p == P - 1) s_n[h] = run;
  __syncthreads();
  if (tid == 0) {
    int off = b * T * K;  // < 2^31: checked on the host
    for (int hh = 0; hh < H; ++hh) {
      seg_offsets[(size_t)b * H + hh] = off;
      off += s_n[hh];
    }
    if (b == B - 1) seg_offsets[(size_t)B * H] = off;
  }
}

// Ranks of one chunk's (token, slot) pairs (Sec. 3.2 Eq. namoh-head-rope): rho = chunk base
// + rank among this chunk's earlier tokens for the head (warp ballots).  s_cbase and s_soff
// (chunk base and segment offset per head) must be ready in shared memory; `mask` holds the
// thread's picked heads (0 past the end).  Ends with no block barrier pending.
struct RankSmem {
  uint32_t bal[kChunk / 32][NAMOH_MAX_HEADS];
  int wbase[kChunk / 32][NAMOH_MAX_HEADS];
  int cbase[NAMOH_MAX_HEADS];  // rank of the chunk's first token for each head
  int soff[NAMOH_MAX_HEADS];   // segment offset of each head in this sequence
};

__device__ __forceinline__ void rank_chunk(RankSmem& sm, uint64_t mask, bool valid, size_t tok, int H, int K,
                                           const int32_t* topk_head, int32_t* __restrict__ rank,
                                           int32_t* __restrict__ row, int32_t* __restrict__ row_src) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  for (int h = 0; h < H; ++h) {
    const uint32_t bal = __ballot_sync(0xffffffffu, (mask >> h) & 1ull);
    if (lane == 0) sm.bal[warp][h] = bal;
  }
  __syncthreads();
  for (int i = tid; i < (kChunk / 32) * H; i += kChunk) {
    const int w = i / H, h = i % H;
    int before = 0;
    for (int q = 0; q < w; ++q) before += __popc(sm.bal[q][h]);
    sm.wbase[w][h] = before;
  }
  __syncthreads();
  if (!valid) return;
  const uint32_t lt = (1u << lane) - 1u;
  for (int k = 0; k < K; ++k) {
    const int h = topk_head[tok * K + k];
    const int rho = sm.cbase[h] + sm.wbase[warp][h] + __popc(sm.bal[warp][h] & lt);
    const int r = sm.soff[h] + rho;
    rank[tok * K + k] = rho;
    row[tok * K + k] = r;
    row_src[r] = (int32_t)(tok * K + k);
  }
}

__global__ void __launch_bounds__(kChunk) route_rank_kernel(const int32_t* __restrict__ topk_head, int T, int H,
                                                            int K, int nchunks,
                                                            const int32_t* __restrict__ chunk_base,
                                                            const int32_t* __restrict__ seg_offsets,
                                                            int32_t* __restrict__ rank, int32_t* __restrict__ row,
                                                            int32_t* __restrict__ row_src) {
  __shared__ RankSmem sm;
  const int c = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x;
  const int t = c * kChunk + tid;
  const bool valid = t < T;
  const size_t tok = (size_t)b * T + t;
  if (tid < H) {
    sm.cbase[tid] = chunk_base[((size_t)b * nchunks + c) * H + tid];
    sm.soff[tid] = seg_offsets[(size_t)b * H + tid];
  }
  uint64_t mask = 0;
  if (valid)
    for (int k = 0; k < K; ++k) mask |= 1ull << __ldg(topk_head + tok * K + k);
  rank_chunk(sm, mask, valid, tok, H, K, topk_head, rank, row, row_src);
}

// Grid barrier for a cooperative launch.  *count must be 0 at launch (the host clears it);
// every block adds 1 and waits, bounded, until all have.  Returns false after a timeout
// (NAMOH_DEV_TIMEOUT is reported).
__device__ __forceinline__ bool grid_barrier(unsigned* count, unsigned nblocks, uint32_t* status) {
  __shared__ int s_ok;
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(count, 1u);
    int ok = 1;
    const uint64_t t0 = global_timer_ns();
    for (;;) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(count) : "memory");
      if (v >= nblocks) break;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        report(status, NAMOH_DEV_TIMEOUT);
        ok = 0;
        break;
      }
      __nanosleep(64);
    }
    s_ok = ok;
  }
  __syncthreads();
  return s_ok != 0;
}

// The whole of routing in one cooperative launch: grid = B * nchunks blocks, all resident.
template <int HMAX>
__global__ void __launch_bounds__(kChunk) route_fused_kernel(const float* __restrict__ scores, int T, int H, int K,
                                                             int nchunks, int32_t* __restrict__ topk_head,
                                                             float* __restrict__ gate, int32_t* chunk_count,
                                                             unsigned* barrier, int32_t* __restrict__ rank,
                                                             int32_t* __restrict__ row,
                                                             int32_t* __restrict__ seg_offsets,
                                                             int32_t* __restrict__ row_src, int B,
                                                             uint32_t* __restrict__ status) {
  __shared__ RankSmem sm;
  __shared__ int s_cnt[NAMOH_MAX_HEADS];
  __shared__ int s_tot[kChunk];
  __shared__ int s_bef[kChunk];
  __shared__ int s_bad;
  const int c = blockIdx.x % nchunks;
  const int b = blockIdx.x / nchunks;
  const int tid = threadIdx.x;
  const int t = c * kChunk + tid;
  const bool valid = t < T;
  const size_t tok = (size_t)b * T + t;
  if (tid < NAMOH_MAX_HEADS) s_cnt[tid] = 0;
  if (tid == 0) s_bad = 0;
  __syncthreads();
  uint64_t mask = 0;
  if (valid) mask = topk_token<HMAX>(scores, tok, H, K, topk_head, gate, s_cnt, &s_bad);
  __syncthreads();
  if (tid < H) chunk_count[((size_t)b * nchunks + c) * H + tid] = s_cnt[tid];
  if (tid == 0 && s_bad) report(status, NAMOH_DEV_NONFINITE_SCORE);
  if (!grid_barrier(barrier, gridDim.x, status)) return;

  // this sequence's count table: thread (h, p) sums chunks p, p + P, ... (L2 reads)
  const int P = kChunk / H;
  const int h = tid % H, p = tid / H;
  int tot = 0, bef = 0;
  if (p < P) {
    const int32_t* cc = chunk_count + (size_t)b * nchunks * H + h;
    for (int cj = p; cj < nchunks; cj += P) {
      const int v = __ldcg(cc + (size_t)cj * H);
      tot += v;
      bef += (cj < c) ? v : 0;
    }
  }
  s_tot[tid] = tot;
  s_bef[tid] = bef;
  __syncthreads();
  if (tid < H) {
    int n = 0, cb = 0;
    for (int q = 0; q < P; ++q) {
      n += s_tot[q * H + tid];
      cb += s_bef[q * H + tid];
    }
    sm.cbase[tid] = cb;
    s_tot[tid] = n;  // rows q >= 1 of s_tot are no longer read
  }
  __syncthreads();
  if (tid == 0) {
    int off = b * T * K;  // < 2^31: checked on the host
    for (int hh = 0; hh < H; ++hh) {
      sm.soff[hh] = off;
      off += s_tot[hh];
    }
  }
  __syncthreads();
  if (c == 0 && tid < H) seg_offsets[(size_t)b * H + tid] = sm.soff[tid];
  if (c == 0 && b == B - 1 && tid == 0) seg_offsets[(size_t)B * H] = B * T * K;
  rank_chunk(sm, mask, valid, tok, H, K, topk_head, rank, row, row_src);
}

constexpr int kFusedMaxTable = 1 << 15;  // chunk-count entries one sequence may have on the fused path

// Blocks of route_fused_kernel<HMAX> that fit on the current device at once (0 if the
// device cannot launch cooperatively).  Cached per device.
template <int HMAX>
int fused_capacity() {
  static std::mutex mu;
  static int cached[64] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  std::lock_guard<std::mutex> lock(mu);
  if (cached[dev] == 0) {
    int coop = 0, sms = 0, per_sm = 0;
    if (cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, route_fused_kernel<HMAX>, kChunk, 0) != cudaSuccess) {
      cudaGetLastError();
      return 0;
    }
    cached[dev] = coop ? sms * per_sm : -1;
  }
  return cached[dev] > 0 ? cached[dev] : 0;
}

struct RouteArgs {
  const float* scores;
  int B, T, H, K, nchunks;
  int32_t *topk_head, *rank, *row, *seg_offsets, *row_src;
  float* gate;
  int32_t *chunk_count, *chunk_base;
  unsigned* barrier;
  uint32_t* status;
};

// Returns 1 when launched on the fused path, 0 when the shape needs the three-launch path,
// or a negative status.
template <int HMAX>
int try_fused(const RouteArgs& a, cudaStream_t stream) {
  const long long nblocks = (long long)a.B * a.nchunks;
  if ((long long)a.nchunks * a.H > kFusedMaxTable || nblocks > fused_capacity<HMAX>()) return 0;
  cudaError_t e = cudaMemsetAsync(a.barrier, 0, sizeof(unsigned), stream);
  if (e != cudaSuccess) return cuda_fail(e, "route barrier memset");
  const float* scores = a.scores;
  int T = a.T, H = a.H, K = a.K, nchunks = a.nchunks, B = a.B;
  int32_t *topk = a.topk_head, *cc = a.chunk_count, *rank = a.rank, *row = a.row, *so = a.seg_offsets,
          *rs = a.row_src;
  float* gate = a.gate;
  unsigned* bar = a.barrier;
  uint32_t* st = a.status;
  void* args[] = {&scores, &T, &H, &K, &nchunks, &topk, &gate, &cc, &bar, &rank, &row, &so, &rs, &B, &st};
  e = cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(route_fused_kernel<HMAX>), dim3((unsigned)nblocks),
                                  dim3(kChunk), args, 0, stream);
  if (e != cudaSuccess) return cuda_fail(e, "route_fused_kernel cooperative launch");
  return 1;
}

template <int HMAX>
int launch_route(const RouteArgs& a, cudaStream_t stream) {
  const bool compact = a.seg_offsets != nullptr;
  if (compact) {
    const int f = try_fused<HMAX>(a, stream);
    if (f != 0) return f < 0 ? f : NAMOH_OK;
  }
  route_topk_kernel<HMAX><<<dim3(a.nchunks, a.B), kChunk, 0, stream>>>(a.scores, a.T, a.H, a.K, a.nchunks, a.topk_head,
                                                                       a.gate, a.chunk_count, a.status);
  if (const int st = cuda_check_launch("route_topk_kernel launch")) return st;
  if (!compact) return NAMOH_OK;
  const int scan_threads = 1024 - (1024 % a.H);
  route_scan_kernel<<<a.B, scan_threads, 0, stream>>>(a.chunk_count, a.B, a.T, a.H, a.K, a.nchunks, a.chunk_base,
                                                      a.seg_offsets);
  if (const int st = cuda_check_launch("route_scan_kernel launch")) return st;
  route_rank_kernel<<<dim3(a.nchunks, a.B), kChunk, 0, stream>>>(a.topk_head, a.T, a.H, a.K, a.nchunks, a.chunk_base,
                                                                 a.seg_offsets, a.rank, a.row, a.row_src);
  return cuda_check_launch("route_rank_kernel launch");
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
  ws.take<unsigned>(1);                       // grid barrier counter
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
  RouteArgs a{};
  a.scores = scores;
  a.B = B;
  a.T = T;
  a.H = H;
  a.K = K;
  a.nchunks = (T + kChunk - 1) / kChunk;
  a.topk_head = topk_head;
  a.gate = gate;
  a.rank = rank;
  a.row = row;
  a.seg_offsets = seg_offsets;
  a.row_src = row_src;
  a.status = dev_status;
  if (compact) {
    if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
    WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
    a.chunk_count = ws.take<int32_t>((size_t)B * a.nchunks * H);
    a.chunk_base = ws.take<int32_t>((size_t)B * a.nchunks * H);
    a.barrier = ws.take<unsigned>(1);
    if (!ws.fits()) return NAMOH_ERR_WORKSPACE;
  }
  if (H <= 8) return launch_route<8>(a, stream);
  if (H <= 16) return launch_route<16>(a, stream);
  if (H <= 32) return launch_route<32>(a, stream);
  return launch_route<64>(a, stream);
}

// ---------------------------------------------------------------------------
// Routing with built-in scratch (no caller workspace, no allocation).
// The scratch is a file-scope device array; host code only ever passes the
// device address obtained from cudaGetSymbolAddress, never the array's name.
// ---------------------------------------------------------------------------

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
