// proj_out.cu -- the output projection (Sec. 3.1, Eq. namoh-attention):
//   o_t = sum_{i in S_K(t)} g_{t,i} h_{t,i} W_O^(i)
// from the combine's per-slot terms y = g h (App. C: a KV group's g query heads each have
// their own W_O, stacked along the contraction: y_r [W_O^(ig); ...; W_O^(ig+g-1)]).
//
// Work is cut by token windows, so that every token's K slots meet in one CTA and o is
// written once, without atomics:
//   1. pack_rows_kernel    y in packed-row order: row r = y[row_src[r]] (so the rows of a
//                          segment are contiguous and load as TMA tiles).
//   2. window_table_kernel for window w (kWin consecutive tokens of the flat token axis) and
//                          segment s: the first row of s whose token is >= w kWin (rows ascend
//                          in token inside a segment), so the rows of s in w are
//                          [table[w][s], table[w+1][s]); then window_bounds_kernel: the range
//                          of segments with rows in each window (the sequences it overlaps).
//   3. proj_out_kernel     one persistent CTA per SM over items (window, 64-column chunk of
//                          d_model).  For each segment with rows in the window and each 128-row
//                          tile of them: tcgen05.mma of the tile's y rows against the segment
//                          group's W_O chunk into TMEM (four accumulators in turn); the
//                          epilogue adds each row into a shared-memory fp32 accumulator at its
//                          token's place in the window (rows of one segment are distinct
//                          tokens; the epilogue warps meet before the next segment's rows).
//                          After the window's last tile the accumulator holds complete o rows
//                          and is written (or added) to o.  Each role reads a window's table
//                          slice warp-wide (one load for 32 segments) and walks it by shuffles.
//   warps 0-3 epilogue, warp 4 TMA loads (A = 128 packed y rows, B = 64 rows of W_O), warp 5
//   TMEM owner and MMA issue.  Every wait is bounded (NAMOH_DEV_TIMEOUT).
#include "common.cuh"

namespace namoh {
namespace projo {

constexpr int BM = 128;    // packed rows per MMA tile
constexpr int BN = 64;     // o columns per item
constexpr int BK = 64;     // contraction elements per stage
constexpr int kWin = 512;  // tokens per window
constexpr int kThreads = 192;
constexpr int kStages = 3;
constexpr int kA = BM * 128;              // 16 KB
constexpr int kB = BN * 128;              // 8 KB
constexpr int kStage = kA + kB;
constexpr int kAcc = kWin * BN * 4;       // 128 KB fp32 window accumulator
constexpr int kAccBufs = 4;               // TMEM accumulators of 64 columns
constexpr int kAccOff = kStages * kStage;
constexpr int kBar = kAccOff + kAcc;
constexpr int kAlloc = kBar + 256 + 1024;

struct Params {
  const int32_t* table;     // [(nwin + 1) * nseg]
  const int2* bounds;       // [nwin]: segments [x, y) have rows in the window
  const int32_t* row_src;   // [R]
  int nseg, Hr, Kr, nwin, ntok, d_model, kdim;
  float* o;
  int accumulate;
  uint32_t* status;
};

struct Bars {
  uint64_t full[kStages], empty[kStages];
  uint64_t acc_full[kAccBufs], acc_empty[kAccBufs];
  uint32_t tmem_base;
  int abort_flag;
};

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, volatile int* abort_flag, uint32_t* status) {
  const bool ok = mbar_wait(bar, parity, abort_flag, status);
  return __all_sync(0xffffffffu, ok);
}


__global__ void pack_rows_kernel(const uint16_t* __restrict__ y, const int32_t* __restrict__ row_src, long long R,
                                 int gd, long long y_rows, uint16_t* __restrict__ yp) {
  const int vpr = gd / 8;  // 16-byte vectors per row
  const long long n = R * vpr;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const long long r = i / vpr;
    const int c = (int)(i - r * vpr);
    long long src = __ldg(row_src + r);
    src = src < 0 ? 0 : (src >= y_rows ? y_rows - 1 : src);
    reinterpret_cast<uint4*>(yp)[i] = __ldg(reinterpret_cast<const uint4*>(y + src * gd) + c);
  }
}

__global__ void window_table_kernel(const int32_t* __restrict__ seg_offsets, const int32_t* __restrict__ row_src,
                                    int nseg, int nwin, int Kr, int32_t* __restrict__ table) {
  const long long n = (long long)(nwin + 1) * nseg;
  for (long long i = blockIdx.x * (long long)blockDim.x + threadIdx.x; i < n; i += (long long)gridDim.x * blockDim.x) {
    const int w = (int)(i / nseg), s = (int)(i - (long long)w * nseg);
    const int lo0 = __ldg(seg_offsets + s);
    const int hi0 = max(lo0, __ldg(seg_offsets + s + 1));
    int lo = lo0, hi = hi0;
    if (w >= nwin) {
      lo = hi0;
    } else {
      const long long target = (long long)w * kWin;  // first row whose token is >= target
      while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if ((long long)(__ldg(row_src + mid) / Kr) < target) lo = mid + 1; else hi = mid;
      }
    }
    table[i] = lo;
  }
}

__global__ void window_bounds_kernel(const int32_t* __restrict__ table, int nseg, int nwin, int2* __restrict__ bounds) {
  for (int w = blockIdx.x * blockDim.x + threadIdx.x; w < nwin; w += gridDim.x * blockDim.x) {
    int first = nseg, last = 0;
    for (int s = 0; s < nseg; ++s) {
      if (__ldg(table + (long long)w * nseg + s) < __ldg(table + (long long)(w + 1) * nseg + s)) {
        first = min(first, s);
        last = s + 1;
      }
    }
    bounds[w] = make_int2(first, last);
  }
}

__global__ void __launch_bounds__(kThreads, 1) proj_out_kernel(const __grid_constant__ CUtensorMap tm_a,
                                                               const __grid_constant__ CUtensorMap tm_b, Params p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  Bars* bars = reinterpret_cast<Bars*>(smem + kBar);
  float4* acc = reinterpret_cast<float4*>(smem + kAccOff);  // [kWin][16], vector v of row r at (v + r) & 15
  volatile int* abort_flag = &bars->abort_flag;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&bars->full[i], 1);
      mbar_init(&bars->empty[i], 1);
    }
    for (int i = 0; i < kAccBufs; ++i) {
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
    tmem_alloc(&bars->tmem_base, kAccBufs * BN);
    tmem_relinquish();
  }
  if (warp < 4)
    for (int i = threadIdx.x; i < kWin * 16; i += 128) acc[i] = make_float4(0.f, 0.f, 0.f, 0.f);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem_base;
  pdl_wait();  // the packed y rows and the window table are visible from here

  const int nchunks = p.d_model / BN;
  const int nitems = p.nwin * nchunks;
  const int nk = p.kdim / BK;
  // The segments of window w with their rows [lo, hi), walked warp-wide: lane l loads the
  // table entries of segment base + l, then fn(s, lo, hi) runs for each in order (all lanes).
  // fn returns false to stop.
  auto for_segments = [&](int w, auto&& fn) {
    const int2 sb = __ldg(p.bounds + w);
    for (int base = sb.x; base < sb.y; base += 32) {
      const int sl = base + lane;
      int lo_l = 0, hi_l = 0;
      if (sl < sb.y) {
        lo_l = __ldg(p.table + (long long)w * p.nseg + sl);
        hi_l = __ldg(p.table + (long long)(w + 1) * p.nseg + sl);
      }
      const int cnt = min(32, sb.y - base);
      for (int j = 0; j < cnt; ++j) {
        const int lo = __shfl_sync(0xffffffffu, lo_l, j), hi = __shfl_sync(0xffffffffu, hi_l, j);
        if (lo < hi && !fn(base + j, lo, hi)) return false;
      }
    }
    return true;
  };

  if (warp == 4) {
    // ---- loads (lane 0 issues; the warp walks the tables)
    uint32_t it = 0;
    for (int item = blockIdx.x; item < nitems; item += gridDim.x) {
      const int w = item / nchunks, nc = item - w * nchunks;
      const bool ok = for_segments(w, [&](int s, int lo, int hi) {
        const int b_row = (s % p.Hr) * p.d_model + nc * BN;
        for (int m = lo; m < hi; m += BM) {
          for (int kb = 0; kb < nk; ++kb, ++it) {
            const int slot = it % kStages;
            if (it >= (uint32_t)kStages &&
                !warp_wait(&bars->empty[slot], ((it / kStages) - 1) & 1, abort_flag, p.status))
              return false;
            uint8_t* a = smem + slot * kStage;
            if (lane == 0) {
              mbar_arrive_expect_tx(&bars->full[slot], kStage);
              tma_load_2d(a, &tm_a, kb * BK, m, &bars->full[slot]);
              tma_load_2d(a + kA, &tm_b, kb * BK, b_row, &bars->full[slot]);
            }
          }
        }
        return true;
      });
      if (!ok) break;
    }
  } else if (warp == 5) {
    constexpr uint32_t idesc = make_idesc_bf16(BM, BN, false, false);
    uint32_t it = 0, sub = 0;
    for (int item = blockIdx.x; item < nitems; item += gridDim.x) {
      const int w = item / nchunks;
      const bool ok = for_segments(w, [&](int s, int lo, int hi) {
        for (int m = lo; m < hi; m += BM, ++sub) {
          const int buf = sub % kAccBufs;
          if (sub >= kAccBufs &&
              !warp_wait(&bars->acc_empty[buf], ((sub / kAccBufs) - 1) & 1, abort_flag, p.status))
            return false;
          tc_fence_after();
          const uint32_t d_tmem = tmem + buf * BN;
          for (int kb = 0; kb < nk; ++kb, ++it) {
            const int slot = it % kStages;
            if (!warp_wait(&bars->full[slot], (it / kStages) & 1, abort_flag, p.status)) return false;
            tc_fence_after();
            const uint64_t a_desc = make_smem_desc_sw128(smem_u32(smem + slot * kStage), 16, 1024);
            const uint64_t b_desc = make_smem_desc_sw128(smem_u32(smem + slot * kStage + kA), 16, 1024);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              mma_bf16_ss(d_tmem, a_desc + (uint64_t)(kk * 2), b_desc + (uint64_t)(kk * 2), idesc,
                          (kb | kk) ? 1u : 0u);
            mma_commit(&bars->empty[slot]);
          }
          mma_commit(&bars->acc_full[buf]);
        }
        return true;
      });
      if (!ok) break;
    }
  } else {
    // ---- epilogue: thread = tile row = TMEM lane; the 128 threads share the window accumulator
    const int row = warp * 32 + lane;
    const uint32_t lane_addr = (uint32_t)(warp * 32) << 16;
    uint32_t sub = 0;
    bool ok = true;
    // The four warps meet on hardware barrier 1 and vote: every warp reaches every meeting
    // (a warp whose wait gave up skips its work, not the meeting), so all leave together.
    auto epi_sync = [&]() {
      uint32_t all;
      asm volatile(
          "{\n\t.reg .pred p, q;\n\t"
          "setp.ne.u32 p, %1, 0;\n\t"
          "bar.red.and.pred q, 1, 128, p;\n\t"
          "selp.u32 %0, 1, 0, q;\n\t}"
          : "=r"(all)
          : "r"((uint32_t)ok)
          : "memory");
      ok = all != 0;
    };
    for (int item = blockIdx.x; item < nitems && ok; item += gridDim.x) {
      const int w = item / nchunks, nc = item - w * nchunks;
      const long long w0 = (long long)w * kWin;
      for_segments(w, [&](int s, int lo, int hi) {
        for (int m = lo; m < hi && ok; m += BM, ++sub) {
          const int buf = sub % kAccBufs;
          const bool valid = m + row < hi;
          // issued here, ahead of the wait (a plain load may be sunk to its first use after it)
          const int src = valid ? ld_issue_s32(p.row_src + m + row) : 0;
          if (!warp_wait(&bars->acc_full[buf], (sub / kAccBufs) & 1, abort_flag, p.status)) {
            ok = false;
            break;
          }
          tc_fence_after();
          uint32_t v0[32], v1[32];
          tmem_ld32(tmem + lane_addr + buf * BN, v0);
          tmem_ld32(tmem + lane_addr + buf * BN + 32, v1);
          tmem_wait_ld();
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty[buf]);
          const long long slot = (long long)(src / p.Kr) - w0;
          if (valid && slot >= 0 && slot < kWin) {
            float4* ar = acc + slot * 16;
#pragma unroll
            for (int v = 0; v < 16; ++v) {
              const uint32_t* src4 = v < 8 ? v0 + 4 * v : v1 + 4 * (v - 8);
              float4& a = ar[(v + (int)slot) & 15];
              a.x += __uint_as_float(src4[0]);
              a.y += __uint_as_float(src4[1]);
              a.z += __uint_as_float(src4[2]);
              a.w += __uint_as_float(src4[3]);
            }
          }
        }
        epi_sync();  // the next segment's rows may share tokens with this one's
        return ok;
      });
      epi_sync();  // every tile of the window is in the accumulator
      if (!ok) break;
      // the window's o rows are complete: write (or add) them and clear the accumulator;
      // 16 threads per row, 4 columns each, 8 rows per pass with their loads issued together
      const int vec = threadIdx.x & 15;
      for (int r0 = threadIdx.x >> 4; r0 < kWin; r0 += 64) {
        float4 old[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const long long tok = w0 + r0 + 8 * j;
          old[j] = make_float4(0.f, 0.f, 0.f, 0.f);
          if (p.accumulate && tok < p.ntok)
            old[j] = reinterpret_cast<const float4*>(p.o + tok * p.d_model + nc * BN)[vec];
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int r = r0 + 8 * j;
          const long long tok = w0 + r;
          float4& a = acc[r * 16 + ((vec + r) & 15)];
          const float4 val = make_float4(a.x + old[j].x, a.y + old[j].y, a.z + old[j].z, a.w + old[j].w);
          a = make_float4(0.f, 0.f, 0.f, 0.f);
          if (tok < p.ntok) reinterpret_cast<float4*>(p.o + tok * p.d_model + nc * BN)[vec] = val;
        }
      }
      epi_sync();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag && threadIdx.x == 0) {
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < 1000000ull) {
    }
  }
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    tmem_dealloc(tmem, kAccBufs * BN);
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

struct OutWs {
  uint16_t* yp;
  int32_t* table;
  int2* bounds;
};
void carve_out(WorkspaceCarver& ws, OutWs* out, long long R, int gd, int nwin, int nseg) {
  out->yp = ws.take<uint16_t>((size_t)R * gd);
  out->table = ws.take<int32_t>((size_t)(nwin + 1) * nseg);
  out->bounds = ws.take<int2>((size_t)nwin);
}

}  // namespace projo

// Workspace of namoh_proj_out (the packed y rows and the window table).
size_t proj_out_workspace(long long total_tokens, int Kr, int gd, int nseg) {
  WorkspaceCarver ws{nullptr, 0, 0};
  projo::OutWs o;
  const int nwin = (int)((total_tokens + projo::kWin - 1) / projo::kWin);
  projo::carve_out(ws, &o, total_tokens * Kr, gd, nwin, nseg);
  return align_up(ws.used, 256);
}

int launch_proj_out(const uint16_t* y, int total_tokens, int d_model, const uint16_t* w_o, int Hr, int Kr, int gd,
                    int nseg, const int32_t* seg_offsets, const int32_t* row_src, float* o, int accumulate,
                    void* workspace, size_t workspace_bytes, uint32_t* dev_status, int sm_count, cudaStream_t stream) {
  using namespace projo;
  if (d_model % BN) return NAMOH_ERR_UNSUPPORTED;
  const long long R = (long long)total_tokens * Kr;
  const int nwin = (total_tokens + kWin - 1) / kWin;
  if (!workspace || (reinterpret_cast<uintptr_t>(workspace) & 255u)) return NAMOH_ERR_WORKSPACE;
  WorkspaceCarver ws{static_cast<char*>(workspace), workspace_bytes, 0};
  OutWs ow;
  carve_out(ws, &ow, R, gd, nwin, nseg);
  if (!ws.fits()) return NAMOH_ERR_WORKSPACE;

  pack_rows_kernel<<<sm_count * 4, 256, 0, stream>>>(y, row_src, R, gd, R, ow.yp);
  if (const int st = cuda_check_launch("pack_rows_kernel launch")) return st;
  const long long tn = (long long)(nwin + 1) * nseg;
  window_table_kernel<<<(unsigned)((tn + 255) / 256), 256, 0, stream>>>(seg_offsets, row_src, nseg, nwin, Kr,
                                                                          ow.table);
  if (const int st = cuda_check_launch("window_table_kernel launch")) return st;
  window_bounds_kernel<<<(nwin + 255) / 256, 256, 0, stream>>>(ow.table, nseg, nwin, ow.bounds);
  if (const int st = cuda_check_launch("window_bounds_kernel launch")) return st;

  CUtensorMap ta, tb;
  if (!encode_map(&ta, ow.yp, R, gd, BM) || !encode_map(&tb, w_o, (long long)Hr * d_model, gd, BN))
    return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled");
  Params p{};
  p.table = ow.table;
  p.bounds = ow.bounds;
  p.row_src = row_src;
  p.nseg = nseg;
  p.Hr = Hr;
  p.Kr = Kr;
  p.nwin = nwin;
  p.ntok = total_tokens;
  p.d_model = d_model;
  p.kdim = gd;
  p.o = o;
  p.accumulate = accumulate;
  p.status = dev_status;
  cudaError_t e = cudaFuncSetAttribute(proj_out_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kAlloc);
  if (e != cudaSuccess) return cuda_fail(e, "proj_out_kernel shared memory attribute");
  e = launch_pdl(proj_out_kernel, dim3(sm_count), dim3(kThreads), (size_t)kAlloc, stream, ta, tb, p);
  return e == cudaSuccess ? NAMOH_OK : cuda_fail(e, "proj_out_kernel launch");
}

}  // namespace namoh
