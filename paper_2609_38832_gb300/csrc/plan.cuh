// plan.cuh -- length-aware work list of the attention kernel (Sec. 3.2 "Efficient
// execution": length-aware scheduling of query tiles).
//
// Items are the 128-row query tiles q of every segment and group head j, ordered by
// decreasing cost (tile q needs q + 1 key tiles), then (segment, j).  Each item carries
// {segment * g + j, q, seg_offsets[segment], n}, so a CTA starts on it after one load.
// Segments longer than their cache capacity (seg_cap, when given) are left out.  The
// header holds {next item, CTAs finished, item count}; the attention kernel's CTAs take
// item blockIdx first and then items in order from an atomic counter, and its last CTA
// resets the first two words.
#pragma once

#include "common.cuh"

namespace namoh {

constexpr int kPlanTileRows = 128;

// Shared-memory ints the plan needs: two per query-tile index and one per segment.
__host__ __device__ inline int plan_smem_ints(int max_qtiles, int nseg) { return 2 * max_qtiles + nseg; }

// Executed by one whole block (any size) with plan_smem_ints(...) ints of shared memory.
__device__ inline void build_plan(const int32_t* __restrict__ seg_offsets, int nseg, const int32_t* __restrict__ seg_cap,
                                  int g, int max_qtiles, int* __restrict__ header, int4* __restrict__ items,
                                  int* s_mem) {
  int* s_count = s_mem;                   // [max_qtiles]: segments with more than q query tiles
  int* s_start = s_mem + max_qtiles;      // [max_qtiles]: first item of cost q + 1
  int* s_ntile = s_mem + 2 * max_qtiles;  // [nseg]: query tiles of each segment (0 if skipped)
  const int tid = threadIdx.x;
  for (int q = tid; q < max_qtiles; q += blockDim.x) s_count[q] = 0;
  for (int s = tid; s < nseg; s += blockDim.x) {
    const int n = __ldg(seg_offsets + s + 1) - __ldg(seg_offsets + s);
    const bool skip = seg_cap && n > __ldg(seg_cap + s);
    s_ntile[s] = skip || n <= 0 ? 0 : min((n + kPlanTileRows - 1) / kPlanTileRows, max_qtiles);
  }
  __syncthreads();
  for (int s = tid; s < nseg; s += blockDim.x)
    if (s_ntile[s] > 0) atomicAdd(&s_count[s_ntile[s] - 1], 1);  // histogram of tile counts
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
    for (int s = 0; s < nseg; ++s)
      if (s_ntile[s] > q) {
        const int off = __ldg(seg_offsets + s), n = __ldg(seg_offsets + s + 1) - off;
        for (int j = 0; j < g; ++j) items[pos++] = make_int4(s * g + j, q, off, n);
      }
  }
}

}  // namespace namoh
