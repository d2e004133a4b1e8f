// route.cuh - seed routing shared by the attention kernels and the exported
// routing kernel. Seeds form a set of positions (Section 3, decoding protocol;
// Section 5.1); an entry outside [0, L) is ignored and, when a position is
// named more than once, the lowest slot is the one used.
#pragma once

#include <stdint.h>

namespace cover {

constexpr int kNoSlot = 0x7fffffff;

// Fills slot[0 .. rows) for positions [row0, row0 + rows) of one batch row:
// slot[r] = lowest s with seed_idx[s] == row0 + r, else kNoSlot. Must be
// called by all `nthreads` threads of the CTA (thread index `tid`), with a
// __syncthreads() between the two phases provided by the caller:
//   route_clear(...); __syncthreads(); route_scan(...); __syncthreads();
__device__ __forceinline__ void route_clear(int* slot, int rows, int tid, int nthreads) {
  for (int r = tid; r < rows; r += nthreads) slot[r] = kNoSlot;
}

__device__ __forceinline__ void route_scan(int* slot, const int32_t* __restrict__ seeds_b, int n_seeds, int row0,
                                           int rows, int L, int tid, int nthreads) {
  for (int s = tid; s < n_seeds; s += nthreads) {
    const int p = __ldg(seeds_b + s);
    if (p >= row0 && p < row0 + rows && p < L) atomicMin(slot + (p - row0), s);
  }
}

}  // namespace cover
