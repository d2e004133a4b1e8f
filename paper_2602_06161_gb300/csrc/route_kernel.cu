// route_kernel.cu - exported seed routing (slot map, per-128-row bitmap and
// count of ignored entries), built on the same device routine the attention
// kernels run in their prologue.
#include "kernels.cuh"
#include "route.cuh"

namespace cover {
namespace {

constexpr int kRows = 128;

// grid (ceil(L / 128), B), 128 threads: one CTA per 128-row tile of one batch row.
__global__ void __launch_bounds__(kRows)
    seed_route_kernel(const int32_t* __restrict__ seed_idx, int n_seeds, int L, int32_t* __restrict__ slot_out,
                      uint32_t* __restrict__ bitmap_out, int32_t* __restrict__ n_invalid_out) {
  __shared__ int slot[kRows];
  const int tile = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int row0 = tile * kRows;
  const int32_t* seeds_b = seed_idx + static_cast<size_t>(b) * n_seeds;
  route_clear(slot, kRows, tid, kRows);
  __syncthreads();
  route_scan(slot, seeds_b, n_seeds, row0, kRows, L, tid, kRows);
  __syncthreads();

  const int r = row0 + tid;
  const int s = slot[tid];
  const bool is_seed = (r < L) && (s != kNoSlot);
  if (r < L) slot_out[static_cast<size_t>(b) * L + r] = is_seed ? s : -1;
  const uint32_t word = __ballot_sync(0xffffffffu, is_seed);
  const int n_tiles = (L + kRows - 1) / kRows;
  if ((tid & 31) == 0) bitmap_out[(static_cast<size_t>(b) * n_tiles + tile) * 4 + tid / 32] = word;

  // ignored entries: those naming a position in this tile that lost to a lower
  // slot; out-of-range entries are counted once per batch row by tile 0
  int bad = 0;
  for (int t = tid; t < n_seeds; t += kRows) {
    const int p = seeds_b[t];
    if (p >= row0 && p < row0 + kRows && p < L) {
      if (slot[p - row0] != t) ++bad;
    } else if (tile == 0 && (p < 0 || p >= L)) {
      ++bad;
    }
  }
  for (int o = 16; o > 0; o >>= 1) bad += __shfl_xor_sync(0xffffffffu, bad, o);
  if ((tid & 31) == 0 && bad) atomicAdd(n_invalid_out, bad);
}

}  // namespace

int launch_seed_route(const int32_t* seed_idx, int n_seeds, int B, int L, int32_t* slot_out, uint32_t* bitmap_out,
                      int32_t* n_invalid_out, cudaStream_t stream) {
  if (cudaMemsetAsync(n_invalid_out, 0, sizeof(int32_t), stream) != cudaSuccess) return -3;
  dim3 grid((L + kRows - 1) / kRows, B);
  seed_route_kernel<<<grid, kRows, 0, stream>>>(seed_idx, n_seeds, L, slot_out, bitmap_out, n_invalid_out);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
