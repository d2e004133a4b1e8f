// kv_kernel.cu - the seed key/value cache of Section 5.1 ("KV cache override
// yields a stable drafting view").
//
// At selection the per-layer states of the new seeds are cached:
//   cache[b, h, s, :] = state[b, h, seed_idx[b, s], :]                 (gather)
// At the next step the memory computed from the masked input is overridden at
// the seed positions with the cached states, and the masked-input states move
// into the cache buffer, which then holds the diagonal pairs (k_i, v_i) that
// the attention kernel restores for the leave-one-out views:
//   swap(state[b, h, seed_idx[b, s], :], cache[b, h, s, :])            (override)
// A slot names its position only if the position is in [0, L) and no lower
// slot of the same batch row names it (the lowest slot wins, as in the
// attention kernel's routing); other slots copy zeros (gather) or leave both
// buffers untouched (override).
//
// Pure data movement: one CTA per (batch row, KV head, 16 slots), one thread
// per 16-byte vector of a row.
#include <stdint.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace cover {
namespace {

constexpr int kThreads = 256;
constexpr int kSlotsPerCta = 16;

struct KvParams {
  uint8_t* k;
  uint8_t* v;
  const int32_t* seed_idx;
  int S, L, Hkv;
  int row_vecs;       // 16-byte vectors per row
  uint8_t* k_cache;
  uint8_t* v_cache;
};

template <bool kOverride>
__global__ void __launch_bounds__(kThreads) seed_kv_kernel(const KvParams p) {
  __shared__ int s_pos[kSlotsPerCta];
  __shared__ int s_dup[kSlotsPerCta];
  // programmatic dependent launch: wait for the stream's previous kernel, let the next one be
  // scheduled
  griddep_wait();
  griddep_launch_dependents();
  const int bh = blockIdx.x;               // b * Hkv + h
  const int b = bh / p.Hkv;
  const int slot0 = blockIdx.y * kSlotsPerCta;
  const int tid = threadIdx.x;
  const int32_t* seeds = p.seed_idx + static_cast<size_t>(b) * p.S;

  if (tid < kSlotsPerCta) {
    const int s = slot0 + tid;
    int j = -1;
    if (s < p.S) {
      j = seeds[s];
      if (j < 0 || j >= p.L) j = -1;
    }
    s_pos[tid] = j;
    s_dup[tid] = 0;
  }
  __syncthreads();
  if (kOverride) {
    // a slot that repeats the position of a lower slot does not own it
    const int total = kSlotsPerCta * (slot0 + kSlotsPerCta);
    for (int w = tid; w < total; w += kThreads) {
      const int slot = w % kSlotsPerCta;
      const int other = w / kSlotsPerCta;
      const int j = s_pos[slot];
      if (j >= 0 && other < slot0 + slot && seeds[other] == j) s_dup[slot] = 1;
    }
    __syncthreads();
    if (tid < kSlotsPerCta && s_dup[tid]) s_pos[tid] = -1;
    __syncthreads();
  }

  const size_t row_bytes = static_cast<size_t>(p.row_vecs) * 16;
  for (int w = tid; w < kSlotsPerCta * p.row_vecs; w += kThreads) {
    const int slot = w / p.row_vecs, vec = w % p.row_vecs;
    const int s = slot0 + slot;
    if (s >= p.S) continue;
    const int j = s_pos[slot];
    const size_t mem_off = (static_cast<size_t>(bh) * p.L + (j < 0 ? 0 : j)) * row_bytes + vec * 16;
    const size_t cache_off = (static_cast<size_t>(bh) * p.S + s) * row_bytes + vec * 16;
    uint4* kc = reinterpret_cast<uint4*>(p.k_cache + cache_off);
    uint4* vc = reinterpret_cast<uint4*>(p.v_cache + cache_off);
    if (!kOverride) {
      uint4 kv = make_uint4(0, 0, 0, 0), vv = make_uint4(0, 0, 0, 0);
      if (j >= 0) {
        kv = *reinterpret_cast<const uint4*>(p.k + mem_off);
        vv = *reinterpret_cast<const uint4*>(p.v + mem_off);
      }
      *kc = kv;
      *vc = vv;
    } else if (j >= 0) {
      uint4* km = reinterpret_cast<uint4*>(p.k + mem_off);
      uint4* vm = reinterpret_cast<uint4*>(p.v + mem_off);
      const uint4 a = *km, c = *kc, d = *vm, e = *vc;
      *km = c;
      *kc = a;
      *vm = e;
      *vc = d;
    }
  }
}

}  // namespace

int launch_seed_kv(bool override_swap, void* k, void* v, const int32_t* seed_idx, int n_seeds, int B, int Hkv, int L,
                   int row_bytes, void* k_cache, void* v_cache, cudaStream_t stream) {
  if (n_seeds == 0) return 0;
  const long long bh = static_cast<long long>(B) * Hkv;
  const long long chunks = (n_seeds + kSlotsPerCta - 1) / kSlotsPerCta;
  if (bh > 0x7fffffffLL || chunks > 65535) return -2;
  KvParams p{static_cast<uint8_t*>(k), static_cast<uint8_t*>(v), seed_idx, n_seeds, L, Hkv, row_bytes / 16,
             static_cast<uint8_t*>(k_cache), static_cast<uint8_t*>(v_cache)};
  const dim3 grid(static_cast<unsigned>(bh), static_cast<unsigned>(chunks));
  cudaLaunchAttribute attr[1];
  const cudaLaunchConfig_t cfg = pdl_config(grid, dim3(kThreads), 0, stream, attr);
  const cudaError_t e = override_swap ? cudaLaunchKernelEx(&cfg, seed_kv_kernel<true>, p)
                                      : cudaLaunchKernelEx(&cfg, seed_kv_kernel<false>, p);
  return e == cudaSuccess && cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
