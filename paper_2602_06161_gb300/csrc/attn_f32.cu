// attn_f32.cu - two-view override attention in fp32 on CUDA cores.
//
// Section 5.1: every query attends once over the overridden memory K', V'
// (scale 1/sqrt(d)); a seed query i sees its diagonal entry restored to the
// masked-input pair (k_i, v_i). The kernel applies Appendix B's diagonal
// correction in exclusion form: the cached diagonal term (k'_i, v'_i) is left
// out of the online softmax, and the masked self term is merged into the
// running (max, sum, output) at the end. In exact arithmetic this equals the
// closed form o_i = (o_ovr_i - alpha_i v'_i + alpha_i e^delta_i v_i) / r_i,
// without its division by r_i (which tends to 0 as alpha_i -> 1 and
// delta_i -> -inf).
//
// One warp per query row; lane l holds elements l, l + 32, ... of q and o.
#include <math.h>

#include "kernels.cuh"
#include "ptx.cuh"
#include "route.cuh"

namespace cover {
namespace {

constexpr int kWarps = 4;

template <int D>
__global__ void __launch_bounds__(kWarps * 32)
    attn_f32_kernel(const float* __restrict__ q, const float* __restrict__ kc, const float* __restrict__ vc,
                    const float* __restrict__ km, const float* __restrict__ vm, const int32_t* __restrict__ seed_idx,
                    int n_seeds, int B, int Hq, int Hkv, int Lq, int L, int q0, float* __restrict__ out,
                    float* __restrict__ lse) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31;
  const long long row = static_cast<long long>(blockIdx.x) * kWarps + threadIdx.x / 32;
  const long long rows = static_cast<long long>(B) * Hq * Lq;
  if (row >= rows) return;
  const int i = q0 + static_cast<int>(row % Lq);   // memory position of this query row
  const int hq = static_cast<int>((row / Lq) % Hq);
  const int b = static_cast<int>(row / (static_cast<long long>(Lq) * Hq));
  const int hkv = hq / (Hq / Hkv);
  const float scale = 1.0f / sqrtf(static_cast<float>(D));

  // seed slot of this row: lowest s with seed_idx[b, s] == i
  int my_slot = kNoSlot;
  for (int s = lane; s < n_seeds; s += 32)
    if (seed_idx[static_cast<size_t>(b) * n_seeds + s] == i) my_slot = min(my_slot, s);
  for (int o = 16; o > 0; o >>= 1) my_slot = min(my_slot, __shfl_xor_sync(0xffffffffu, my_slot, o));
  const bool is_seed = my_slot != kNoSlot;

  float qr[E], acc[E];
  const float* qrow = q + row * D;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    qr[e] = qrow[lane + 32 * e];
    acc[e] = 0.0f;
  }
  const size_t kv_head = (static_cast<size_t>(b) * Hkv + hkv) * L * D;
  float m = -INFINITY, l = 0.0f;
  for (int j = 0; j < L; ++j) {
    if (is_seed && j == i) continue;   // cached diagonal term excluded
    const float* krow = kc + kv_head + static_cast<size_t>(j) * D;
    float dot = 0.0f;
#pragma unroll
    for (int e = 0; e < E; ++e) dot = fmaf(qr[e], krow[lane + 32 * e], dot);
    for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    const float s = dot * scale;
    const float m_new = fmaxf(m, s);
    const float a = expf(m - m_new);   // m = -inf on the first term gives 0
    const float p = expf(s - m_new);
    l = l * a + p;
    const float* vrow = vc + kv_head + static_cast<size_t>(j) * D;
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = acc[e] * a + p * vrow[lane + 32 * e];
    m = m_new;
  }
  if (is_seed) {
    // merge the masked-input self term (k_i, v_i)
    const size_t mrow = ((static_cast<size_t>(b) * Hkv + hkv) * n_seeds + my_slot) * D;
    float dot = 0.0f;
#pragma unroll
    for (int e = 0; e < E; ++e) dot = fmaf(qr[e], km[mrow + lane + 32 * e], dot);
    for (int o = 16; o > 0; o >>= 1) dot += __shfl_xor_sync(0xffffffffu, dot, o);
    const float s = dot * scale;
    const float m_new = fmaxf(m, s);
    const float a = (m == -INFINITY) ? 0.0f : expf(m - m_new);
    const float p = expf(s - m_new);
    l = l * a + p;
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = acc[e] * a + p * vm[mrow + lane + 32 * e];
    m = m_new;
  }
  const float inv = 1.0f / l;
#pragma unroll
  for (int e = 0; e < E; ++e) out[row * D + lane + 32 * e] = acc[e] * inv;
  if (lse != nullptr && lane == 0) lse[row] = m + logf(l);
}

}  // namespace

int launch_attn_f32(const AttnArgs& a, int* /*status*/, cudaStream_t stream) {
  const long long rows = static_cast<long long>(a.B) * a.Hq * a.Lq;
  const long long blocks = (rows + kWarps - 1) / kWarps;
  if (blocks > 0x7fffffffLL) return -2;
  const float* q = static_cast<const float*>(a.q);
  const float* kc = static_cast<const float*>(a.k_cached);
  const float* vc = static_cast<const float*>(a.v_cached);
  const float* km = static_cast<const float*>(a.k_seedmask);
  const float* vm = static_cast<const float*>(a.v_seedmask);
  float* out = static_cast<float*>(a.out);
  if (a.D == 64)
    attn_f32_kernel<64><<<static_cast<unsigned>(blocks), kWarps * 32, 0, stream>>>(
        q, kc, vc, km, vm, a.seed_idx, a.n_seeds, a.B, a.Hq, a.Hkv, a.Lq, a.L, a.q0, out, a.lse);
  else
    attn_f32_kernel<128><<<static_cast<unsigned>(blocks), kWarps * 32, 0, stream>>>(
        q, kc, vc, km, vm, a.seed_idx, a.n_seeds, a.B, a.Hq, a.Hkv, a.Lq, a.L, a.q0, out, a.lse);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
