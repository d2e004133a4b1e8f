// score_kernel.cu - fused per-position scoring over the vocabulary and top-k
// seed selection.
//
// Per row (one CTA per row, the row streamed once from HBM):
//   greedy token y_hat = argmax p and confidence c = max p       (Section 3)
//   entropy H = -sum p ln p                                       (Section 6.1)
//   uncertainty u = -log p(y), Score = u (1 + d_in)/(1 + d_out)   (Section 5.3)
// with p = softmax(logits) at temperature 1. Each thread keeps, for its share
// of the row, the running maximum m (exact bf16 compare, first index kept),
// Z = sum 2^t and S = sum t 2^t with t = x log2(e) - m log2(e), Kahan
// compensated; partials are re-referenced to the row maximum and summed in
// fp64. Then c = 1/Z, H = ln Z - ln(2) S / Z, u = ln Z - (x_y - m).
//
// Top-k (Section 5.3): the last CTA to finish a segment (sequence) - found
// with a self-resetting atomicInc counter per segment - sorts the segment's
// eligible rows by (score descending, index ascending) with a bitonic sort of
// 64-bit keys in shared memory and writes the first k.
#include <math.h>
#include <stdint.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace cover {
namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;
constexpr float kLog2e = 1.4426950408889634f;

struct RowAcc {
  float m;     // running maximum logit of this thread's elements
  int mi;      // first index where it occurs
  float mref;  // m * log2(e), the exponent reference
  float z, zc; // Kahan sum of 2^t and its compensation
  float s, sc; // Kahan sum of t 2^t and its compensation
};

__device__ __forceinline__ void kahan_add(float& sum, float& c, float x) {
  const float y = x - c;
  const float t = sum + y;
  c = (t - sum) - y;
  sum = t;
}

// Move the exponent reference to a larger maximum new_m.
__device__ __forceinline__ void raise_max(RowAcc& a, float new_m, int new_i) {
  const float new_ref = new_m * kLog2e;
  if (a.m != -INFINITY) {
    const float d = a.mref - new_ref;  // <= 0
    const float f = ex2_approx(d);
    const float z = a.z - a.zc;
    const float s = a.s - a.sc;
    a.s = f * fmaf(d, z, s);
    a.z = f * z;
  }
  a.zc = 0.0f;
  a.sc = 0.0f;
  a.m = new_m;
  a.mi = new_i;
  a.mref = new_ref;
}

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

__device__ __forceinline__ float bf16_to_f32(uint16_t h) { return __uint_as_float(static_cast<uint32_t>(h) << 16); }

// Accumulate 8 consecutive values (one 16-byte vector) whose first index is i0.
__device__ __forceinline__ void acc_vec8(RowAcc& a, const float (&x)[8]) {
  float e[8], te[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    const float t = fmaf(x[k], kLog2e, -a.mref);
    e[k] = ex2_approx(t);
    te[k] = t * e[k];
  }
  const float pz = ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
  const float ps = ((te[0] + te[1]) + (te[2] + te[3])) + ((te[4] + te[5]) + (te[6] + te[7]));
  kahan_add(a.z, a.zc, pz);
  kahan_add(a.s, a.sc, ps);
}

__device__ __forceinline__ void acc_scalar(RowAcc& a, float x, int idx) {
  if (x > a.m) raise_max(a, x, idx);
  const float t = fmaf(x, kLog2e, -a.mref);
  const float e = ex2_approx(t);
  kahan_add(a.z, a.zc, e);
  kahan_add(a.s, a.sc, t * e);
}

__device__ __forceinline__ void unpack8(const uint4& w, float (&x)[8]) {
  const uint32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    x[2 * k] = __uint_as_float(v[k] << 16);
    x[2 * k + 1] = __uint_as_float(v[k] & 0xffff0000u);
  }
}

__device__ __forceinline__ uint32_t order_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float order_key_inv(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

__global__ void __launch_bounds__(kThreads, 2)
    score_kernel(const uint16_t* __restrict__ logits, int V, int per_seq, const int32_t* __restrict__ cur_tok,
                 const float* __restrict__ d_in, const float* __restrict__ d_out,
                 const uint8_t* __restrict__ eligible, int topk, int sort_n, float* __restrict__ maxprob,
                 float* __restrict__ entropy, int32_t* __restrict__ argmax, float* __restrict__ score,
                 int32_t* __restrict__ topk_idx, float* __restrict__ topk_score, uint32_t* __restrict__ counters) {
  extern __shared__ uint64_t keys[];
  __shared__ float red_m[kWarps];
  __shared__ int red_i[kWarps];
  __shared__ double red_z[kWarps], red_s[kWarps];
  __shared__ float s_max;
  __shared__ int s_last;

  const int n = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const size_t row_off = static_cast<size_t>(n) * V;
  const uint16_t* row = logits + row_off;

  RowAcc a{-INFINITY, 0x7fffffff, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};

  // elements before the first 16-byte boundary of the row
  const int head = min(static_cast<int>((8 - (row_off & 7)) & 7), V);
  const int nvec = (V - head) / 8;
  const int tail0 = head + nvec * 8;
  if (tid < head) acc_scalar(a, bf16_to_f32(row[tid]), tid);

  const uint4* vrow = reinterpret_cast<const uint4*>(row + head);
  int v = tid;
  for (; v + (kUnroll - 1) * kThreads < nvec; v += kUnroll * kThreads) {
    uint4 w[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) w[u] = ld_stream(vrow + v + u * kThreads);
    float x[kUnroll][8];
    float bmax = -INFINITY;
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      unpack8(w[u], x[u]);
#pragma unroll
      for (int k = 0; k < 8; ++k) bmax = fmaxf(bmax, x[u][k]);
    }
    if (bmax > a.m) {
      int idx = 0x7fffffff;
#pragma unroll
      for (int u = kUnroll - 1; u >= 0; --u)
#pragma unroll
        for (int k = 7; k >= 0; --k)
          if (x[u][k] == bmax) idx = head + (v + u * kThreads) * 8 + k;
      raise_max(a, bmax, idx);
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) acc_vec8(a, x[u]);
  }
  for (; v < nvec; v += kThreads) {
    float x[8];
    unpack8(ld_stream(vrow + v), x);
    float bmax = -INFINITY;
#pragma unroll
    for (int k = 0; k < 8; ++k) bmax = fmaxf(bmax, x[k]);
    if (bmax > a.m) {
      int idx = 0x7fffffff;
#pragma unroll
      for (int k = 7; k >= 0; --k)
        if (x[k] == bmax) idx = head + v * 8 + k;
      raise_max(a, bmax, idx);
    }
    acc_vec8(a, x);
  }
  if (tail0 + tid < V) acc_scalar(a, bf16_to_f32(row[tail0 + tid]), tail0 + tid);

  // ---- row maximum and first index attaining it ----
  float m = a.m;
  int mi = a.mi;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, mi, o);
    if (m2 > m || (m2 == m && i2 < mi)) {
      m = m2;
      mi = i2;
    }
  }
  if (lane == 0) {
    red_m[warp] = m;
    red_i[warp] = mi;
  }
  __syncthreads();
  if (warp == 0) {
    m = lane < kWarps ? red_m[lane] : -INFINITY;
    mi = lane < kWarps ? red_i[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, mi, o);
      if (m2 > m || (m2 == m && i2 < mi)) {
        m = m2;
        mi = i2;
      }
    }
    if (lane == 0) {
      s_max = m;
      red_i[0] = mi;
    }
  }
  __syncthreads();
  const float M = s_max;
  const float Mref = M * kLog2e;

  // ---- partial sums re-referenced to the row maximum, summed in fp64 ----
  double zd = 0.0, sd = 0.0;
  if (a.m != -INFINITY) {
    const float d = a.mref - Mref;
    const float f = ex2_approx(d);
    const float z = a.z - a.zc;
    const float s = a.s - a.sc;
    zd = static_cast<double>(f * z);
    sd = static_cast<double>(f * fmaf(d, z, s));
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    zd += __shfl_xor_sync(0xffffffffu, zd, o);
    sd += __shfl_xor_sync(0xffffffffu, sd, o);
  }
  if (lane == 0) {
    red_z[warp] = zd;
    red_s[warp] = sd;
  }
  __syncthreads();
  if (tid == 0) {
    double Z = 0.0, S = 0.0;
    for (int w = 0; w < kWarps; ++w) {
      Z += red_z[w];
      S += red_s[w];
    }
    const int yhat = red_i[0];
    const double lnZ = log(Z);
    const double H = lnZ - 0.6931471805599453 * S / Z;
    const int y = cur_tok != nullptr ? cur_tok[n] : yhat;
    double u = nan("");                      // a current token outside [0, V) has no probability
    if (y >= 0 && y < V) {
      const double xy = (y == yhat) ? static_cast<double>(M) : static_cast<double>(bf16_to_f32(row[y]));
      u = lnZ - (xy - static_cast<double>(M));
    }
    const double din = d_in != nullptr ? static_cast<double>(d_in[n]) : 0.0;
    const double dout = d_out != nullptr ? static_cast<double>(d_out[n]) : 0.0;
    const float sc = static_cast<float>(u * (1.0 + din) / (1.0 + dout));
    maxprob[n] = static_cast<float>(1.0 / Z);
    entropy[n] = static_cast<float>(H);
    argmax[n] = yhat;
    score[n] = sc;
    s_last = 0;
    if (topk > 0) {
      __threadfence();
      const unsigned seg = static_cast<unsigned>(n / per_seq);
      const unsigned old = atomicInc(counters + seg, static_cast<unsigned>(per_seq - 1));
      s_last = (old == static_cast<unsigned>(per_seq - 1));
    }
  }
  __syncthreads();
  if (!s_last) return;

  // ---- last CTA of the segment: top-k by (score desc, index asc) ----
  __threadfence();
  const int seg = n / per_seq;
  const int base = seg * per_seq;
  for (int i = tid; i < sort_n; i += kThreads) {
    uint64_t key = 0;
    if (i < per_seq && (eligible == nullptr || eligible[base + i] != 0)) {
      const float sc = __ldcg(score + base + i);
      key = (static_cast<uint64_t>(order_key(sc)) << 32) | (0xffffffffu - static_cast<uint32_t>(i));
    }
    keys[i] = key;
  }
  __syncthreads();
  for (int k = 2; k <= sort_n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = tid; i < sort_n; i += kThreads) {
        const int p = i ^ j;
        if (p > i) {
          const uint64_t x = keys[i], y = keys[p];
          const bool desc = (i & k) == 0;
          if (desc ? (x < y) : (x > y)) {
            keys[i] = y;
            keys[p] = x;
          }
        }
      }
      __syncthreads();
    }
  }
  for (int t = tid; t < topk; t += kThreads) {
    const uint64_t key = keys[t];
    const bool valid = key != 0;
    topk_idx[static_cast<size_t>(seg) * topk + t] =
        valid ? static_cast<int32_t>(0xffffffffu - static_cast<uint32_t>(key)) : -1;
    if (topk_score != nullptr)
      topk_score[static_cast<size_t>(seg) * topk + t] =
          valid ? order_key_inv(static_cast<uint32_t>(key >> 32)) : -INFINITY;
  }
}

}  // namespace

int launch_score(const ScoreArgs& a, int* /*status*/, cudaStream_t stream) {
  const int per = a.N / a.n_seq;
  int sort_n = 1;
  while (sort_n < per) sort_n <<= 1;
  const size_t smem = a.topk > 0 ? sizeof(uint64_t) * static_cast<size_t>(sort_n) : 0;
  score_kernel<<<a.N, kThreads, smem, stream>>>(static_cast<const uint16_t*>(a.logits), a.V, per, a.cur_tok, a.d_in,
                                                a.d_out, a.eligible, a.topk, sort_n, a.maxprob, a.entropy, a.argmax,
                                                a.score, a.topk_idx, a.topk_score, a.counters);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
