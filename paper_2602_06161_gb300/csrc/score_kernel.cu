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
// compensated; partials are re-referenced to the row maximum and summed across
// the warp and then across the warps in fp32 with error-free TwoSum pairs.
// Then c = 1/Z, H = ln Z - ln(2) S / Z, u = ln Z - (x_y - m).
//
// Top-k (Section 5.3): the last CTA to finish a segment (sequence) - found
// with a self-resetting counter per segment, incremented with acquire-release
// semantics - takes the segment's k best eligible rows by (score descending,
// index ascending) on 64-bit keys: by rank when every row has its own thread,
// else by warp sorts and merges (k <= 32) or a bitonic sort in shared memory.
//
// Decision step (cover_score_decide_fwd, Sections 5.2, 3 and 5.3): the row
// pass keeps u of the current token and ln Z (= u of the greedy token) in a
// workspace; the last CTA of a segment then drafts the most confident masked
// rows above the threshold (at most B), applies Keep / Replace / ReMask to the
// previous seeds, scores the updated state, counts the scores above their mean
// (n_t pi_t), and selects ceil(sqrt(n_t pi_t)) new seeds among the rows that
// were not seeds and have ReMasks left, with the same 64-bit key sort.
//
// Two ways to stream a row:
//  * score_bulk_kernel (rows 16-byte aligned, V % 8 == 0): a producer warp
//    issues cp.async.bulk copies of 16 KB chunks into a 3-stage shared-memory
//    ring (mbarrier full / empty), 8 consumer warps reduce from shared memory;
//    bytes in flight do not cost registers, and 4 CTAs share an SM.
//  * score_kernel (any V): 16-byte non-allocating global loads, scalar head and
//    tail for rows that do not start on a 16-byte boundary.
#include <math.h>
#include <stdint.h>

#include <algorithm>

#include "context.cuh"
#include "kernels.cuh"
#include "ptx.cuh"

namespace cover {
namespace {

constexpr int kThreads = 512;              // register-load kernel
constexpr int kWarps = kThreads / 32;
constexpr int kUnroll = 4;
constexpr int kConsumerWarps = 8;          // bulk kernel: consumers + 1 producer warp
constexpr int kBulkThreads = (kConsumerWarps + 1) * 32;
constexpr int kChunkElems = 8192;          // 16 KB of bf16 per bulk copy
constexpr int kChunkBytes = kChunkElems * 2;
constexpr int kRingStages = 3;
constexpr int kVecPerThread = kChunkElems / 8 / (kConsumerWarps * 32);   // 4
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kMaxPerSeq = 4096;            // rows per segment (the entry points refuse more)
constexpr int kRowLoads = 4;                // rows whose state a thread loads at once (general paths)
constexpr int kRoundsMax = 32;              // selections up to this size by rounds or warp sorts (top_select)
constexpr int kRoundsFew = 8;               // selections up to this size by per-warp rounds (top_rounds)
constexpr int kMaxWarps = 16;               // every kernel here runs at most 512 threads

struct RowAcc {
  float m;     // running maximum logit of this thread's elements
  int mi;      // where m was first reached: the element's index (mu == 0), else the first index of
               // the batch that held it, mu vectors of 8 values a kernel-constant stride apart
  int mu;
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
__device__ __forceinline__ void raise_max(RowAcc& a, float new_m, int new_i, int new_u) {
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
  a.mu = new_u;
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

__device__ __forceinline__ void acc_scalar(RowAcc& a, float x, int idx) {
  if (x > a.m) raise_max(a, x, idx, 0);
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


// ---------------------------------------------------------------------------
// per-row finish (all threads of the CTA call it; NW = warps in the CTA)
// ---------------------------------------------------------------------------
struct RowOut {
  float M;      // row maximum
  int yhat;     // first index attaining it
  float Z;      // sum 2^t re-referenced to M log2(e)
  float q;      // (sum t 2^t) / Z
};

// a + b = s + e exactly (Knuth's TwoSum)
__device__ __forceinline__ void two_sum(float a, float b, float& s, float& e) {
  s = a + b;
  const float bb = s - a;
  e = (a - (s - bb)) + (b - bb);
}

// A thread's recorded batch is re-read from the row in global memory, in up to four vectors
// kStride elements apart; the loads are issued by the threads that hold their warp's maximum
// before the block-wide maximum is known, so their latency overlaps the reduction.
constexpr int kMaxBatch = 4;
static_assert(kVecPerThread <= kMaxBatch && kUnroll <= kMaxBatch, "batches hold at most four vectors");

template <int kStride>
__device__ __forceinline__ void load_batch(const RowAcc& a, const uint16_t* row, uint4 (&w)[kMaxBatch]) {
#pragma unroll
  for (int u = 0; u < kMaxBatch; ++u)
    if (u < a.mu) w[u] = ld_stream(reinterpret_cast<const uint4*>(row + a.mi + u * kStride));
}

// First index of the value M in the thread's recorded batch w.
template <int kStride>
__device__ __forceinline__ int first_index_of(const RowAcc& a, float M, const uint4 (&w)[kMaxBatch]) {
  if (a.mu == 0) return a.mi;
  int idx = 0x7fffffff;
#pragma unroll
  for (int u = kMaxBatch - 1; u >= 0; --u) {
    if (u >= a.mu) continue;
    float x[8];
    unpack8(w[u], x);
#pragma unroll
    for (int k = 7; k >= 0; --k)
      if (x[k] == M) idx = a.mi + u * kStride + k;
  }
  return idx;
}

template <int NW, int kStride>
__device__ __forceinline__ RowOut row_reduce(const RowAcc& a, const uint16_t* row, float* red_m, int* red_i,
                                             float2* red_z, float2* red_s) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  float m = a.m;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
  const bool cand = a.m == m && m != -INFINITY;   // may hold the row maximum
  uint4 w[kMaxBatch];
  if (cand) load_batch<kStride>(a, row, w);
  if (lane == 0) red_m[warp] = m;
  __syncthreads();
  float M = red_m[0];
#pragma unroll
  for (int i = 1; i < NW; ++i) M = fmaxf(M, red_m[i]);
  const float Mref = M * kLog2e;
  // partials re-referenced to the row maximum, summed across the warp in fp32
  // with error-free TwoSum pairs (value, rounding error), then across the warps
  // the same way by thread 0
  float z = 0.0f, ze = 0.0f, sv = 0.0f, se = 0.0f;
  if (a.m != -INFINITY) {
    const float d = a.mref - Mref;
    const float f = ex2_approx(d);
    const float zz = a.z - a.zc;
    const float ss = a.s - a.sc;
    z = f * zz;
    sv = f * fmaf(d, zz, ss);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float z2 = __shfl_xor_sync(0xffffffffu, z, o), ze2 = __shfl_xor_sync(0xffffffffu, ze, o);
    const float s2 = __shfl_xor_sync(0xffffffffu, sv, o), se2 = __shfl_xor_sync(0xffffffffu, se, o);
    float t = z + z2, bb = t - z;
    ze += ze2 + ((z - (t - bb)) + (z2 - bb));
    z = t;
    t = sv + s2;
    bb = t - sv;
    se += se2 + ((sv - (t - bb)) + (s2 - bb));
    sv = t;
  }
  // the threads holding the row maximum find its first index in their recorded batches
  const int mi = __reduce_min_sync(0xffffffffu, cand && a.m == M ? first_index_of<kStride>(a, M, w) : 0x7fffffff);
  if (lane == 0) {
    red_i[warp] = mi;
    red_z[warp] = make_float2(z, ze);
    red_s[warp] = make_float2(sv, se);
  }
  __syncthreads();
  RowOut r{M, 0x7fffffff, 0.0f, 0.0f};
  if (tid == 0) {
    int I = red_i[0];
#pragma unroll
    for (int w = 1; w < NW; ++w) I = min(I, red_i[w]);
    r.yhat = I;
    // the warps' (value, error) pairs added with TwoSum in fp32 (no fp64: this GPU's fp64 adds
    // have long latencies, and this runs at the end of every row with no copy in flight)
    float zh = red_z[0].x, zl = red_z[0].y, sh = red_s[0].x, sl = red_s[0].y;
#pragma unroll
    for (int w = 1; w < NW; ++w) {
      float t, e;
      two_sum(zh, red_z[w].x, t, e);
      zl += e + red_z[w].y;
      zh = t;
      two_sum(sh, red_s[w].x, t, e);
      sl += e + red_s[w].y;
      sh = t;
    }
    // S / Z with one correction step on the pairs: q = sh / zh, then the residual of
    // (sh + sl) - q (zh + zl) divided by zh
    const float q0 = sh / zh;
    const float res = fmaf(-q0, zh, sh) + (sl - q0 * zl);
    r.q = q0 + res / zh;
    r.Z = zh + zl;
  }
  return r;
}

// Thread 0 writes the row's outputs; returns (to thread 0) whether this CTA is
// the last of its segment to finish.
__device__ __forceinline__ bool row_write(const RowOut& r, int n, const uint16_t* row, int V, int per_seq,
                                          const int32_t* cur_tok, const float* d_in, const float* d_out, int topk,
                                          float* maxprob, float* entropy, int32_t* argmax, float* score,
                                          uint32_t* counters, float* ws_u = nullptr, float* ws_lnz = nullptr) {
  const float Zf = r.Z;
  const float lnZ = logf(Zf);
  const float H = lnZ - 0.6931471805599453f * r.q;
  const int y = cur_tok != nullptr ? cur_tok[n] : r.yhat;
  float u = __int_as_float(0x7fc00000);   // a current token outside [0, V) has no probability
  if (y >= 0 && y < V) {
    const float xy = (y == r.yhat) ? r.M : bf16_to_f32(row[y]);
    u = lnZ - (xy - r.M);
  }
  const float din = d_in != nullptr ? d_in[n] : 0.0f;
  const float dout = d_out != nullptr ? d_out[n] : 0.0f;
  maxprob[n] = 1.0f / Zf;
  entropy[n] = H;
  argmax[n] = r.yhat;
  if (ws_u != nullptr) {
    // decision step: the seed score is formed after the state update
    ws_u[n] = u;
    ws_lnz[n] = lnZ;
  } else {
    score[n] = u * (1.0f + din) / (1.0f + dout);
    if (topk <= 0) return false;
  }
  // The counter increment is a release (thread 0 wrote all of the row's results above) and an
  // acquire: the segment's last CTA, after its block barrier, reads the results of the others.
  const unsigned seg = static_cast<unsigned>(n / per_seq);
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.inc.u32 %0, [%1], %2;"
               : "=r"(old)
               : "l"(counters + seg), "r"(static_cast<unsigned>(per_seq - 1))
               : "memory");
  return old == static_cast<unsigned>(per_seq - 1);
}

struct ScoreParams {
  const uint16_t* logits;
  int V, per_seq;
  const int32_t* cur_tok;
  const float* d_in;
  const float* d_out;
  const uint8_t* eligible;
  int topk, sort_n;
  float* maxprob;
  float* entropy;
  int32_t* argmax;
  float* score;
  int32_t* topk_idx;
  float* topk_score;
  uint32_t* counters;
  int decide;          // 1: run the decision step instead of the top-k
  DecideArgs dec;
};

// Descending bitonic sort of n (a power of two) 64-bit keys in shared memory;
// all threads of the CTA call it.
__device__ __forceinline__ void bitonic_sort_desc(uint64_t* keys, int n) {
  const int tid = threadIdx.x, nt = blockDim.x;
  for (int k = 2; k <= n; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = tid; i < n; i += nt) {
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
}

// Sum over the CTA (blockDim a multiple of 32); every thread gets the total,
// added in the same order everywhere. scratch: 32 entries.
template <typename T>
__device__ __forceinline__ T block_sum(T v, T* scratch) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if (lane == 0) scratch[warp] = v;
  __syncthreads();
  T t = 0;
  for (int w = 0; w < nw; ++w) t += scratch[w];
  return t;
}

// A finite fp32 score as a 64-bit fixed-point integer on the binade of the segment's largest
// score (biased exponent emax): s 2^(26 - E), |result| < 2^50. Exact for a score within a factor
// 2^26 of the largest; a smaller one is truncated toward zero. Sums of up to 4096 of them and
// their products with counts up to 4096 stay below 2^62, so the mean test n_t s > sum s is an
// exact integer comparison on these values.
__device__ __forceinline__ long long fixed_of(float s, uint32_t emax) {
  const uint32_t bits = __float_as_uint(s);
  const uint32_t eb = (bits >> 23) & 0xffu;
  // s = m 2^(eb - 150) (m with its leading bit; a denormal has eb 0 and exponent 1 - 150)
  const uint32_t m = eb != 0u ? ((bits & 0x7fffffu) | 0x800000u) : (bits & 0x7fffffu);
  const int shift = static_cast<int>(eb == 0u ? 1u : eb) - static_cast<int>(emax) + 26;
  const long long mag = shift >= 0 ? (static_cast<long long>(m) << shift) : (shift > -25 ? (m >> -shift) : 0);
  return (bits >> 31) ? -mag : mag;
}

// key of row i ordered by value descending, then index ascending; 0 = no row
__device__ __forceinline__ uint64_t rank_key(float v, int i) {
  return (static_cast<uint64_t>(order_key(v)) << 32) | (0xffffffffu - static_cast<uint32_t>(i));
}
__device__ __forceinline__ int rank_key_row(uint64_t key) {
  return static_cast<int>(0xffffffffu - static_cast<uint32_t>(key));
}

// Descending bitonic sorts of G independent sets of 32 keys across the warp (key[g]: lane t's
// key of set g), by shuffles; the G sets go through the network together.
template <int G>
__device__ __forceinline__ void warp_sort_desc(uint64_t (&key)[G], int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
    const bool desc = (lane & size) == 0;
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const bool take_max = ((lane & stride) == 0) == desc;
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const uint64_t other = __shfl_xor_sync(0xffffffffu, key[g], stride);
        key[g] = take_max ? (key[g] > other ? key[g] : other) : (key[g] < other ? key[g] : other);
      }
    }
  }
}
__device__ __forceinline__ uint64_t warp_sort_desc(uint64_t key, int lane) {
  uint64_t k1[1] = {key};
  warp_sort_desc<1>(k1, lane);
  return k1[0];
}

// a[g] becomes the 32 largest of the descending lists a[g] and b[g] (lane t holds the t-th of
// each), descending: the larger of a[t] and b[31 - t] is a bitonic sequence holding them, which
// the half-cleaners of strides 16 .. 1 put in order. The G merges go through together.
template <int G>
__device__ __forceinline__ void warp_merge_desc(uint64_t (&a)[G], const uint64_t (&b)[G], int lane) {
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const uint64_t br = __shfl_sync(0xffffffffu, b[g], 31 - lane);
    a[g] = a[g] > br ? a[g] : br;
  }
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) {
    const bool take_max = (lane & stride) == 0;
#pragma unroll
    for (int g = 0; g < G; ++g) {
      const uint64_t other = __shfl_xor_sync(0xffffffffu, a[g], stride);
      a[g] = take_max ? (a[g] > other ? a[g] : other) : (a[g] < other ? a[g] : other);
    }
  }
}

// Number of entries of the descending list l[0 .. 32) larger than x (x not in the list).
__device__ __forceinline__ int count_above(const uint64_t* l, uint64_t x) {
  int c = 0;
#pragma unroll
  for (int step = 32; step > 0; step >>= 1)
    if (c + step <= 32 && l[c + step - 1] > x) c += step;
  return c;
}

// Largest of the warp's 64-bit values (two 32-bit reductions: the high words, then the low
// words of the lanes that hold the largest high word).
__device__ __forceinline__ uint64_t warp_max_u64(uint64_t x) {
  const uint32_t hi = __reduce_max_sync(0xffffffffu, static_cast<uint32_t>(x >> 32));
  const uint32_t lo = __reduce_max_sync(0xffffffffu, static_cast<uint32_t>(x >> 32) == hi ? static_cast<uint32_t>(x) : 0u);
  return (static_cast<uint64_t>(hi) << 32) | lo;
}

// The k largest (k <= kRoundsFew) of the n keys in shared memory (keys are distinct, 0 = none),
// in descending order: out[t] gets the t-th (0 once the nonzero keys run out). Each warp takes
// its own k largest by k rounds of a warp-wide maximum below the previous round's (no block
// barrier per round), over the keys its lanes read (i = tid, tid + blockDim, ...); a key can be
// among the k largest only if it is among its warp's, so ranking the warps' lists against each
// other is exact below k. All threads call it with the same k.
__device__ __forceinline__ void top_rounds(const uint64_t* keys, int n, int k, uint64_t* out) {
  __shared__ uint64_t s_list[kMaxWarps * kRoundsFew];
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, warp = tid >> 5, nw = nt >> 5;
  if (k <= 0) return;
  uint64_t prev = ~0ull;
  for (int t = 0; t < k; ++t) {
    uint64_t m = 0;
    for (int i = tid; i < n; i += nt) {
      const uint64_t x = keys[i];
      if (x < prev && x > m) m = x;
    }
    prev = warp_max_u64(m);
    if (lane == 0) s_list[warp * k + t] = prev;   // 0 once the warp's keys run out
  }
  const int nl = nw * k;
  __syncthreads();
  const uint64_t key = tid < nl ? s_list[tid] : 0;
  const int listed = __syncthreads_count(key != 0);
  if (key != 0) {
    int r = 0;
    for (int j = 0; j < nl; ++j) r += s_list[j] > key ? 1 : 0;
    if (r < k) out[r] = key;
  }
  for (int t = min(listed, k) + tid; t < k; t += nt) out[t] = 0;
  __syncthreads();
}

// The k largest (k <= 32) of the n keys in shared memory (distinct, 0 = none), in descending
// order: out[t] gets the t-th (0 once the nonzero keys run out). Each warp keeps the 32 largest
// keys it has read in registers (lane t: the t-th). It reads four sets of 32 keys at a time
// (every (warps)-th set of the array), sorts them together, merges them pairwise and folds the
// result into its list, skipping the work when no key passes the list's k-th. A key can be
// among the k largest only if it is among its warp's, so the warps' lists decide the result:
// a listed key's rank is its position in its own list plus the number of larger keys in each
// other list (a binary search, the lists being sorted), exact below k. The lists are staged in
// keys[0 .. 32 * warps), which n >= blockDim.x guarantees; the keys are not read afterwards.
// All threads call it with the same k.
__device__ __forceinline__ void top_warps(uint64_t* keys, int n, int k, uint64_t* out) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  if (k <= 0) return;
  constexpr int kSets = 4;
  uint64_t top[1] = {0};
  for (int j0 = warp * 32 + lane; j0 - lane < n; j0 += kSets * nw * 32) {
    uint64_t b[kSets];
#pragma unroll
    for (int g = 0; g < kSets; ++g) {
      const int j = j0 + g * nw * 32;
      b[g] = j < n ? keys[j] : 0;
    }
    const uint64_t kth = __shfl_sync(0xffffffffu, top[0], k - 1);
    if (!__any_sync(0xffffffffu, b[0] > kth || b[1] > kth || b[2] > kth || b[3] > kth)) continue;
    warp_sort_desc<kSets>(b, lane);
    uint64_t p[2] = {b[0], b[2]};
    const uint64_t q[2] = {b[1], b[3]};
    warp_merge_desc<2>(p, q, lane);
    const uint64_t p1[1] = {p[1]};
    uint64_t p0[1] = {p[0]};
    warp_merge_desc<1>(p0, p1, lane);
    warp_merge_desc<1>(top, p0, lane);
  }
  __syncthreads();   // every warp is done reading the keys
  keys[warp * 32 + lane] = lane < k ? top[0] : 0;
  const int published = __syncthreads_count(lane < k && top[0] != 0);
  if (lane < k && top[0] != 0) {
    int r = lane;
#pragma unroll 4
    for (int w = 0; w < nw; ++w)
      if (w != warp) r += count_above(keys + w * 32, top[0]);
    if (r < k) out[r] = top[0];
  }
  for (int t = min(published, k) + tid; t < k; t += blockDim.x) out[t] = 0;
  __syncthreads();
}

// The k largest (k <= kRoundsMax) of n keys in shared memory into out, by rounds for a few keys
// and by warp sorts otherwise; the first 32 * warps keys may be overwritten.
__device__ __forceinline__ void top_select(uint64_t* keys, int n, int k, uint64_t* out) {
  if (k <= kRoundsFew)
    top_rounds(keys, n, k, out);
  else
    top_warps(keys, n, k, out);
}

// Sections 5.2 and 3, run by the last CTA of a segment: drafting and the
// revision of the previous seeds. Updates tok, remask_cnt, flags (bit 1 marks
// the rows drafted in this step; a drafted row loses bit 0) and ws_u (the
// uncertainty of each row's updated token: ln Z for drafted and replaced rows).
// Rows written by other CTAs are read through L2 (__ldcg). The drafting sort
// runs only when more rows pass the threshold than the budget allows.
__device__ void segment_update(uint64_t* keys, int seg, int per_seq, int sort_n, const ScoreParams& P) {
  __shared__ unsigned long long s_fallback;
  __shared__ uint32_t s_draft_bits[kMaxPerSeq / 32];
  __shared__ int s_ri[32];
  __shared__ int s_cnt[3][32];
  __shared__ uint64_t s_sel[kRoundsMax];
  const DecideArgs& d = P.dec;
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, warp = tid >> 5, nw = nt >> 5;
  const int base = seg * per_seq;
  if (tid == 0) s_fallback = ~0ull;
  __syncthreads();

  // Section 5.2 drafting: masked rows in the allowed set whose confidence exceeds tau. Each
  // thread loads the state of kRowLoads rows before it uses any of it (the loads of a batch
  // overlap instead of waiting on one another's results).
  int ncand = 0;
  uint64_t fb_min = ~0ull;   // the thread's lowest (entropy, index) key among allowed rows
  for (int i0 = tid; i0 < per_seq; i0 += kRowLoads * nt) {
    bool allowed[kRowLoads];
    float c[kRowLoads], h[kRowLoads];
#pragma unroll
    for (int u = 0; u < kRowLoads; ++u) {
      const int i = i0 + u * nt;
      const bool in = i < per_seq;
      const int n = base + (in ? i : 0);
      allowed[u] = in && d.tok[n] == d.mask_id & (d.draft_ok == nullptr || d.draft_ok[n] != 0);
      c[u] = __ldcg(P.maxprob + n);
      h[u] = __ldcg(P.entropy + n);
    }
#pragma unroll
    for (int u = 0; u < kRowLoads; ++u) {
      if (!allowed[u]) continue;
      if (c[u] > d.tau) ++ncand;
      // lowest entropy, then lowest index
      const uint64_t fb = (static_cast<uint64_t>(order_key(h[u])) << 32) | static_cast<uint32_t>(i0 + u * nt);
      fb_min = fb < fb_min ? fb : fb_min;
    }
  }
  if (d.min_one) {
    // one shared-memory atomic per warp (a 64-bit minimum by two 32-bit reductions)
    const uint32_t hi = __reduce_min_sync(0xffffffffu, static_cast<uint32_t>(fb_min >> 32));
    const uint32_t lo =
        __reduce_min_sync(0xffffffffu, static_cast<uint32_t>(fb_min >> 32) == hi ? static_cast<uint32_t>(fb_min) : ~0u);
    const uint64_t wmin = (static_cast<uint64_t>(hi) << 32) | lo;   // ~0 only when no lane has a row
    if (lane == 0 && wmin != ~0ull) atomicMin(&s_fallback, static_cast<unsigned long long>(wmin));
  }
  ncand = block_sum(ncand, s_ri);
  const bool all_cand = ncand <= d.budget;   // every row above tau is drafted
  int n_drafted = min(ncand, d.budget);
  const bool fallback = n_drafted == 0 && d.min_one && s_fallback != ~0ull;
  if (!all_cand) {
    // more candidates than the budget: the `budget` most confident (ties to the lower index)
    for (int i0 = tid; i0 < sort_n; i0 += kRowLoads * nt) {
      bool allowed[kRowLoads];
      float c[kRowLoads];
#pragma unroll
      for (int u = 0; u < kRowLoads; ++u) {
        const int i = i0 + u * nt;
        const bool in = i < per_seq;
        const int n = base + (in ? i : 0);
        allowed[u] = in && d.tok[n] == d.mask_id & (d.draft_ok == nullptr || d.draft_ok[n] != 0);
        c[u] = __ldcg(P.maxprob + n);
      }
#pragma unroll
      for (int u = 0; u < kRowLoads; ++u) {
        const int i = i0 + u * nt;
        if (i < sort_n) keys[i] = allowed[u] && c[u] > d.tau ? rank_key(c[u], i) : 0;
      }
    }
    __syncthreads();
    if (n_drafted <= kRoundsMax)
      top_select(keys, sort_n, n_drafted, s_sel);
    else
      bitonic_sort_desc(keys, sort_n);
  }
  // the drafted rows, marked for the pass below when they were selected (more candidates than
  // the budget) or are the fallback row; with every candidate drafted the pass decides itself
  if (!all_cand || fallback) {
    for (int w = tid; w < kMaxPerSeq / 32; w += nt) s_draft_bits[w] = 0u;
    __syncthreads();
    const uint64_t* picked = n_drafted <= kRoundsMax ? s_sel : keys;
    for (int t = tid; t < (fallback ? 1 : n_drafted); t += nt) {
      const int i = fallback ? static_cast<int>(static_cast<uint32_t>(s_fallback)) : rank_key_row(picked[t]);
      atomicOr(&s_draft_bits[i >> 5], 1u << (i & 31));
    }
    __syncthreads();
  }
  const bool marked = !all_cand || fallback;
  if (fallback) n_drafted = 1;

  // Section 5.2 revision of the previous seeds, Section 3 state update
  int kept = 0, replaced = 0, remasked = 0;
  for (int i0 = tid; i0 < per_seq; i0 += kRowLoads * nt) {
    int y[kRowLoads], yh[kRowLoads];
    uint32_t fl[kRowLoads], rc[kRowLoads];
    bool ok[kRowLoads];
    float c[kRowLoads], lz[kRowLoads];
#pragma unroll
    for (int u = 0; u < kRowLoads; ++u) {
      const int i = i0 + u * nt;
      const int n = base + (i < per_seq ? i : 0);
      y[u] = d.tok[n];
      fl[u] = d.flags[n];
      rc[u] = d.remask_cnt[n];
      ok[u] = d.draft_ok == nullptr || d.draft_ok[n] != 0;
      c[u] = __ldcg(P.maxprob + n);
      yh[u] = __ldcg(P.argmax + n);
      lz[u] = __ldcg(d.ws_lnz + n);
    }
#pragma unroll
    for (int u = 0; u < kRowLoads; ++u) {
      const int i = i0 + u * nt;
      if (i >= per_seq) continue;
      const int n = base + i;
      const bool drafted = marked ? (s_draft_bits[i >> 5] >> (i & 31)) & 1u
                                  : y[u] == d.mask_id && ok[u] && c[u] > d.tau;
      if (drafted) {
        // a drafted row takes its greedy token, whose uncertainty is ln Z
        d.tok[n] = yh[u];
        d.ws_u[n] = lz[u];
        d.flags[n] = static_cast<uint8_t>((fl[u] & ~1u) | 2u);
      } else if ((fl[u] & 1u) != 0 && y[u] != d.mask_id) {
        if (yh[u] == y[u]) {
          ++kept;
        } else if (c[u] > d.tau) {
          ++replaced;
          d.tok[n] = yh[u];
          d.ws_u[n] = lz[u];
        } else {
          ++remasked;
          d.tok[n] = d.mask_id;
          d.remask_cnt[n] = static_cast<uint8_t>(min(rc[u] + 1u, 255u));
        }
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    kept += __shfl_xor_sync(0xffffffffu, kept, o);
    replaced += __shfl_xor_sync(0xffffffffu, replaced, o);
    remasked += __shfl_xor_sync(0xffffffffu, remasked, o);
  }
  if (lane == 0) {
    s_cnt[0][warp] = kept;
    s_cnt[1][warp] = replaced;
    s_cnt[2][warp] = remasked;
  }
  __syncthreads();
  if (tid == 0 && d.stats != nullptr) {
    kept = replaced = remasked = 0;
    for (int w = 0; w < nw; ++w) {
      kept += s_cnt[0][w];
      replaced += s_cnt[1][w];
      remasked += s_cnt[2][w];
    }
    int32_t* st = d.stats + static_cast<size_t>(seg) * kDecideStats;
    st[0] = n_drafted;
    st[1] = kept;
    st[2] = replaced;
    st[3] = remasked;
  }
}

// Section 5.3 on the updated state of one segment (all threads of the CTA):
// seed score of every unmasked row, the adaptive revision rate, and the
// selection among rows that were not previous seeds and have ReMasks left.
// Clears flag bits 0 and 1 everywhere, then sets bit 0 on the new seeds.
// keys: sort_n 64-bit slots of shared memory followed by sort_n floats.
__device__ void segment_select(uint64_t* keys, int seg, int per_seq, int sort_n, const DecideArgs& d,
                               const float* d_in, const float* d_out, float* score) {
  __shared__ int s_ri[32];
  __shared__ int s_nt[32];
  __shared__ uint32_t s_em[32];
  __shared__ long long s_fx[32];
  __shared__ uint64_t s_sel[kRoundsMax];
  const int tid = threadIdx.x, nt = blockDim.x, lane = tid & 31, warp = tid >> 5, nw = nt >> 5;
  const int base = seg * per_seq;
  float* sscore = reinterpret_cast<float*>(keys + sort_n);   // per-row seed score

  int n_t = 0;
  uint32_t emax = 0;   // largest biased exponent of the finite scores
  for (int i0 = tid; i0 < sort_n; i0 += kRowLoads * nt) {
    // the state of kRowLoads rows, loaded before any of it is used
    uint32_t fl[kRowLoads], rc[kRowLoads];
    int tk[kRowLoads];
    float din[kRowLoads], dout[kRowLoads], uu[kRowLoads];
#pragma unroll
    for (int u = 0; u < kRowLoads; ++u) {
      const int i = i0 + u * nt;
      const int n = base + (i < per_seq ? i : 0);
      fl[u] = d.flags[n];
      rc[u] = d.remask_cnt[n];
      tk[u] = d.tok[n];
      din[u] = d_in != nullptr ? d_in[n] : 0.0f;
      dout[u] = d_out != nullptr ? d_out[n] : 0.0f;
      uu[u] = __ldcg(d.ws_u + n);
    }
#pragma unroll
    for (int u = 0; u < kRowLoads; ++u) {
      const int i = i0 + u * nt;
      if (i >= sort_n) continue;
      uint64_t key = 0;
      if (i < per_seq) {
        const int n = base + i;
        float s = -INFINITY;
        if (tk[u] != d.mask_id) {
          const float sc = uu[u] * (1.0f + din[u]) / (1.0f + dout[u]);
          if (isfinite(sc)) {
            s = sc;
            ++n_t;
            emax = max(emax, (__float_as_uint(sc) >> 23) & 0xffu);
            if ((fl[u] & 1u) == 0 && static_cast<int>(rc[u]) < d.remask_budget) key = rank_key(sc, i);
          }
        }
        score[n] = s;
        sscore[i] = s;
        d.flags[n] = static_cast<uint8_t>(fl[u] & ~3u);
      }
      keys[i] = key;
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) n_t += __shfl_xor_sync(0xffffffffu, n_t, o);
  emax = __reduce_max_sync(0xffffffffu, emax);
  if (lane == 0) {
    s_nt[warp] = n_t;
    s_em[warp] = emax;
  }
  __syncthreads();
  n_t = 0;
  emax = 0;
  for (int w = 0; w < nw; ++w) {
    n_t += s_nt[w];
    emax = max(emax, s_em[w]);
  }
  // the sum of the scores, exact in fixed point (fixed_of)
  long long part = 0;
  for (int i = tid; i < per_seq; i += nt) {
    const float s = sscore[i];
    if (s != -INFINITY) part += fixed_of(s, emax);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) part += __shfl_xor_sync(0xffffffffu, part, o);
  if (lane == 0) s_fx[warp] = part;
  __syncthreads();
  long long total = 0;
  for (int w = 0; w < nw; ++w) total += s_fx[w];

  // adaptive revision rate: n_t pi_t = #{ s_j > mean } = #{ n_t s_j > sum s }
  int above = 0;
  for (int i = tid; i < per_seq; i += nt) {
    const float s = sscore[i];
    if (s != -INFINITY && static_cast<long long>(n_t) * fixed_of(s, emax) > total) ++above;
  }
  above = block_sum(above, s_ri);
  int k = 0;
  while (k * k < above) ++k;   // ceil(sqrt(n_t pi_t))
  k = min(k, d.max_seeds);

  // the k best eligible rows (keys written above)
  const uint64_t* best = keys;
  if (k > 0 && k <= kRoundsMax) {
    top_select(keys, sort_n, k, s_sel);
    best = s_sel;
  } else if (k > 0) {
    bitonic_sort_desc(keys, sort_n);
  }
  int chosen = 0;
  for (int t = tid; t < d.max_seeds; t += nt) {
    int pos = -1;
    if (t < k && t < sort_n && best[t] != 0) {
      const int i = rank_key_row(best[t]);
      pos = d.pos0 + i;
      d.flags[base + i] = static_cast<uint8_t>(d.flags[base + i] | 1u);
      ++chosen;
    }
    d.seed_idx[static_cast<size_t>(seg) * d.max_seeds + t] = pos;
  }
  chosen = block_sum(chosen, s_ri);
  if (tid == 0) {
    d.n_seeds[seg] = chosen;
    if (d.stats != nullptr) {
      int32_t* st = d.stats + static_cast<size_t>(seg) * kDecideStats;
      st[4] = n_t;
      st[5] = above;
    }
  }
}

// ---------------------------------------------------------------------------
// Fast path of the per-segment work when the segment has at most one row per
// thread of the CTA (per_seq <= blockDim.x): row i belongs to thread i, which
// loads the row's state once (independent loads, one round trip to L2), keeps
// it in registers and writes it back once. Each count takes one barrier
// (__syncthreads_count). A top selection ranks every candidate against the
// other candidates' keys in shared memory: its rank is the number of larger
// keys, so the row of rank r < k is the (r+1)-th best and fills slot r. Keys
// embed the row index, so they are distinct and the result is the general
// path's (the sort or the warp sorts) exactly.
// ---------------------------------------------------------------------------

// Rank of x among keys[0 .. n) (16-byte aligned): the number of larger keys, counted only while
// it can still be below k. All threads read the same entries at the same time (shared-memory
// broadcasts, two keys per load); a warp stops once every lane's count has reached k (x = 0,
// no key, counts as already there), and the result is then some value >= k.
__device__ __forceinline__ int rank_below(const uint64_t* keys, int n, uint64_t x, int k) {
  int r = x != 0 ? 0 : k;
  const ulonglong2* k2 = reinterpret_cast<const ulonglong2*>(keys);
  int j = 0;
  for (; j + 32 <= n; j += 32) {
    if (__all_sync(0xffffffffu, r >= k)) return r;
#pragma unroll
    for (int q = 0; q < 16; ++q) {
      const ulonglong2 y = k2[(j >> 1) + q];
      r += (y.x > x ? 1 : 0) + (y.y > x ? 1 : 0);
    }
  }
  for (; j < n; ++j) r += keys[j] > x ? 1 : 0;
  return r;
}


// The k largest (k <= 32) of the CTA's keys, one per thread (distinct, 0 = none). Each warp sorts
// its keys and publishes its k largest in cand[warp * k ..]; a key can be among the CTA's k
// largest only if it is among its warp's, and the number of larger published keys is its rank,
// exact while below k (a warp publishes at most k). Returns, for the key this lane holds after
// its warp's sort (*held), its slot 0 .. k-1 among the CTA's k largest, else -1. All threads of
// the CTA call it; cand holds blockDim.x keys.
__device__ __forceinline__ int top_small(uint64_t key, int k, uint64_t* cand, uint64_t* held) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  const uint64_t sorted = warp_sort_desc(key, lane);
  if (lane < k) cand[warp * k + lane] = sorted;
  __syncthreads();
  int slot = -1;
  if (lane < k && sorted != 0) {
    int r = 0;
    for (int j = 0; j < nw * k; ++j) r += cand[j] > sorted ? 1 : 0;
    if (r < k) slot = r;
  }
  *held = sorted;
  return slot;
}

// Section 5.3 on the updated state, one row per thread (see segment_select for the
// general path): seed score, n_t and the mean, n_t pi_t = #{n_t s_j > sum s}, and
// the selection of ceil(sqrt(n_t pi_t)) rows by rank. Writes score, flags and the
// segment's seed list, count and stats[4..5].
__device__ void select_fast(uint64_t* keys, int seg, int per_seq, const DecideArgs& d, bool in, int tok,
                            uint32_t& fl, uint32_t rc, float u, float din, float dout, float* score) {
  __shared__ long long s_fx[32];
  __shared__ uint32_t s_emax;
  __shared__ int s_elig;
  __shared__ uint8_t s_mark[512];   // blockDim <= 512
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, nw = blockDim.x >> 5;
  const int n = seg * per_seq + tid;
  float sc = -INFINITY;
  bool valid = false;
  uint64_t key = 0;
  if (in && tok != d.mask_id) {
    const float v = u * (1.0f + din) / (1.0f + dout);
    if (isfinite(v)) {
      sc = v;
      valid = true;
      if ((fl & 1u) == 0 && static_cast<int>(rc) < d.remask_budget) key = rank_key(v, tid);
    }
  }
  // n_t pi_t = #{n_t s_j > sum s} in exact integer arithmetic on the scores' fixed-point values
  // (fixed_of); a score too small to be exact lies far below the mean, and the sum's error
  // stays below n_t units, 2^-50 of the largest score. This GPU's fp64 units have long
  // latencies, so no fp64 is used here.
  const uint32_t sbits = __float_as_uint(sc);
  const uint32_t ebias = valid ? ((sbits >> 23) & 0xffu) : 0u;
  const uint32_t emax_w = __reduce_max_sync(0xffffffffu, ebias);
  const uint32_t eb = __ballot_sync(0xffffffffu, key != 0);
  if (tid == 0) {
    s_elig = 0;
    s_emax = 0u;
  }
  if (in) keys[tid] = key;
  __syncthreads();
  if (lane == 0) {
    atomicMax(&s_emax, emax_w);
    if (eb != 0u) atomicAdd(&s_elig, __popc(eb));
  }
  const int n_t = __syncthreads_count(valid);
  const long long fx = valid ? fixed_of(sc, s_emax) : 0;
  long long tot = fx;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
  if (lane == 0) s_fx[warp] = tot;
  __syncthreads();
  long long total = 0;
  for (int w = 0; w < nw; ++w) total += s_fx[w];
  const bool is_above = valid && static_cast<long long>(n_t) * fx > total;
  const int above = __syncthreads_count(is_above);
  int k = 0;
  while (k * k < above) ++k;   // ceil(sqrt(n_t pi_t))
  k = min(k, d.max_seeds);
  const int chosen = min(k, s_elig);
  bool chosen_row = false;
  if (k > 0 && k <= 32) {
    // few seeds: per-warp sorts and the ranks of the published keys; the lane holding a chosen
    // key writes its slot and marks the row for its owner thread
    uint64_t held;
    if (in) s_mark[tid] = 0;
    const int slot = top_small(key, k, keys, &held);
    if (slot >= 0) {
      const int row = rank_key_row(held);
      d.seed_idx[static_cast<size_t>(seg) * d.max_seeds + slot] = d.pos0 + row;
      s_mark[row] = 1;
    }
    __syncthreads();
    chosen_row = in && s_mark[tid] != 0;
  } else if (k > 0) {
    const int r = rank_below(keys, per_seq, key, k);
    if (key != 0 && r < k) {
      chosen_row = true;
      d.seed_idx[static_cast<size_t>(seg) * d.max_seeds + r] = d.pos0 + tid;
    }
  }
  if (in) {
    score[n] = sc;
    fl = (fl & ~3u) | (chosen_row ? 1u : 0u);
  }
  for (int t = chosen + tid; t < d.max_seeds; t += blockDim.x) d.seed_idx[static_cast<size_t>(seg) * d.max_seeds + t] = -1;
  if (tid == 0) {
    d.n_seeds[seg] = chosen;
    if (d.stats != nullptr) {
      int32_t* st = d.stats + static_cast<size_t>(seg) * kDecideStats;
      st[4] = n_t;
      st[5] = above;
    }
  }
}

// One segment's decision step, one row per thread (see segment_update and
// segment_select for the general path).
__device__ void decide_fast(uint64_t* keys, int seg, int per_seq, const ScoreParams& P) {
  __shared__ unsigned long long s_fallback;
  __shared__ int s_cnt[3];
  __shared__ uint8_t s_draft[512];   // blockDim <= 512
  const DecideArgs& d = P.dec;
  const int tid = threadIdx.x, lane = tid & 31;
  const bool in = tid < per_seq;
  const int n = seg * per_seq + tid;
  const bool select = d.phase == 0;
  // the row's whole state, in one round trip (other CTAs' results through L2)
  int tok = 0, yhat = 0;
  uint32_t fl = 0, rc = 0;
  float c = 0.0f, H = 0.0f, u = 0.0f, lnz = 0.0f, din = 0.0f, dout = 0.0f;
  bool ok_draft = false;
  if (in) {
    tok = d.tok[n];
    fl = d.flags[n];
    rc = d.remask_cnt[n];
    ok_draft = d.draft_ok == nullptr || d.draft_ok[n] != 0;
    c = __ldcg(P.maxprob + n);
    H = __ldcg(P.entropy + n);
    yhat = __ldcg(P.argmax + n);
    u = __ldcg(d.ws_u + n);
    lnz = __ldcg(d.ws_lnz + n);
    if (select) {
      din = P.d_in != nullptr ? P.d_in[n] : 0.0f;
      dout = P.d_out != nullptr ? P.d_out[n] : 0.0f;
    }
  }
  if (tid == 0) {
    s_fallback = ~0ull;
    s_cnt[0] = s_cnt[1] = s_cnt[2] = 0;
  }
  __syncthreads();

  // Section 5.2 drafting: masked rows in the allowed set whose confidence exceeds tau
  const bool allowed = in && tok == d.mask_id && ok_draft;
  const bool cand = allowed && c > d.tau;
  if (d.min_one) {
    // lowest entropy, then lowest index: a warp minimum (two 32-bit reductions), then one
    // shared-memory atomic per warp
    const uint64_t fb = allowed ? (static_cast<uint64_t>(order_key(H)) << 32) | static_cast<uint32_t>(tid) : ~0ull;
    const uint32_t hi = __reduce_min_sync(0xffffffffu, static_cast<uint32_t>(fb >> 32));
    const uint32_t lo =
        __reduce_min_sync(0xffffffffu, static_cast<uint32_t>(fb >> 32) == hi ? static_cast<uint32_t>(fb) : ~0u);
    const uint64_t wmin = (static_cast<uint64_t>(hi) << 32) | lo;   // ~0 only when no lane has a row
    if (lane == 0 && wmin != ~0ull) atomicMin(&s_fallback, static_cast<unsigned long long>(wmin));
  }
  const int ncand = __syncthreads_count(cand);
  const bool all_cand = ncand <= d.budget;   // every row above tau is drafted
  int n_drafted = min(ncand, d.budget);
  bool drafted = all_cand && cand;
  if (!all_cand) {
    // more candidates than the budget: the `budget` most confident (ties to the lower index)
    const uint64_t ck = cand ? rank_key(c, tid) : 0ull;
    if (d.budget <= 32) {
      if (in) s_draft[tid] = 0;
      uint64_t held;
      const int slot = top_small(ck, d.budget, keys, &held);
      if (slot >= 0) s_draft[rank_key_row(held)] = 1;
      __syncthreads();
      drafted = in && s_draft[tid] != 0;
    } else {
      if (in) keys[tid] = ck;
      __syncthreads();
      drafted = rank_below(keys, per_seq, ck, d.budget) < d.budget && cand;
    }
    __syncthreads();   // the keys are rewritten by the selection
  }
  if (n_drafted == 0 && d.min_one && s_fallback != ~0ull) {
    n_drafted = 1;
    drafted = in && tid == static_cast<int>(static_cast<uint32_t>(s_fallback));
  }

  // Section 5.2 revision of the previous seeds, Section 3 state update
  bool kept = false, replaced = false, remasked = false;
  if (drafted) {
    // a drafted row takes its greedy token, whose uncertainty is ln Z
    tok = yhat;
    u = lnz;
    fl = (fl & ~1u) | 2u;
  } else if (in && (fl & 1u) != 0 && tok != d.mask_id) {
    if (yhat == tok) {
      kept = true;
    } else if (c > d.tau) {
      replaced = true;
      tok = yhat;
      u = lnz;
    } else {
      remasked = true;
      tok = d.mask_id;
      rc = min(rc + 1u, 255u);
    }
  }
  const uint32_t bk = __ballot_sync(0xffffffffu, kept), br = __ballot_sync(0xffffffffu, replaced),
                 bm = __ballot_sync(0xffffffffu, remasked);
  if (lane == 0) {
    if (bk) atomicAdd(&s_cnt[0], __popc(bk));
    if (br) atomicAdd(&s_cnt[1], __popc(br));
    if (bm) atomicAdd(&s_cnt[2], __popc(bm));
  }
  if (select) select_fast(keys, seg, per_seq, d, in, tok, fl, rc, u, din, dout, P.score);
  else __syncthreads();
  if (in) {
    d.tok[n] = tok;
    d.flags[n] = static_cast<uint8_t>(fl);
    d.remask_cnt[n] = static_cast<uint8_t>(rc);
    d.ws_u[n] = u;
  }
  if (tid == 0 && d.stats != nullptr) {
    int32_t* st = d.stats + static_cast<size_t>(seg) * kDecideStats;
    st[0] = n_drafted;
    st[1] = s_cnt[0];
    st[2] = s_cnt[1];
    st[3] = s_cnt[2];
  }
}

// The last CTA of a segment in decision mode: the update, then (unless only the
// update was asked for) the selection with the caller's d_in / d_out.
__device__ void segment_decide(uint64_t* keys, int seg, int per_seq, int sort_n, const ScoreParams& P) {
  if (per_seq <= static_cast<int>(blockDim.x)) {
    decide_fast(keys, seg, per_seq, P);
    return;
  }
  segment_update(keys, seg, per_seq, sort_n, P);
  if (P.dec.phase == 0) {
    __syncthreads();
    segment_select(keys, seg, per_seq, sort_n, P.dec, P.d_in, P.d_out, P.score);
  }
}

// The last CTA of a segment: top-k by (score desc, index asc) over eligible rows.
__device__ __forceinline__ void segment_topk(uint64_t* keys, int seg, int per_seq, int sort_n, int topk,
                                             const float* score, const uint8_t* eligible, int32_t* topk_idx,
                                             float* topk_score) {
  const int tid = threadIdx.x, nt = blockDim.x;
  const int base = seg * per_seq;
  if (per_seq <= nt) {
    // one row per thread: rank every eligible row against the others (see decide_fast)
    uint64_t key = 0;
    float sc = 0.0f;
    if (tid < per_seq) {
      // both loads issued together: the score is read whether or not the row is eligible
      sc = __ldcg(score + base + tid);
      if (eligible == nullptr || eligible[base + tid] != 0) key = rank_key(sc, tid);
    }
    if (tid < per_seq) keys[tid] = key;
    const int n_elig = __syncthreads_count(key != 0);
    {
      const int r = rank_below(keys, per_seq, key, topk);
      if (key != 0 && r < topk) {
        topk_idx[static_cast<size_t>(seg) * topk + r] = tid;
        if (topk_score != nullptr) topk_score[static_cast<size_t>(seg) * topk + r] = sc;
      }
    }
    for (int t = min(n_elig, topk) + tid; t < topk; t += nt) {
      topk_idx[static_cast<size_t>(seg) * topk + t] = -1;
      if (topk_score != nullptr) topk_score[static_cast<size_t>(seg) * topk + t] = -INFINITY;
    }
    return;
  }
  // the scores and flags of kLoads rows per thread are loaded before any key is stored, so the
  // loads of a thread overlap instead of waiting one after the other
  constexpr int kLoads = 4;
  for (int i0 = tid; i0 < sort_n; i0 += kLoads * nt) {
    float sc[kLoads];
    bool el[kLoads];
#pragma unroll
    for (int u = 0; u < kLoads; ++u) {
      const int i = i0 + u * nt;
      const bool in = i < per_seq;
      sc[u] = in ? __ldcg(score + base + i) : 0.0f;
      el[u] = in && (eligible == nullptr || eligible[base + i] != 0);
    }
#pragma unroll
    for (int u = 0; u < kLoads; ++u) {
      const int i = i0 + u * nt;
      if (i < sort_n) keys[i] = el[u] ? rank_key(sc[u], i) : 0;
    }
  }
  __syncthreads();
  // a short list by warp sorts and merges, a long one by sorting
  __shared__ uint64_t s_sel[kRoundsMax];
  const uint64_t* best = keys;
  if (topk <= kRoundsMax) {
    top_select(keys, sort_n, topk, s_sel);
    best = s_sel;
  } else {
    bitonic_sort_desc(keys, sort_n);
  }
  for (int t = tid; t < topk; t += nt) {
    const uint64_t key = best[t];
    const bool valid = key != 0;
    topk_idx[static_cast<size_t>(seg) * topk + t] =
        valid ? static_cast<int32_t>(0xffffffffu - static_cast<uint32_t>(key)) : -1;
    if (topk_score != nullptr)
      topk_score[static_cast<size_t>(seg) * topk + t] =
          valid ? order_key_inv(static_cast<uint32_t>(key >> 32)) : -INFINITY;
  }
}

// Accumulate U vectors of 8 values; the first index of vector u is i0 + u * istride, istride
// being the kernel's constant batch stride when U > 1.
// Per pair of values: one packed FMA for t, two ex2, one packed add into Z and
// one packed FMA into S; two independent accumulator chains.
template <int U>
__device__ __forceinline__ void acc_batch(RowAcc& a, const uint4 (&w)[U], int i0) {
  float x[U][8];
  float bmax = -INFINITY;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    unpack8(w[u], x[u]);
#pragma unroll
    for (int k = 0; k < 8; k += 2) bmax = fmax3(bmax, x[u][k], x[u][k + 1]);
  }
  // the batch is recorded, not searched: only the row maximum's first index is needed, and
  // row_reduce finds it in the recorded batches of the threads that hold that maximum
  if (bmax > a.m) raise_max(a, bmax, i0, U);
  const uint64_t c2 = f2_pack(kLog2e, kLog2e);
  const uint64_t nm2 = f2_pack(-a.mref, -a.mref);
  uint64_t z[2] = {0, 0}, sacc[2] = {0, 0};
#pragma unroll
  for (int u = 0; u < U; ++u) {
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint64_t t2 = f2_fma(f2_pack(x[u][2 * k], x[u][2 * k + 1]), c2, nm2);
      float t0, t1;
      f2_unpack(t2, t0, t1);
      const uint64_t e2 = f2_pack(ex2_approx(t0), ex2_approx(t1));
      z[k & 1] = f2_add(z[k & 1], e2);
      sacc[k & 1] = f2_fma(t2, e2, sacc[k & 1]);
    }
  }
  float z0, z1, s0, s1;
  f2_unpack(f2_add(z[0], z[1]), z0, z1);
  f2_unpack(f2_add(sacc[0], sacc[1]), s0, s1);
  kahan_add(a.z, a.zc, z0 + z1);
  kahan_add(a.s, a.sc, s0 + s1);
}


// ---------------------------------------------------------------------------
// register-load kernel (any V)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(kThreads, 2) score_kernel(const ScoreParams P) {
  extern __shared__ __align__(16) uint64_t keys[];
  __shared__ float red_m[kWarps];
  __shared__ int red_i[kWarps];
  __shared__ float2 red_z[kWarps], red_s[kWarps];
  __shared__ int s_last;
  // programmatic dependent launch: wait for the stream's previous kernel, let the next one be
  // scheduled
  griddep_wait();
  griddep_launch_dependents();

  const int n = blockIdx.x;
  const int tid = threadIdx.x;
  const int V = P.V;
  const size_t row_off = static_cast<size_t>(n) * V;
  const uint16_t* row = P.logits + row_off;
  RowAcc a{-INFINITY, 0x7fffffff, 0, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};

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
    acc_batch<kUnroll>(a, w, head + v * 8);
  }
  for (; v < nvec; v += kThreads) {
    uint4 w[1] = {ld_stream(vrow + v)};
    acc_batch<1>(a, w, head + v * 8);
  }
  if (tail0 + tid < V) acc_scalar(a, bf16_to_f32(row[tail0 + tid]), tail0 + tid);

  const RowOut r = row_reduce<kWarps, kThreads * 8>(a, row, red_m, red_i, red_z, red_s);
  if (tid == 0)
    s_last = row_write(r, n, row, V, P.per_seq, P.decide ? P.dec.tok : P.cur_tok, P.d_in, P.d_out, P.topk,
                       P.maxprob, P.entropy, P.argmax, P.score, P.counters, P.decide ? P.dec.ws_u : nullptr,
                       P.decide ? P.dec.ws_lnz : nullptr);
  __syncthreads();
  if (s_last) {
    if (P.decide)
      segment_decide(keys, n / P.per_seq, P.per_seq, P.sort_n, P);
    else
      segment_topk(keys, n / P.per_seq, P.per_seq, P.sort_n, P.topk, P.score, P.eligible, P.topk_idx, P.topk_score);
  }
}

// ---------------------------------------------------------------------------
// bulk-copy kernel (rows 16-byte aligned)
// ---------------------------------------------------------------------------
__device__ __forceinline__ void bulk_load(void* smem_dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(smem_dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__global__ void __launch_bounds__(kBulkThreads, 4) score_bulk_kernel(const ScoreParams P, int* status) {
  extern __shared__ __align__(128) uint8_t dsmem[];   // ring, reused for top-k keys
  __shared__ uint64_t bar_full[kRingStages], bar_empty[kRingStages];
  __shared__ float red_m[kConsumerWarps + 1];
  __shared__ int red_i[kConsumerWarps + 1];
  __shared__ float2 red_z[kConsumerWarps + 1], red_s[kConsumerWarps + 1];
  __shared__ int s_last, s_abort;
  // programmatic dependent launch: wait for the stream's previous kernel, let the next one be
  // scheduled
  griddep_wait();
  griddep_launch_dependents();

  const int n = blockIdx.x;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int V = P.V;
  const uint16_t* row = P.logits + static_cast<size_t>(n) * V;
  const int nchunks = (V + kChunkElems - 1) / kChunkElems;
  uint8_t* ring = dsmem;

  if (warp == kConsumerWarps && lane == 0) {
    // the producer initialises the ring and issues its first chunks at once, so their latency
    // overlaps the block barrier
    for (int s = 0; s < kRingStages; ++s) {
      mbar_init(&bar_full[s], 1);
      mbar_init(&bar_empty[s], kConsumerWarps);
    }
    s_abort = 0;
    fence_mbar_init();
    for (int c = 0; c < kRingStages && c < nchunks; ++c) {
      const int elems = min(kChunkElems, V - c * kChunkElems);
      mbar_arrive_expect_tx(&bar_full[c], static_cast<uint32_t>(elems * 2));
      bulk_load(ring + c * kChunkBytes, row + static_cast<size_t>(c) * kChunkElems, static_cast<uint32_t>(elems * 2),
                &bar_full[c]);
    }
  }
  __syncthreads();

  RowAcc a{-INFINITY, 0x7fffffff, 0, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
  if (warp == kConsumerWarps) {
    // producer: one lane streams the row chunk by chunk
    if (lane == 0) {
      for (int c = kRingStages; c < nchunks; ++c) {
        const int st = c % kRingStages;
        if (!mbar_wait(&bar_empty[st], ((c / kRingStages) - 1) & 1, &s_abort)) {
          report_status(status, kStatusTimeout, 200);
          s_abort = 1;
          break;
        }
        const int elems = min(kChunkElems, V - c * kChunkElems);
        mbar_arrive_expect_tx(&bar_full[st], static_cast<uint32_t>(elems * 2));
        bulk_load(ring + st * kChunkBytes, row + static_cast<size_t>(c) * kChunkElems,
                  static_cast<uint32_t>(elems * 2), &bar_full[st]);
      }
      // every copy issued has been consumed once the consumers pass their last
      // full-barrier wait; nothing is left in flight at the final barrier
    }
  } else {
    for (int c = 0; c < nchunks; ++c) {
      const int st = c % kRingStages;
      const bool ok = mbar_wait(&bar_full[st], (c / kRingStages) & 1, &s_abort);
      if (!__all_sync(0xffffffffu, ok)) {
        if (lane == 0) {
          report_status(status, kStatusTimeout, 201);
          s_abort = 1;
        }
        break;
      }
      const int elems = min(kChunkElems, V - c * kChunkElems);
      const uint4* src = reinterpret_cast<const uint4*>(ring + st * kChunkBytes);
      const int nv = elems / 8;
      constexpr int kStride = kConsumerWarps * 32;
      if (tid + (kVecPerThread - 1) * kStride < nv) {
        uint4 w[kVecPerThread];
#pragma unroll
        for (int u = 0; u < kVecPerThread; ++u) w[u] = src[tid + u * kStride];
        acc_batch<kVecPerThread>(a, w, c * kChunkElems + tid * 8);
      } else {
        for (int v = tid; v < nv; v += kStride) {
          uint4 w[1] = {src[v]};
          acc_batch<1>(a, w, c * kChunkElems + v * 8);
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&bar_empty[st]);
    }
  }
  // if the producer gave up, wait (bounded) for the copies it already issued
  if (warp == kConsumerWarps && lane == 0 && s_abort) {
    for (int c = max(0, nchunks - kRingStages); c < nchunks; ++c)
      mbar_wait(&bar_full[c % kRingStages], (c / kRingStages) & 1, nullptr, 1000000ull);
  }

  const RowOut r = row_reduce<kConsumerWarps + 1, kConsumerWarps * 32 * 8>(a, row, red_m, red_i, red_z, red_s);
  if (tid == 0)
    s_last = row_write(r, n, row, V, P.per_seq, P.decide ? P.dec.tok : P.cur_tok, P.d_in, P.d_out, P.topk,
                       P.maxprob, P.entropy, P.argmax, P.score, P.counters, P.decide ? P.dec.ws_u : nullptr,
                       P.decide ? P.dec.ws_lnz : nullptr);
  __syncthreads();
  if (s_last) {
    if (P.decide)
      segment_decide(reinterpret_cast<uint64_t*>(ring), n / P.per_seq, P.per_seq, P.sort_n, P);
    else
      segment_topk(reinterpret_cast<uint64_t*>(ring), n / P.per_seq, P.per_seq, P.sort_n, P.topk, P.score,
                   P.eligible, P.topk_idx, P.topk_score);
  }
}

// Section 5.3 selection as its own launch (one CTA per segment), after the
// update phase and the d_in / d_out pass.
constexpr int kSelectThreads = 512;
static_assert(kThreads <= 32 * kMaxWarps && kBulkThreads <= 32 * kMaxWarps && kSelectThreads <= 32 * kMaxWarps,
              "top_rounds keeps a list per warp for at most kMaxWarps warps");
__global__ void __launch_bounds__(kSelectThreads) seed_select_kernel(const DecideArgs d, const float* d_in,
                                                                    const float* d_out, float* score, int per_seq,
                                                                    int sort_n) {
  extern __shared__ __align__(16) uint64_t sel_keys[];
  // programmatic dependent launch: wait for the stream's previous kernel, let the next one be
  // scheduled
  griddep_wait();
  griddep_launch_dependents();
  const int tid = threadIdx.x;
  if (per_seq <= static_cast<int>(blockDim.x)) {
    // one row per thread: the state in registers, selection by rank
    const int n = blockIdx.x * per_seq + tid;
    const bool in = tid < per_seq;
    int tok = 0;
    uint32_t fl = 0, rc = 0;
    float u = 0.0f, din = 0.0f, dout = 0.0f;
    if (in) {
      tok = d.tok[n];
      fl = d.flags[n];
      rc = d.remask_cnt[n];
      u = d.ws_u[n];
      din = d_in != nullptr ? d_in[n] : 0.0f;
      dout = d_out != nullptr ? d_out[n] : 0.0f;
    }
    select_fast(sel_keys, blockIdx.x, per_seq, d, in, tok, fl, rc, u, din, dout, score);
    if (in) d.flags[n] = static_cast<uint8_t>(fl);
    return;
  }
  segment_select(sel_keys, blockIdx.x, per_seq, sort_n, d, d_in, d_out, score);
}

}  // namespace

namespace {

int launch_score_impl(const ScoreArgs& a, const DecideArgs* d, int* status, cudaStream_t stream) {
  const int per = a.N / a.n_seq;
  int sort_n = 1;
  while (sort_n < per) sort_n <<= 1;
  ScoreParams P{static_cast<const uint16_t*>(a.logits), a.V, per, a.cur_tok, a.d_in, a.d_out, a.eligible,
                a.topk, sort_n, a.maxprob, a.entropy, a.argmax, a.score, a.topk_idx, a.topk_score, a.counters,
                d != nullptr ? 1 : 0, d != nullptr ? *d : DecideArgs{}};
  // top-k keys; the decision step also keeps a float score per row behind them. At least one key
  // per thread of the register-load kernel: the one-row-per-thread selection publishes up to
  // 32 keys per warp.
  const size_t key_slots = static_cast<size_t>(std::max(sort_n, kThreads));
  const size_t keys_bytes = d != nullptr ? (sizeof(uint64_t) + sizeof(float)) * key_slots
                            : a.topk > 0 ? sizeof(uint64_t) * key_slots : 0;
  const bool aligned_rows = (a.V % 8) == 0 && (reinterpret_cast<uintptr_t>(a.logits) % 16) == 0;
  if (aligned_rows) {
    const size_t smem = std::max(keys_bytes, static_cast<size_t>(kRingStages) * kChunkBytes);
    // the ring's shared-memory limit is a function attribute of the current context
    static ContextCache<int> setup;
    int unused = 0;
    const int rc = setup.get(&unused, [](int&) {
      return cudaFuncSetAttribute(score_bulk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(kRingStages * kChunkBytes)) == cudaSuccess ? 0 : -3;
    });
    if (rc != 0) return rc;
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = pdl_config(dim3(a.N), dim3(kBulkThreads), smem, stream, attr);
    if (cudaLaunchKernelEx(&cfg, score_bulk_kernel, P, status) != cudaSuccess) return -3;
  } else {
    // decision keys of the longest segment: 4096 x 12 bytes, above the 48 KB a launch gets
    // without opting in (with the static shared memory)
    static ContextCache<int> setup_reg;
    int unused = 0;
    const int rc = setup_reg.get(&unused, [](int&) {
      return cudaFuncSetAttribute(score_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>((sizeof(uint64_t) + sizeof(float)) * kMaxPerSeq)) == cudaSuccess
                 ? 0 : -3;
    });
    if (rc != 0) return rc;
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg = pdl_config(dim3(a.N), dim3(kThreads), keys_bytes, stream, attr);
    if (cudaLaunchKernelEx(&cfg, score_kernel, P) != cudaSuccess) return -3;
  }
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace

int launch_score(const ScoreArgs& a, int* status, cudaStream_t stream) {
  return launch_score_impl(a, nullptr, status, stream);
}

int launch_score_decide(const ScoreArgs& a, const DecideArgs& d, int* status, cudaStream_t stream) {
  return launch_score_impl(a, &d, status, stream);
}

int launch_seed_select(int N, int n_seq, const DecideArgs& d, const float* d_in, const float* d_out, float* score,
                       cudaStream_t stream) {
  const int per = N / n_seq;
  int sort_n = 1;
  while (sort_n < per) sort_n <<= 1;
  // at least one key per thread: the one-row-per-thread selection publishes up to 32 keys per warp
  const size_t smem = (sizeof(uint64_t) + sizeof(float)) * static_cast<size_t>(std::max(sort_n, kSelectThreads));
  // the longest segment's keys and scores (48 KB) need the opt-in above the default limit
  static ContextCache<int> setup;
  int unused = 0;
  const int rc = setup.get(&unused, [](int&) {
    return cudaFuncSetAttribute(seed_select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>((sizeof(uint64_t) + sizeof(float)) * kMaxPerSeq)) == cudaSuccess
               ? 0 : -3;
  });
  if (rc != 0) return rc;
  cudaLaunchAttribute attr[1];
  const cudaLaunchConfig_t cfg = pdl_config(dim3(n_seq), dim3(kSelectThreads), smem, stream, attr);
  if (cudaLaunchKernelEx(&cfg, seed_select_kernel, d, d_in, d_out, score, per, sort_n) != cudaSuccess) return -3;
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

// ---------------------------------------------------------------------------
// Allocation-free variant: the same kernels, with the per-segment counters in
// a fixed device array of this library instead of a caller workspace.
// ---------------------------------------------------------------------------
namespace {

// Counters for at most kNoAllocMaxSegments segments (16 KB). Every device that
// loads the library holds one copy until the process exits.
static __device__ __align__(256) uint32_t g_noalloc_counters[kNoAllocMaxSegments];

// Device address of the counter array in the current device's context. In host
// code the array's name is only a host-side stand-in, so the address is looked up
// (cudaGetSymbolAddress, with the device current) the first time a context calls,
// and again in a context created anew after cudaDeviceReset.
uint32_t* noalloc_counters() {
  static ContextCache<uint32_t*> cache;
  uint32_t* p = nullptr;
  const int rc = cache.get(&p, [](uint32_t*& v) {
    void* a = nullptr;
    if (cudaGetSymbolAddress(&a, g_noalloc_counters) != cudaSuccess || a == nullptr) return -3;
    v = static_cast<uint32_t*>(a);
    return 0;
  });
  return rc == 0 ? p : nullptr;
}

}  // namespace

int launch_score_noalloc(ScoreArgs a, int* status, cudaStream_t stream) {
  if (a.n_seq > kNoAllocMaxSegments) return -1;
  uint32_t* counters = noalloc_counters();
  if (counters == nullptr) return -3;
  // the array keeps whatever the previous call left: the counters this call
  // uses must start at zero
  if (a.topk > 0 &&
      cudaMemsetAsync(counters, 0, sizeof(uint32_t) * static_cast<size_t>(a.n_seq), stream) != cudaSuccess)
    return -3;
  a.counters = counters;
  return launch_score(a, status, stream);
}

}  // namespace cover
