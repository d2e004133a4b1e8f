// mass_kernel.cu - the influence terms of the seed score (Section 5.3):
//   d_in(j)  = sum over still-masked queries q of A[q -> j]
//   d_out(j) = sum over positions i drafted in this step of A[j -> i]
// with A the attention matrix of the current pass averaged over the heads,
// for the response positions pos0 .. pos0 + per - 1 of every batch row.
//
// The weights are recomputed from the attention pass's inputs and its
// log-sum-exp: A_h[q -> j] = exp(q.k'_j / sqrt(d) - lse_h(q)), where a seed
// query's diagonal entry uses its masked-input key k_q (its leave-one-out view,
// Section 5.1; the stored lse is that of the corrected distribution), so each
// row sums to one over the whole memory. Only response queries and response
// keys contribute, so the pass covers a per x per block of each head.
//
// Per CTA: 128 query rows of one head. S = Q K'^T on the tensor cores
// (tcgen05, double-buffered in tensor memory: no P.V here), one thread per
// row turns its S row into weights; the weights to drafted keys are summed in
// registers (d_out), the weights of masked rows are summed per key through a
// padded shared-memory transpose (d_in). Each CTA writes its partial sums;
// a second kernel adds the partials of all heads and row tiles in a fixed
// order (deterministic) and divides by the head count.
//
// Warps: 0-3 rows (thread = row = tensor-memory lane), 4 allocates tensor
// memory and issues the products (lane 0), 5 issues TMA loads (lane 0).
#include <cuda_bf16.h>
#include <math.h>

#include "context.cuh"
#include "kernels.cuh"
#include "ptx.cuh"
#include "route.cuh"
#include "tmap.cuh"

namespace cover {
namespace {

constexpr int kD = 128;
constexpr int kBM = 128;                    // query rows per CTA
constexpr int kBN = 128;                    // keys per tile
constexpr int kThreads = 256;
constexpr int kRowThreads = 128;
constexpr int kMmaWarp = 4;
constexpr int kTmaWarp = 5;
constexpr int kTileBytes = kBM * kD * 2;    // 32 KB
constexpr int kBoxBytes = kTileBytes / 2;   // one 64-column, 128-byte-swizzled box
constexpr int kStride = 132;                // floats per staging row: conflict-free float4 rows, column reads
constexpr int kRowBar = 1;                  // named barrier of the 128 row threads

struct MassSmem {
  uint8_t q[kTileBytes];
  uint8_t k[2][kTileBytes];
  float stage[kBM * kStride];
  uint64_t bar_q;
  uint64_t bar_k_full[2];
  uint64_t bar_k_empty[2];
  uint64_t bar_s_full[2];
  uint64_t bar_s_empty[2];
  uint64_t bar_drain;
  uint32_t tmem_base;
  int abort;
  int slot[kBM];
  uint32_t drafted[2][kBN / 32];            // drafted bits of a tile's keys, by tile parity
};

__device__ __forceinline__ void row_bar_sync() {
  asm volatile("bar.sync %0, %1;" ::"r"(kRowBar), "r"(kRowThreads) : "memory");
}

// barrier of the row threads that also ANDs / ORs a predicate over them
__device__ __forceinline__ bool row_bar_and(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(kRowBar), "r"(kRowThreads)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ bool row_bar_or(bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(kRowBar), "r"(kRowThreads)
      : "memory");
  return r != 0;
}

__global__ void __launch_bounds__(kThreads, 1)
    mass_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                const __nv_bfloat16* __restrict__ k_seedmask, const int32_t* __restrict__ seed_idx, int n_seeds,
                const float* __restrict__ lse, int Hq, int Hkv, int L, int pos0, int per, int n_qt,
                const int32_t* __restrict__ tok, const uint8_t* __restrict__ flags, int mask_id, float scale_log2,
                float* __restrict__ part_in, float* __restrict__ part_out, int* status) {
  extern __shared__ uint8_t smem_raw[];
  MassSmem& sm = *reinterpret_cast<MassSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const int qt = blockIdx.x % n_qt;
  const int hq = (blockIdx.x / n_qt) % Hq;
  const int b = blockIdx.x / (n_qt * Hq);
  const int hkv = hq / (Hq / Hkv);
  const int nkv = (per + kBN - 1) / kBN;
  const int qrow0 = qt * kBM;               // first response row of this CTA

  if (tid == 0) {
    mbar_init(&sm.bar_q, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.bar_k_full[s], 1);
      mbar_init(&sm.bar_k_empty[s], 1);
      mbar_init(&sm.bar_s_full[s], 1);
      mbar_init(&sm.bar_s_empty[s], kRowThreads);
    }
    mbar_init(&sm.bar_drain, 1);
    sm.abort = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&sm.tmem_base, 256);
    tmem_relinquish();
  }
  route_clear(sm.slot, kBM, tid, kThreads);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  route_scan(sm.slot, seed_idx + static_cast<size_t>(b) * n_seeds, n_seeds, pos0 + qrow0, kBM, L, tid, kThreads);
  __syncthreads();
  const uint32_t tbase = sm.tmem_base;

  if (warp == kTmaWarp) {
    if (lane == 0) {
      tma_prefetch_desc(&tm_q);
      tma_prefetch_desc(&tm_k);
      mbar_arrive_expect_tx(&sm.bar_q, kTileBytes);
      for (int h = 0; h < 2; ++h) tma_load_4d(sm.q + h * kBoxBytes, &tm_q, &sm.bar_q, 64 * h, pos0 + qrow0, hq, b);
      int last = -1;
      bool ok = true;
      for (int j = 0; j < nkv; ++j) {
        const int st = j & 1;
        if (j >= 2 && !mbar_wait(&sm.bar_k_empty[st], ((j - 2) >> 1) & 1, &sm.abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&sm.bar_k_full[st], kTileBytes);
        for (int h = 0; h < 2; ++h)
          tma_load_4d(sm.k[st] + h * kBoxBytes, &tm_k, &sm.bar_k_full[st], 64 * h, pos0 + j * kBN, hkv, b);
        last = j;
      }
      if (!ok) {
        report_status(status, kStatusTimeout, 50);
        sm.abort = 1;
        // let every copy already issued land before the CTA's shared memory is released
        mbar_wait(&sm.bar_q, 0, nullptr);
        for (int jj = max(0, last - 1); jj <= last; ++jj) mbar_wait(&sm.bar_k_full[jj & 1], (jj >> 1) & 1, nullptr);
      }
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t id_qk = idesc_bf16_f32(kBM, kBN, false, false);
      constexpr uint64_t kTileDesc = kTileBytes >> 4;
      bool ok = mbar_wait(&sm.bar_q, 0, &sm.abort);
      tc_fence_after_sync();
      const uint64_t dq = sdesc_sw128(smem_u32(sm.q), 16, 1024);
      const uint64_t dk0 = sdesc_sw128(smem_u32(sm.k[0]), 16, 1024);
      for (int j = 0; j < nkv && ok; ++j) {
        const int st = j & 1;
        ok = mbar_wait(&sm.bar_k_full[st], (j >> 1) & 1, &sm.abort);
        if (ok && j >= 2) ok = mbar_wait(&sm.bar_s_empty[st], ((j - 2) >> 1) & 1, &sm.abort);
        if (!ok) break;
        tc_fence_after_sync();
        // S_st = Q . K(j)^T, both K-major with 128-byte swizzle
#pragma unroll
        for (int ks = 0; ks < kD / 16; ++ks) {
          const uint64_t off = static_cast<uint64_t>(((ks >> 2) * kBoxBytes + (ks & 3) * 32) >> 4);
          umma_ss(tbase + st * 128, dq + off, dk0 + st * kTileDesc + off, id_qk, ks > 0 ? 1u : 0u);
        }
        umma_commit(&sm.bar_s_full[st]);
        umma_commit(&sm.bar_k_empty[st]);
      }
      if (!ok) {
        report_status(status, kStatusTimeout, 51);
        sm.abort = 1;
      }
      // all tensor-core work of this CTA must finish before tensor memory is released
      umma_commit(&sm.bar_drain);
      mbar_wait(&sm.bar_drain, 0, nullptr);
    }
  } else if (warp < 4) {
    // ---------------- rows ----------------
    const int r = tid;                                 // row of the CTA = tensor-memory lane
    const uint32_t trow = tbase + (static_cast<uint32_t>(warp * 32) << 16);
    const int row = qrow0 + r;                         // response row
    const bool valid = row < per;
    const size_t srow = static_cast<size_t>(b) * per + row;
    const bool masked = valid && tok[srow] == mask_id;
    const float lse2 = valid ? lse[(static_cast<size_t>(b) * Hq + hq) * L + pos0 + row] * 1.4426950408889634f : 0.0f;
    const int my_slot = sm.slot[r];
    const bool is_seed = valid && my_slot != kNoSlot;
    const bool any_masked = row_bar_or(masked);        // uniform over the CTA's rows
    bool ok = true;

    // seed rows: diagonal weight from the masked-input key (row and key tiles align)
    float p_self = 0.0f;
    if (__any_sync(0xffffffffu, is_seed)) {
      ok = mbar_wait(&sm.bar_q, 0, &sm.abort);
      if (ok && is_seed) {
        const uint4* kmv =
            reinterpret_cast<const uint4*>(k_seedmask + ((static_cast<size_t>(b) * Hkv + hkv) * n_seeds + my_slot) * kD);
        float dot[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
        for (int ch = 0; ch < 16; ++ch) {
          const int h = ch >> 3, c8 = ch & 7;
          const uint4 qv =
              *reinterpret_cast<const uint4*>(sm.q + h * kBoxBytes + r * 128 + ((c8 ^ (r & 7)) * 16));
          const uint4 kv = __ldg(kmv + ch);
          const __nv_bfloat162* qp = reinterpret_cast<const __nv_bfloat162*>(&qv);
          const __nv_bfloat162* kp = reinterpret_cast<const __nv_bfloat162*>(&kv);
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 qf = __bfloat1622float2(qp[e]);
            const float2 kf = __bfloat1622float2(kp[e]);
            dot[e] = fmaf(qf.x, kf.x, dot[e]);
            dot[e] = fmaf(qf.y, kf.y, dot[e]);
          }
        }
        p_self = ex2_approx(((dot[0] + dot[1]) + (dot[2] + dot[3])) * scale_log2 - lse2);
      }
    }

    float acc_out = 0.0f;
    for (int j = 0; j < nkv; ++j) {
      const int st = j & 1;
      bool w = ok && mbar_wait(&sm.bar_s_full[st], (j >> 1) & 1, &sm.abort);
      // drafted bits of this tile's keys (key j * 128 + r)
      const int key = j * kBN + r;
      const bool dr = key < per && (flags[static_cast<size_t>(b) * per + key] & 2u) != 0;
      const uint32_t bits = __ballot_sync(0xffffffffu, dr);
      if (lane == 0) sm.drafted[st][warp] = bits;
      ok = row_bar_and(w);                             // uniform decision; drafted words visible
      if (!ok) break;
      tc_fence_after_sync();
      uint32_t raw[4][32];
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld32(trow + st * 128 + 32 * c, raw[c]);
#pragma unroll
      for (int c = 0; c < 4; ++c) tmem_ld_wait(raw[c]);
      tc_fence_before_sync();
      mbar_arrive(&sm.bar_s_empty[st]);
      float* s = reinterpret_cast<float*>(&raw[0][0]);
      const int nvalid = min(kBN, per - j * kBN);
      const uint32_t dw[4] = {sm.drafted[st][0], sm.drafted[st][1], sm.drafted[st][2], sm.drafted[st][3]};
      float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int c = 0; c < kBN; ++c) {
        float pc = c < nvalid ? ex2_approx(fmaf(s[c], scale_log2, -lse2)) : 0.0f;
        if (is_seed && j == qt && c == r) pc = p_self;
        if (!valid) pc = 0.0f;
        s[c] = pc;
        if ((dw[c >> 5] >> (c & 31)) & 1u) acc[c & 3] += pc;
      }
      acc_out += (acc[0] + acc[1]) + (acc[2] + acc[3]);
      float colsum = 0.0f;
      if (any_masked) {
        float4* dst = reinterpret_cast<float4*>(sm.stage + r * kStride);
#pragma unroll
        for (int c4 = 0; c4 < kBN / 4; ++c4)
          dst[c4] = masked ? make_float4(s[4 * c4], s[4 * c4 + 1], s[4 * c4 + 2], s[4 * c4 + 3])
                           : make_float4(0.0f, 0.0f, 0.0f, 0.0f);
        row_bar_sync();
        // column r of this tile: the mass the CTA's masked rows put on key j * 128 + r
        float cs[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll 8
        for (int q = 0; q < kBM; ++q) cs[q & 3] += sm.stage[q * kStride + r];
        colsum = (cs[0] + cs[1]) + (cs[2] + cs[3]);
      }
      if (key < per) part_in[((static_cast<size_t>(b) * Hq + hq) * n_qt + qt) * per + key] = colsum;
    }
    if (!ok) {
      if (!sm.abort) {
        report_status(status, kStatusTimeout, 52);
        sm.abort = 1;
      }
    } else if (valid) {
      part_out[(static_cast<size_t>(b) * Hq + hq) * per + row] = acc_out;
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  if (warp == kMmaWarp) tmem_dealloc(tbase, 256);
}

// d_in / d_out of row n = b * per + i: the partial sums of every head (and row
// tile) in a fixed order, divided by the head count.
__global__ void mass_reduce_kernel(const float* __restrict__ part_in, const float* __restrict__ part_out, int B,
                                   int Hq, int per, int n_qt, float* __restrict__ d_in, float* __restrict__ d_out) {
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= B * per) return;
  const int b = n / per, i = n % per;
  float si = 0.0f, so = 0.0f;
  for (int h = 0; h < Hq; ++h) {
    const size_t bh = static_cast<size_t>(b) * Hq + h;
    for (int t = 0; t < n_qt; ++t) si += part_in[(bh * n_qt + t) * per + i];
    so += part_out[bh * per + i];
  }
  const float inv = 1.0f / static_cast<float>(Hq);
  d_in[n] = si * inv;
  d_out[n] = so * inv;
}

}  // namespace

size_t mass_workspace_bytes(int B, int Hq, int per) {
  const size_t n_qt = (per + kBM - 1) / kBM;
  return sizeof(float) * static_cast<size_t>(B) * Hq * per * (n_qt + 1);
}

int launch_attn_mass(const MassArgs& a, int* status, cudaStream_t stream) {
  CUtensorMap tq, tk;
  if (!make_bf16_map_4d(&tq, a.q, kD, a.L, a.Hq, a.B, kBM) || !make_bf16_map_4d(&tk, a.k_cached, kD, a.L, a.Hkv, a.B, kBN))
    return -3;
  const int n_qt = (a.per + kBM - 1) / kBM;
  const long long grid = static_cast<long long>(n_qt) * a.Hq * a.B;
  if (grid > 0x7fffffffLL) return -2;
  float* part_in = static_cast<float*>(a.workspace);
  float* part_out = part_in + static_cast<size_t>(a.B) * a.Hq * n_qt * a.per;
  const size_t smem = sizeof(MassSmem) + 1024;
  // the shared-memory limit is a function attribute of the current context
  static ContextCache<int> setup;
  int unused = 0;
  const int rc = setup.get(&unused, [&](int&) {
    return cudaFuncSetAttribute(mass_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem)) ==
                   cudaSuccess ? 0 : -3;
  });
  if (rc != 0) return rc;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kD));
  mass_kernel<<<static_cast<unsigned>(grid), kThreads, smem, stream>>>(
      tq, tk, static_cast<const __nv_bfloat16*>(a.k_seedmask), a.seed_idx, a.n_seeds, a.lse, a.Hq, a.Hkv, a.L, a.pos0,
      a.per, n_qt, a.tok, a.flags, a.mask_id, scale_log2, part_in, part_out, status);
  if (cudaGetLastError() != cudaSuccess) return -3;
  const int rows = a.B * a.per;
  mass_reduce_kernel<<<(rows + 255) / 256, 256, 0, stream>>>(part_in, part_out, a.B, a.Hq, a.per, n_qt, a.d_in,
                                                             a.d_out);
  return cudaGetLastError() == cudaSuccess ? 0 : -3;
}

}  // namespace cover
