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
// Both sums become row sums held in registers by computing the block twice on
// the tensor cores, once per orientation, in two kinds of CTA per (b, hq, tile):
//   rows CTA    S  = Q_t K_j^T for every key tile j: thread = query row of tile
//               t, sums its weights over the drafted keys (d_out partial);
//   columns CTA S' = K_t Q_j^T for every query tile j: thread = key of tile t,
//               sums exp(s - lse(q)) over the masked queries q, whose lse is
//               staged per column in shared memory (+inf for a query that is
//               not masked, so its weight is exactly 0) (d_in partial).
// The resident tile (Q_t or K_t) is loaded once; the other operand streams
// through a two-stage ring, and S double-buffers in tensor memory so a tile's
// product overlaps the previous tile's exponentials. A 32-column chunk with no
// drafted key (rows) or no masked query (columns) is skipped as a whole (its
// predicate is the same for every thread). Each CTA writes one partial per
// row of its tile; a second kernel adds the partials of the Hq heads in a
// fixed order (deterministic) and divides by the head count.
//
// Warps: 0-3 rows / keys of the tile (thread = tensor-memory lane), 4 issues
// the TMA loads (lane 0), 5 allocates tensor memory and issues the products
// (lane 0). About 100 KB of shared memory and 256 tensor-memory columns per CTA,
// so two CTAs share an SM.
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
constexpr int kT = 128;                     // rows / keys per tile
constexpr int kThreads = 192;
constexpr int kMathThreads = 128;
constexpr int kTmaWarp = 4;
constexpr int kMmaWarp = 5;
constexpr int kTileBytes = kT * kD * 2;     // 32 KB
constexpr int kBoxBytes = kTileBytes / 2;   // one 64-column, 128-byte-swizzled box
constexpr int kMaxPer = kMassMaxPer;        // per-column staging must fit in shared memory

// 128-byte aligned, so the per-column arrays that follow it start 16-byte aligned (float4 reads)
struct alignas(128) MassSmem {
  uint8_t x[kTileBytes];                    // resident operand: Q_t (rows) or K_t (columns)
  uint8_t y[2][kTileBytes];                 // streamed operand: K_j (rows) or Q_j (columns)
  uint64_t bar_x;
  uint64_t bar_y_full[2];
  uint64_t bar_y_empty[2];
  uint64_t bar_s_full[2];
  uint64_t bar_s_empty[2];
  uint64_t bar_drain;
  uint32_t tmem_base;
  int abort;
  int slot[kT];                             // seed slot of the resident tile's positions
  // followed by the per-column data of the whole block (dynamic size):
  //   uint32_t bits[n_t * 4]  drafted keys (rows) / masked queries (columns)
  //   float colv[n_t * 128]   columns: log2-scaled lse of a masked query, else +inf
};

static_assert(sizeof(MassSmem) % 16 == 0, "per-column arrays must start 16-byte aligned");

__device__ __forceinline__ uint32_t* col_bits(MassSmem& sm) { return reinterpret_cast<uint32_t*>(&sm + 1); }
__device__ __forceinline__ float* col_vals(MassSmem& sm, int n_t) {
  return reinterpret_cast<float*>(col_bits(sm) + n_t * 4);
}

// q_row . k_row over the 128 dimensions, both bf16 rows in global memory.
__device__ __forceinline__ float dot_row(const __nv_bfloat16* qrow, const __nv_bfloat16* krow) {
  const uint4* qv = reinterpret_cast<const uint4*>(qrow);
  const uint4* kv = reinterpret_cast<const uint4*>(krow);
  float d[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
  for (int ch = 0; ch < 16; ++ch) {
    const uint4 a = __ldg(qv + ch), b = __ldg(kv + ch);
    const __nv_bfloat162* ap = reinterpret_cast<const __nv_bfloat162*>(&a);
    const __nv_bfloat162* bp = reinterpret_cast<const __nv_bfloat162*>(&b);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      const float2 af = __bfloat1622float2(ap[e]), bf = __bfloat1622float2(bp[e]);
      d[e] = fmaf(af.x, bf.x, d[e]);
      d[e] = fmaf(af.y, bf.y, d[e]);
    }
  }
  return (d[0] + d[1]) + (d[2] + d[3]);
}

// blockIdx.x = (b * Hq + hq) * n_t + t; blockIdx.y = 0 rows CTA, 1 columns CTA.
__global__ void __launch_bounds__(kThreads, 2)
    mass_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k_seedmask,
                const int32_t* __restrict__ seed_idx, int n_seeds, const float* __restrict__ lse, int Hq, int Hkv,
                int L, int pos0, int per, int n_t, const int32_t* __restrict__ tok, const uint8_t* __restrict__ flags,
                int mask_id, float scale_log2, float* __restrict__ part_in, float* __restrict__ part_out,
                int* status) {
  extern __shared__ uint8_t smem_raw[];
  MassSmem& sm = *reinterpret_cast<MassSmem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));

  const int tid = threadIdx.x;
  const int warp = tid >> 5, lane = tid & 31;
  const bool cols = blockIdx.y != 0;
  const int t = static_cast<int>(blockIdx.x) % n_t;
  const int bh = static_cast<int>(blockIdx.x) / n_t;   // b * Hq + hq
  const int hq = bh % Hq, b = bh / Hq;
  const int hkv = hq / (Hq / Hkv);
  uint32_t* bits = col_bits(sm);
  float* colv = col_vals(sm, n_t);
  // launched as a programmatic dependent of the stream's previous kernel: wait for its results;
  // the reduction kernel behind this one may be scheduled now, it waits for this grid's results
  griddep_wait();
  griddep_launch_dependents();

  const CUtensorMap* tm_x = cols ? &tm_k : &tm_q;
  const CUtensorMap* tm_y = cols ? &tm_q : &tm_k;
  const int hx = cols ? hkv : hq, hy = cols ? hq : hkv;
  if (warp == kTmaWarp && lane == 0) {
    // the TMA thread initialises the barriers and issues the resident tile and the first two
    // streamed tiles at once, so their latency overlaps the rest of the prologue
    mbar_init(&sm.bar_x, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&sm.bar_y_full[s], 1);
      mbar_init(&sm.bar_y_empty[s], 1);
      mbar_init(&sm.bar_s_full[s], 1);
      mbar_init(&sm.bar_s_empty[s], kMathThreads / 32);
    }
    mbar_init(&sm.bar_drain, 1);
    sm.abort = 0;
    fence_mbar_init();
    tma_prefetch_desc(tm_x);
    tma_prefetch_desc(tm_y);
    mbar_arrive_expect_tx(&sm.bar_x, kTileBytes);
    for (int h = 0; h < 2; ++h) tma_load_4d(sm.x + h * kBoxBytes, tm_x, &sm.bar_x, 64 * h, pos0 + t * kT, hx, b);
    for (int j = 0; j < 2 && j < n_t; ++j) {
      mbar_arrive_expect_tx(&sm.bar_y_full[j], kTileBytes);
      for (int h = 0; h < 2; ++h)
        tma_load_4d(sm.y[j] + h * kBoxBytes, tm_y, &sm.bar_y_full[j], 64 * h, pos0 + j * kT, hy, b);
    }
  }
  if (warp == kMmaWarp) {
    tmem_alloc(&sm.tmem_base, 256);
    tmem_relinquish();
  }
  route_clear(sm.slot, kT, tid, kThreads);
  // the first seed entry of this thread, loaded now so that its latency overlaps the column data's
  const int32_t* seeds_b = seed_idx + static_cast<size_t>(b) * n_seeds;
  const int seed0 = tid < n_seeds ? __ldg(seeds_b + tid) : -1;
  // rows CTAs: the log2-scaled lse of the thread's own query (thread = row of the tile)
  float own = 0.0f;
  if (!cols && tid < kMathThreads && t * kT + tid < per)
    own = lse[static_cast<size_t>(bh) * L + pos0 + t * kT + tid] * 1.4426950408889634f;
  // per-column data of the whole block: rows CTAs need the drafted keys, columns CTAs the masked
  // queries and their lse; one warp per 32 columns
  for (int w = warp; w < n_t * 4; w += kThreads / 32) {
    const int c = w * 32 + lane;
    const bool in = c < per;
    const size_t srow = static_cast<size_t>(b) * per + c;
    bool on;
    if (!cols) {
      on = in && (flags[srow] & 2u) != 0;
    } else {
      on = in && tok[srow] == mask_id;
      colv[c] = on ? lse[static_cast<size_t>(bh) * L + pos0 + c] * 1.4426950408889634f : INFINITY;
    }
    const uint32_t word = __ballot_sync(0xffffffffu, on);
    if (lane == 0) bits[w] = word;
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  {
    // seed routing of the resident tile's positions (the lowest slot naming a position wins)
    const int row0 = pos0 + t * kT;
    if (seed0 >= row0 && seed0 < row0 + kT && seed0 < L) atomicMin(sm.slot + (seed0 - row0), tid);
    for (int sidx = tid + kThreads; sidx < n_seeds; sidx += kThreads) {
      const int p = __ldg(seeds_b + sidx);
      if (p >= row0 && p < row0 + kT && p < L) atomicMin(sm.slot + (p - row0), sidx);
    }
  }
  __syncthreads();
  const uint32_t tbase = sm.tmem_base;

  if (warp == kTmaWarp) {
    if (lane == 0) {
      int last = min(n_t, 2) - 1;
      bool ok = true;
      for (int j = 2; j < n_t; ++j) {
        const int st = j & 1;
        if (!mbar_wait(&sm.bar_y_empty[st], ((j - 2) >> 1) & 1, &sm.abort)) {
          ok = false;
          break;
        }
        mbar_arrive_expect_tx(&sm.bar_y_full[st], kTileBytes);
        for (int h = 0; h < 2; ++h)
          tma_load_4d(sm.y[st] + h * kBoxBytes, tm_y, &sm.bar_y_full[st], 64 * h, pos0 + j * kT, hy, b);
        last = j;
      }
      if (!ok) {
        report_status(status, kStatusTimeout, 60);
        sm.abort = 1;
        // let every copy already issued land before the CTA's shared memory is released
        mbar_wait(&sm.bar_x, 0, nullptr);
        for (int jj = max(0, last - 1); jj <= last; ++jj) mbar_wait(&sm.bar_y_full[jj & 1], (jj >> 1) & 1, nullptr);
      }
    }
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t id_s = idesc_bf16_f32(kT, kT, false, false);
      constexpr uint64_t kTileDesc = kTileBytes >> 4;
      bool ok = mbar_wait(&sm.bar_x, 0, &sm.abort);
      tc_fence_after_sync();
      const uint64_t dx = sdesc_sw128(smem_u32(sm.x), 16, 1024);
      const uint64_t dy0 = sdesc_sw128(smem_u32(sm.y[0]), 16, 1024);
      for (int j = 0; j < n_t && ok; ++j) {
        const int st = j & 1;
        ok = mbar_wait(&sm.bar_y_full[st], (j >> 1) & 1, &sm.abort);
        if (ok && j >= 2) ok = mbar_wait(&sm.bar_s_empty[st], ((j - 2) >> 1) & 1, &sm.abort);
        if (!ok) break;
        tc_fence_after_sync();
        // S_st = X . Y(j)^T, both K-major with 128-byte swizzle
#pragma unroll
        for (int ks = 0; ks < kD / 16; ++ks) {
          const uint64_t off = static_cast<uint64_t>(((ks >> 2) * kBoxBytes + (ks & 3) * 32) >> 4);
          umma_ss(tbase + st * kT, dx + off, dy0 + st * kTileDesc + off, id_s, ks > 0 ? 1u : 0u);
        }
        umma_commit(&sm.bar_s_full[st]);
        umma_commit(&sm.bar_y_empty[st]);
      }
      if (!ok) {
        report_status(status, kStatusTimeout, 61);
        sm.abort = 1;
      }
      // all tensor-core work of this CTA must finish before tensor memory is released
      umma_commit(&sm.bar_drain);
      mbar_wait(&sm.bar_drain, 0, nullptr);
    }
  } else {
    // ---------------- rows / keys of the resident tile ----------------
    const int r = tid;                                 // tensor-memory lane
    const uint32_t trow = tbase + (static_cast<uint32_t>(warp * 32) << 16);
    const int i = t * kT + r;                          // response index of this thread's query / key
    const bool valid = i < per;
    const size_t qrow = (static_cast<size_t>(bh) * L + pos0 + i) * kD;
    // the diagonal entry of a seed query uses its masked-input key (leave-one-out view)
    const int my_slot = valid ? sm.slot[r] : kNoSlot;
    float p_self = 0.0f;
    if (my_slot != kNoSlot) {
      const float lse2 = cols ? colv[i] : own;         // +inf for a query that is not masked: weight 0
      const float dot = dot_row(q + qrow, k_seedmask + ((static_cast<size_t>(b) * Hkv + hkv) * n_seeds + my_slot) * kD);
      p_self = ex2_approx(dot * scale_log2 - lse2);
    }
    float acc = 0.0f;
    bool ok = true;
    for (int j = 0; j < n_t; ++j) {
      const int st = j & 1;
      ok = mbar_wait(&sm.bar_s_full[st], (j >> 1) & 1, &sm.abort);
      if (!__all_sync(0xffffffffu, ok)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const int diag = (j == t && my_slot != kNoSlot) ? r : -1;   // column of the seed diagonal
      float a4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
      // two halves of 64 columns keep half of the tile in registers at a time
#pragma unroll
      for (int hf = 0; hf < 2; ++hf) {
        uint32_t raw[2][32];
#pragma unroll
        for (int c = 0; c < 2; ++c) tmem_ld32(trow + st * kT + 64 * hf + 32 * c, raw[c]);
#pragma unroll
        for (int c = 0; c < 2; ++c) tmem_ld_wait(raw[c]);
        if (hf == 1) {
          tc_fence_before_sync();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.bar_s_empty[st]);
        }
        const float* s = reinterpret_cast<const float*>(&raw[0][0]);
#pragma unroll
        for (int cc = 0; cc < 2; ++cc) {
          const int c32 = 2 * hf + cc;
          const uint32_t word = bits[j * 4 + c32];    // the same for every thread: uniform branch
          if (word == 0u) continue;
          if (!cols) {
#pragma unroll
            for (int e = 0; e < 32; ++e) {
              const int c = c32 * 32 + e;
              float p = ex2_approx(fmaf(s[cc * 32 + e], scale_log2, -own));
              if (c == diag) p = p_self;
              a4[e & 3] += ((word >> e) & 1u) ? p : 0.0f;
            }
          } else {
            const float4* cv = reinterpret_cast<const float4*>(colv + j * kT + c32 * 32);
#pragma unroll
            for (int e4 = 0; e4 < 8; ++e4) {
              const float4 v = cv[e4];
              const float vv[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const int c = c32 * 32 + e4 * 4 + e;
                float p = ex2_approx(fmaf(s[cc * 32 + e4 * 4 + e], scale_log2, -vv[e]));
                if (c == diag) p = p_self;
                a4[e] += p;
              }
            }
          }
        }
      }
      acc += (a4[0] + a4[1]) + (a4[2] + a4[3]);
    }
    if (!ok) {
      if (lane == 0 && !sm.abort) {
        report_status(status, kStatusTimeout, 62);
        sm.abort = 1;
      }
    } else if (valid) {
      (cols ? part_in : part_out)[static_cast<size_t>(bh) * per + i] = acc;
    }
  }

  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  if (warp == kMmaWarp) tmem_dealloc(tbase, 256);
}

// d_in / d_out of row n = b * per + i: the partial sums of the Hq heads in a fixed order,
// divided by the head count.
__global__ void mass_reduce_kernel(const float* __restrict__ part_in, const float* __restrict__ part_out, int B,
                                   int Hq, int per, float* __restrict__ d_in, float* __restrict__ d_out) {
  // launched as a programmatic dependent of mass_kernel: wait until its partial sums are complete
  // and visible
  griddep_wait();
  griddep_launch_dependents();
  const int n = blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= B * per) return;
  const int b = n / per, i = n % per;
  float si = 0.0f, so = 0.0f;
  for (int h = 0; h < Hq; ++h) {
    const size_t o = (static_cast<size_t>(b) * Hq + h) * per + i;
    si += part_in[o];
    so += part_out[o];
  }
  const float inv = 1.0f / static_cast<float>(Hq);
  d_in[n] = si * inv;
  d_out[n] = so * inv;
}

}  // namespace

size_t mass_workspace_bytes(int B, int Hq, int per) {
  return 2 * sizeof(float) * static_cast<size_t>(B) * Hq * per;
}

int launch_attn_mass(const MassArgs& a, int* status, cudaStream_t stream) {
  if (a.per > kMaxPer) return -2;
  CUtensorMap tq, tk;
  if (!make_bf16_map_4d(&tq, a.q, kD, a.L, a.Hq, a.B, kT) || !make_bf16_map_4d(&tk, a.k_cached, kD, a.L, a.Hkv, a.B, kT))
    return -3;
  const int n_t = (a.per + kT - 1) / kT;
  const long long grid = static_cast<long long>(n_t) * a.Hq * a.B;
  if (grid > 0x7fffffffLL) return -2;
  float* part_in = static_cast<float*>(a.workspace);
  float* part_out = part_in + static_cast<size_t>(a.B) * a.Hq * a.per;
  const size_t smem = sizeof(MassSmem) + 1024 + static_cast<size_t>(n_t) * (4 * sizeof(uint32_t) + kT * sizeof(float));
  // the shared-memory limit is a function attribute of the current context
  static ContextCache<int> setup;
  int unused = 0;
  const int rc = setup.get(&unused, [](int&) {
    const size_t most = sizeof(MassSmem) + 1024 + static_cast<size_t>((kMaxPer + kT - 1) / kT) *
                                                      (4 * sizeof(uint32_t) + kT * sizeof(float));
    return cudaFuncSetAttribute(mass_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(most)) ==
                   cudaSuccess ? 0 : -3;
  });
  if (rc != 0) return rc;
  const float scale_log2 = 1.4426950408889634f / sqrtf(static_cast<float>(kD));
  {
    cudaLaunchAttribute attr[1];
    const cudaLaunchConfig_t cfg =
        pdl_config(dim3(static_cast<unsigned>(grid), 2), dim3(kThreads), smem, stream, attr);
    if (cudaLaunchKernelEx(&cfg, mass_kernel, tq, tk, static_cast<const __nv_bfloat16*>(a.q),
                           static_cast<const __nv_bfloat16*>(a.k_seedmask), a.seed_idx, a.n_seeds, a.lse, a.Hq, a.Hkv,
                           a.L, a.pos0, a.per, n_t, a.tok, a.flags, a.mask_id, scale_log2, part_in, part_out,
                           status) != cudaSuccess)
      return -3;
  }
  if (cudaGetLastError() != cudaSuccess) return -3;
  // the reduction may launch while the partial sums are still being written (programmatic
  // dependent launch); it waits on the device for them, so its launch latency is hidden
  const int rows = a.B * a.per;
  cudaLaunchAttribute attr[1];
  const cudaLaunchConfig_t cfg = pdl_config(dim3(static_cast<unsigned>((rows + 255) / 256)), dim3(256), 0, stream, attr);
  return cudaLaunchKernelEx(&cfg, mass_reduce_kernel, static_cast<const float*>(part_in),
                            static_cast<const float*>(part_out), a.B, a.Hq, a.per, a.d_in, a.d_out) == cudaSuccess
             ? 0 : -3;
}

}  // namespace cover
