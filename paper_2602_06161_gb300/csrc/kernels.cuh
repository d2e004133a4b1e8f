// kernels.cuh - launchers implemented by the kernel translation units and
// called by the C-ABI layer (cover_api.cu). Arguments are already validated.
// Each returns 0 or a negative cover_status_t code (COVER_ERR_CUDA = -3).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace cover {

struct AttnArgs {
  const void* q;
  const void* k_cached;
  const void* v_cached;
  const void* k_seedmask;
  const void* v_seedmask;
  const int32_t* seed_idx;
  int n_seeds;
  int B, Hq, Hkv, L, D;
  void* out;
  float* lse;
};

int launch_attn_bf16_sm103(const AttnArgs& a, int* status, cudaStream_t stream);
int launch_attn_f32(const AttnArgs& a, int* status, cudaStream_t stream);

int launch_seed_route(const int32_t* seed_idx, int n_seeds, int B, int L, int32_t* slot_out, uint32_t* bitmap_out,
                      int32_t* n_invalid_out, cudaStream_t stream);

struct ScoreArgs {
  const void* logits;
  int N, V, n_seq;
  const int32_t* cur_tok;
  const float* d_in;
  const float* d_out;
  const uint8_t* eligible;
  int topk;
  float* maxprob;
  float* entropy;
  int32_t* argmax;
  float* score;
  int32_t* topk_idx;
  float* topk_score;
  uint32_t* counters;   // [n_seq], zero on entry, zero again on exit
};

int launch_score(const ScoreArgs& a, int* status, cudaStream_t stream);

// Same as launch_score, with the counters in a fixed device array of the
// library (a.counters is ignored). Returns -1 if a.n_seq > kNoAllocMaxSegments.
constexpr int kNoAllocMaxSegments = 4096;
int launch_score_noalloc(ScoreArgs a, int* status, cudaStream_t stream);

int launch_umma_tile(const void* a, const void* b, const void* p, const void* v, float* c1, float* c2, int* status,
                     cudaStream_t stream);
int launch_wait_timeout(uint64_t limit_ns, int* status, cudaStream_t stream);

}  // namespace cover
