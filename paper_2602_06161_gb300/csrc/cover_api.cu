// cover_api.cu - the extern "C" entry points declared in include/cover.h and
// include/cover_debug.h: argument validation, the per-device status block,
// and dispatch to the kernel launchers.
#include <cuda_runtime.h>

#include "context.cuh"
#include "cover.h"
#include "cover_debug.h"
#include "kernels.cuh"

namespace {

// Per-device status block written by kernels that give up on a bounded wait:
// [0] status code, [1] site id, [2] block id, [3] unused.
__device__ int g_status[4];

// Device address of g_status in the current device's context: in host code the
// symbol's name is only a host-side stand-in, so the address is looked up once
// per context (a second device, or a context created anew after cudaDeviceReset,
// gets its own lookup).
int* status_block() {
  static cover::ContextCache<int*> cache;
  int* p = nullptr;
  const int rc = cache.get(&p, [](int*& v) {
    void* a = nullptr;
    if (cudaGetSymbolAddress(&a, g_status) != cudaSuccess || a == nullptr) return -3;
    v = static_cast<int*>(a);
    return 0;
  });
  return rc == 0 ? p : nullptr;
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

int check_attn_args(const void* q, const void* kc, const void* vc, const void* km, const void* vm,
                    const int32_t* seed_idx, int n_seeds, int B, int Hq, int Hkv, int L, int D, const void* out,
                    const float* lse, size_t align) {
  if (q == nullptr || kc == nullptr || vc == nullptr || out == nullptr) return COVER_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || Hkv < 1 || L < 1 || D < 1) return COVER_ERR_INVALID_ARG;
  if (Hq % Hkv != 0) return COVER_ERR_INVALID_ARG;
  if (n_seeds < 0 || n_seeds > L) return COVER_ERR_INVALID_ARG;
  if (n_seeds > 0 && (seed_idx == nullptr || km == nullptr || vm == nullptr)) return COVER_ERR_INVALID_ARG;
  if (!aligned(q, align) || !aligned(kc, align) || !aligned(vc, align) || !aligned(out, align))
    return COVER_ERR_INVALID_ARG;
  if (n_seeds > 0 && (!aligned(km, align) || !aligned(vm, align) || !aligned(seed_idx, 4)))
    return COVER_ERR_INVALID_ARG;
  if (lse != nullptr && !aligned(lse, 4)) return COVER_ERR_INVALID_ARG;
  return COVER_OK;
}

}  // namespace

extern "C" {

int cover_attn_fwd(const void* q, const void* k_cached, const void* v_cached, const void* k_seedmask,
                   const void* v_seedmask, const int32_t* seed_idx, int n_seeds, int B, int Hq, int Hkv, int L, int D,
                   void* out, float* lse, void* stream) {
  int rc = check_attn_args(q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, L, D, out,
                           lse, 16);
  if (rc != COVER_OK) return rc;
  if (D != 128) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::AttnArgs a{q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, L, D, out, lse, L, 0};
  return cover::launch_attn_bf16_sm103(a, st, static_cast<cudaStream_t>(stream));
}

int cover_attn_fwd_f32(const float* q, const float* k_cached, const float* v_cached, const float* k_seedmask,
                       const float* v_seedmask, const int32_t* seed_idx, int n_seeds, int B, int Hq, int Hkv, int L,
                       int D, float* out, float* lse, void* stream) {
  int rc = check_attn_args(q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, L, D, out,
                           lse, 4);
  if (rc != COVER_OK) return rc;
  if (D != 64 && D != 128) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::AttnArgs a{q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, L, D, out, lse, L, 0};
  return cover::launch_attn_f32(a, st, static_cast<cudaStream_t>(stream));
}

static int check_window(int Lq, int Lk, int q0) {
  if (Lq < 1 || Lk < 1 || q0 < 0 || static_cast<long long>(q0) + Lq > Lk) return COVER_ERR_INVALID_ARG;
  return COVER_OK;
}

int cover_attn_fwd_prefix(const void* q, const void* k_cached, const void* v_cached, const void* k_seedmask,
                          const void* v_seedmask, const int32_t* seed_idx, int n_seeds, int B, int Hq, int Hkv,
                          int Lq, int Lk, int q0, int D, void* out, float* lse, void* stream) {
  int rc = check_window(Lq, Lk, q0);
  if (rc != COVER_OK) return rc;
  rc = check_attn_args(q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                       16);
  if (rc != COVER_OK) return rc;
  if (D != 128) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::AttnArgs a{q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                    Lq, q0};
  const int pk = cover::try_launch_attn_window_gqa(a, st, static_cast<cudaStream_t>(stream), false);
  if (pk != cover::kWindowGqaNotTaken) return pk;
  return cover::launch_attn_bf16_sm103(a, st, static_cast<cudaStream_t>(stream));
}

int cover_attn_fwd_prefix_f32(const float* q, const float* k_cached, const float* v_cached, const float* k_seedmask,
                              const float* v_seedmask, const int32_t* seed_idx, int n_seeds, int B, int Hq, int Hkv,
                              int Lq, int Lk, int q0, int D, float* out, float* lse, void* stream) {
  int rc = check_window(Lq, Lk, q0);
  if (rc != COVER_OK) return rc;
  rc = check_attn_args(q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                       4);
  if (rc != COVER_OK) return rc;
  if (D != 64 && D != 128) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::AttnArgs a{q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                    Lq, q0};
  return cover::launch_attn_f32(a, st, static_cast<cudaStream_t>(stream));
}

int cover_seed_route(const int32_t* seed_idx, int n_seeds, int B, int L, int32_t* slot_out, uint32_t* bitmap_out,
                     int32_t* n_invalid_out, void* stream) {
  if (B < 1 || L < 1 || n_seeds < 0 || n_seeds > L) return COVER_ERR_INVALID_ARG;
  if (n_seeds > 0 && seed_idx == nullptr) return COVER_ERR_INVALID_ARG;
  if (slot_out == nullptr || bitmap_out == nullptr || n_invalid_out == nullptr) return COVER_ERR_INVALID_ARG;
  if (B > 65535) return COVER_ERR_UNSUPPORTED;
  return cover::launch_seed_route(seed_idx, n_seeds, B, L, slot_out, bitmap_out, n_invalid_out,
                                  static_cast<cudaStream_t>(stream));
}

int cover_seed_route_debug(const int32_t* seed_idx, int n_seeds, int B, int L, int32_t* slot_out,
                           uint32_t* bitmap_out, int32_t* n_invalid_out, void* stream) {
  return cover_seed_route(seed_idx, n_seeds, B, L, slot_out, bitmap_out, n_invalid_out, stream);
}

size_t cover_score_workspace_bytes(int n_seq) { return n_seq > 0 ? sizeof(uint32_t) * static_cast<size_t>(n_seq) : 0; }

int cover_score_fwd(const void* logits, int N, int V, int n_seq, const int32_t* cur_tok, const float* d_in,
                    const float* d_out, const uint8_t* eligible, int topk, float* maxprob, float* entropy,
                    int32_t* argmax, float* score, int32_t* topk_idx, float* topk_score, void* workspace,
                    void* stream) {
  if (logits == nullptr || maxprob == nullptr || entropy == nullptr || argmax == nullptr || score == nullptr)
    return COVER_ERR_INVALID_ARG;
  if (N < 1 || V < 1 || n_seq < 1 || N % n_seq != 0) return COVER_ERR_INVALID_ARG;
  const int per = N / n_seq;
  if (per > 4096) return COVER_ERR_INVALID_ARG;
  if (topk < 0 || topk > per) return COVER_ERR_INVALID_ARG;
  if (topk > 0 && (topk_idx == nullptr || workspace == nullptr)) return COVER_ERR_INVALID_ARG;
  if (!aligned(logits, 16) || !aligned(maxprob, 4) || !aligned(entropy, 4) || !aligned(argmax, 4) ||
      !aligned(score, 4))
    return COVER_ERR_INVALID_ARG;
  if (workspace != nullptr && !aligned(workspace, 4)) return COVER_ERR_INVALID_ARG;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::ScoreArgs a{logits, N, V, n_seq, cur_tok, d_in, d_out, eligible, topk, maxprob, entropy, argmax,
                     score, topk_idx, topk_score, static_cast<uint32_t*>(workspace)};
  return cover::launch_score(a, st, static_cast<cudaStream_t>(stream));
}

int cover_score_fwd_noalloc(const void* logits, int N, int V, int n_seq, const int32_t* cur_tok, const float* d_in,
                            const float* d_out, const uint8_t* eligible, int topk, float* maxprob, float* entropy,
                            int32_t* argmax, float* score, int32_t* topk_idx, float* topk_score, void* stream) {
  if (logits == nullptr || maxprob == nullptr || entropy == nullptr || argmax == nullptr || score == nullptr)
    return COVER_ERR_INVALID_ARG;
  if (N < 1 || V < 1 || n_seq < 1 || N % n_seq != 0) return COVER_ERR_INVALID_ARG;
  if (n_seq > cover::kNoAllocMaxSegments) return COVER_ERR_INVALID_ARG;
  const int per = N / n_seq;
  if (per > 4096) return COVER_ERR_INVALID_ARG;
  if (topk < 0 || topk > per) return COVER_ERR_INVALID_ARG;
  if (topk > 0 && topk_idx == nullptr) return COVER_ERR_INVALID_ARG;
  if (!aligned(logits, 16) || !aligned(maxprob, 4) || !aligned(entropy, 4) || !aligned(argmax, 4) ||
      !aligned(score, 4))
    return COVER_ERR_INVALID_ARG;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::ScoreArgs a{logits, N, V, n_seq, cur_tok, d_in, d_out, eligible, topk, maxprob, entropy, argmax,
                     score, topk_idx, topk_score, nullptr};
  return cover::launch_score_noalloc(a, st, static_cast<cudaStream_t>(stream));
}

static int seed_kv_call(bool swap, void* k, void* v, const int32_t* seed_idx, int n_seeds, int B, int Hkv, int L,
                        int D, int elem_bytes, void* k_cache, void* v_cache, void* stream) {
  if (k == nullptr || v == nullptr) return COVER_ERR_INVALID_ARG;
  if (B < 1 || Hkv < 1 || L < 1 || D < 1 || n_seeds < 0) return COVER_ERR_INVALID_ARG;
  if (elem_bytes != 2 && elem_bytes != 4) return COVER_ERR_INVALID_ARG;
  const long long row = static_cast<long long>(D) * elem_bytes;
  if (row % 16 != 0 || row > 65536) return COVER_ERR_INVALID_ARG;
  if (n_seeds > 0 && (seed_idx == nullptr || k_cache == nullptr || v_cache == nullptr)) return COVER_ERR_INVALID_ARG;
  if (!aligned(k, 16) || !aligned(v, 16)) return COVER_ERR_INVALID_ARG;
  if (n_seeds > 0 && (!aligned(k_cache, 16) || !aligned(v_cache, 16) || !aligned(seed_idx, 4)))
    return COVER_ERR_INVALID_ARG;
  if (n_seeds == 0) return COVER_OK;
  const int rc = cover::launch_seed_kv(swap, k, v, seed_idx, n_seeds, B, Hkv, L, static_cast<int>(row), k_cache,
                                       v_cache, static_cast<cudaStream_t>(stream));
  return rc == -2 ? COVER_ERR_UNSUPPORTED : rc == 0 ? COVER_OK : COVER_ERR_CUDA;
}

int cover_seed_kv_gather(const void* k, const void* v, const int32_t* seed_idx, int n_seeds, int B, int Hkv, int L,
                         int D, int elem_bytes, void* k_cache, void* v_cache, void* stream) {
  return seed_kv_call(false, const_cast<void*>(k), const_cast<void*>(v), seed_idx, n_seeds, B, Hkv, L, D, elem_bytes,
                      k_cache, v_cache, stream);
}

int cover_seed_kv_override(void* k, void* v, const int32_t* seed_idx, int n_seeds, int B, int Hkv, int L, int D,
                           int elem_bytes, void* k_cache, void* v_cache, void* stream) {
  return seed_kv_call(true, k, v, seed_idx, n_seeds, B, Hkv, L, D, elem_bytes, k_cache, v_cache, stream);
}

size_t cover_decide_workspace_bytes(int N, int n_seq) {
  if (N < 1 || n_seq < 1) return 0;
  // per-segment counters, then u and ln Z per row
  const size_t counters = (sizeof(uint32_t) * static_cast<size_t>(n_seq) + 15) & ~static_cast<size_t>(15);
  return counters + 2 * sizeof(float) * static_cast<size_t>(N);
}

int cover_score_decide_fwd(const void* logits, int N, int V, int n_seq, const float* d_in, const float* d_out,
                           const uint8_t* draft_ok, float tau_draft, int draft_budget, int remask_budget,
                           int mask_id, int min_one, int pos0, int max_seeds, int phase, int32_t* tok,
                           uint8_t* flags, uint8_t* remask_cnt, float* maxprob, float* entropy, int32_t* argmax,
                           float* score, int32_t* seed_idx, int32_t* n_seeds, int32_t* stats, void* workspace,
                           void* stream) {
  if (phase != COVER_DECIDE_ALL && phase != COVER_DECIDE_UPDATE) return COVER_ERR_INVALID_ARG;
  const bool select = phase == COVER_DECIDE_ALL;
  if (logits == nullptr || tok == nullptr || flags == nullptr || remask_cnt == nullptr || maxprob == nullptr ||
      entropy == nullptr || argmax == nullptr || workspace == nullptr)
    return COVER_ERR_INVALID_ARG;
  if (select && (score == nullptr || n_seeds == nullptr)) return COVER_ERR_INVALID_ARG;
  if (N < 1 || V < 1 || n_seq < 1 || N % n_seq != 0 || N / n_seq > 4096) return COVER_ERR_INVALID_ARG;
  if (draft_budget < 0 || remask_budget < 0 || max_seeds < 0) return COVER_ERR_INVALID_ARG;
  if (select && max_seeds > 0 && seed_idx == nullptr) return COVER_ERR_INVALID_ARG;
  if (!aligned(logits, 16) || !aligned(workspace, 16) || !aligned(tok, 4) || !aligned(maxprob, 4) ||
      !aligned(entropy, 4) || !aligned(argmax, 4) || !aligned(score, 4) || !aligned(n_seeds, 4))
    return COVER_ERR_INVALID_ARG;
  if ((seed_idx != nullptr && !aligned(seed_idx, 4)) || (stats != nullptr && !aligned(stats, 4)) ||
      (d_in != nullptr && !aligned(d_in, 4)) || (d_out != nullptr && !aligned(d_out, 4)))
    return COVER_ERR_INVALID_ARG;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const size_t counters_bytes = (sizeof(uint32_t) * static_cast<size_t>(n_seq) + 15) & ~static_cast<size_t>(15);
  float* ws_u = reinterpret_cast<float*>(ws + counters_bytes);
  float* ws_lnz = ws_u + N;
  cover::ScoreArgs a{logits, N, V, n_seq, nullptr, d_in, d_out, nullptr, 0, maxprob, entropy, argmax, score,
                     nullptr, nullptr, reinterpret_cast<uint32_t*>(ws)};
  cover::DecideArgs d{draft_ok, tau_draft, draft_budget, remask_budget, mask_id, min_one != 0 ? 1 : 0, pos0,
                      max_seeds, tok, flags, remask_cnt, seed_idx, n_seeds, stats, ws_u, ws_lnz, phase};
  return cover::launch_score_decide(a, d, st, static_cast<cudaStream_t>(stream));
}

int cover_seed_select_fwd(int N, int n_seq, const float* d_in, const float* d_out, int remask_budget, int mask_id,
                          int pos0, int max_seeds, int32_t* tok, uint8_t* flags, uint8_t* remask_cnt, float* score,
                          int32_t* seed_idx, int32_t* n_seeds, int32_t* stats, void* workspace, void* stream) {
  if (tok == nullptr || flags == nullptr || remask_cnt == nullptr || score == nullptr || n_seeds == nullptr ||
      workspace == nullptr)
    return COVER_ERR_INVALID_ARG;
  if (N < 1 || n_seq < 1 || N % n_seq != 0 || N / n_seq > 4096) return COVER_ERR_INVALID_ARG;
  if (remask_budget < 0 || max_seeds < 0) return COVER_ERR_INVALID_ARG;
  if (max_seeds > 0 && seed_idx == nullptr) return COVER_ERR_INVALID_ARG;
  if (!aligned(workspace, 16) || !aligned(tok, 4) || !aligned(score, 4) || !aligned(n_seeds, 4) ||
      (seed_idx != nullptr && !aligned(seed_idx, 4)) || (stats != nullptr && !aligned(stats, 4)) ||
      (d_in != nullptr && !aligned(d_in, 4)) || (d_out != nullptr && !aligned(d_out, 4)))
    return COVER_ERR_INVALID_ARG;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const size_t counters_bytes = (sizeof(uint32_t) * static_cast<size_t>(n_seq) + 15) & ~static_cast<size_t>(15);
  float* ws_u = reinterpret_cast<float*>(ws + counters_bytes);
  cover::DecideArgs d{nullptr, 0.0f, 0, remask_budget, mask_id, 0, pos0, max_seeds, tok, flags, remask_cnt,
                      seed_idx, n_seeds, stats, ws_u, ws_u + N, COVER_DECIDE_ALL};
  return cover::launch_seed_select(N, n_seq, d, d_in, d_out, score, static_cast<cudaStream_t>(stream)) == 0
             ? COVER_OK
             : COVER_ERR_CUDA;
}

size_t cover_attn_mass_workspace_bytes(int B, int Hq, int per) {
  if (B < 1 || Hq < 1 || per < 1) return 0;
  return cover::mass_workspace_bytes(B, Hq, per);
}

int cover_attn_mass_fwd(const void* q, const void* k_cached, const void* k_seedmask, const int32_t* seed_idx,
                        int n_seeds, const float* lse, int B, int Hq, int Hkv, int L, int D, const int32_t* tok,
                        const uint8_t* flags, int mask_id, int pos0, int per, void* workspace, float* d_in,
                        float* d_out, void* stream) {
  if (q == nullptr || k_cached == nullptr || lse == nullptr || tok == nullptr || flags == nullptr ||
      workspace == nullptr || d_in == nullptr || d_out == nullptr)
    return COVER_ERR_INVALID_ARG;
  if (B < 1 || Hq < 1 || Hkv < 1 || L < 1 || D < 1 || per < 1 || Hq % Hkv != 0) return COVER_ERR_INVALID_ARG;
  if (pos0 < 0 || static_cast<long long>(pos0) + per > L) return COVER_ERR_INVALID_ARG;
  if (n_seeds < 0 || n_seeds > L || (n_seeds > 0 && (seed_idx == nullptr || k_seedmask == nullptr)))
    return COVER_ERR_INVALID_ARG;
  if (!aligned(q, 16) || !aligned(k_cached, 16) || !aligned(workspace, 16) || !aligned(lse, 4) ||
      !aligned(tok, 4) || !aligned(d_in, 4) || !aligned(d_out, 4))
    return COVER_ERR_INVALID_ARG;
  if (n_seeds > 0 && (!aligned(k_seedmask, 16) || !aligned(seed_idx, 4))) return COVER_ERR_INVALID_ARG;
  if (D != 128 || per > cover::kMassMaxPer) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::MassArgs a{q, k_cached, k_seedmask, seed_idx, n_seeds, lse, B, Hq, Hkv, L, pos0, per, tok, flags,
                    mask_id, workspace, d_in, d_out};
  const int rc = cover::launch_attn_mass(a, st, static_cast<cudaStream_t>(stream));
  return rc == -2 ? COVER_ERR_UNSUPPORTED : rc == 0 ? COVER_OK : COVER_ERR_CUDA;
}

// Synchronises the stream, reads the status block into host[4] and clears it.
static int read_status(void* stream, int* host) {
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return COVER_ERR_CUDA;
  if (cudaMemcpyAsync(host, st, 4 * sizeof(int), cudaMemcpyDeviceToHost, s) != cudaSuccess) return COVER_ERR_CUDA;
  if (cudaMemsetAsync(st, 0, 4 * sizeof(int), s) != cudaSuccess) return COVER_ERR_CUDA;
  if (cudaStreamSynchronize(s) != cudaSuccess) return COVER_ERR_CUDA;
  return COVER_OK;
}

int cover_device_status(void* stream) {
  int host[4] = {0, 0, 0, 0};
  const int rc = read_status(stream, host);
  return rc != COVER_OK ? rc : host[0];
}

int cover_debug_status_detail(int32_t* detail, void* stream) {
  if (detail == nullptr) return COVER_ERR_INVALID_ARG;
  int host[4] = {0, 0, 0, 0};
  const int rc = read_status(stream, host);
  if (rc != COVER_OK) return rc;
  for (int i = 0; i < 3; ++i) detail[i] = host[i];
  return COVER_OK;
}

const char* cover_status_str(int code) {
  switch (code) {
    case COVER_OK: return "COVER_OK";
    case COVER_ERR_INVALID_ARG: return "COVER_ERR_INVALID_ARG";
    case COVER_ERR_UNSUPPORTED: return "COVER_ERR_UNSUPPORTED";
    case COVER_ERR_CUDA: return "COVER_ERR_CUDA";
    case COVER_ERR_DEVICE_TIMEOUT: return "COVER_ERR_DEVICE_TIMEOUT";
    default: return "COVER_ERR_UNKNOWN";
  }
}

int cover_debug_umma_tile(const void* a, const void* b, const void* p, const void* v, float* c1, float* c2,
                          void* stream) {
  if (a == nullptr || b == nullptr || p == nullptr || v == nullptr || c1 == nullptr || c2 == nullptr)
    return COVER_ERR_INVALID_ARG;
  if (!aligned(a, 16) || !aligned(b, 16) || !aligned(p, 16) || !aligned(v, 16) || !aligned(c1, 16) ||
      !aligned(c2, 16))
    return COVER_ERR_INVALID_ARG;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  return cover::launch_umma_tile(a, b, p, v, c1, c2, st, static_cast<cudaStream_t>(stream));
}

int cover_debug_attn_prefix_packed(const void* q, const void* k_cached, const void* v_cached, const void* k_seedmask,
                                   const void* v_seedmask, const int32_t* seed_idx, int n_seeds, int B, int Hq,
                                   int Hkv, int Lq, int Lk, int q0, int D, void* out, float* lse, int fault_cta,
                                   int limit_us, void* stream) {
  if (limit_us < 0 || limit_us > 2000000) return COVER_ERR_INVALID_ARG;
  int rc = check_window(Lq, Lk, q0);
  if (rc != COVER_OK) return rc;
  rc = check_attn_args(q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                       16);
  if (rc != COVER_OK) return rc;
  if (D != 128) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::AttnArgs a{q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                    Lq, q0};
  a.fault_cta = fault_cta;
  a.wait_ns = static_cast<uint64_t>(limit_us) * 1000ull;
  rc = cover::try_launch_attn_window_gqa(a, st, static_cast<cudaStream_t>(stream), true);
  return rc == cover::kWindowGqaNotTaken ? COVER_ERR_UNSUPPORTED : rc;
}

int cover_debug_window_model(int B, int Hq, int Hkv, int Lq, int Lk, int q0, int n_sm, const int32_t* max_clusters,
                             int32_t* choice, double* times) {
  if (B < 1 || Hq < 1 || Hkv < 1 || Hq % Hkv != 0 || n_sm < 1 || max_clusters == nullptr || choice == nullptr ||
      times == nullptr)
    return COVER_ERR_INVALID_ARG;
  const int rc = check_window(Lq, Lk, q0);
  if (rc != COVER_OK) return rc;
  for (int c = 0; c < 8; ++c)
    if (max_clusters[c] < 0) return COVER_ERR_INVALID_ARG;
  cover::AttnArgs a{nullptr, nullptr, nullptr, nullptr, nullptr, nullptr, 0, B, Hq, Hkv, Lk, 128, nullptr, nullptr,
                    Lq, q0};
  const cover::WindowChoice c = cover::window_gqa_model(a, n_sm, max_clusters);
  choice[0] = c.supported;
  choice[1] = c.resident;
  choice[2] = c.packed;
  choice[3] = c.T;
  choice[4] = c.nsplit;
  choice[5] = c.n_qt;
  times[0] = c.packed_us;
  times[1] = c.square_us;
  return COVER_OK;
}

int cover_debug_attn_fault(const void* q, const void* k_cached, const void* v_cached, const void* k_seedmask,
                           const void* v_seedmask, const int32_t* seed_idx, int n_seeds, int B, int Hq, int Hkv,
                           int Lq, int Lk, int q0, int D, void* out, float* lse, int fault_cta, int fault_entry,
                           int limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 2000000) return COVER_ERR_INVALID_ARG;
  int rc = check_window(Lq, Lk, q0);
  if (rc != COVER_OK) return rc;
  rc = check_attn_args(q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                       16);
  if (rc != COVER_OK) return rc;
  if (D != 128) return COVER_ERR_UNSUPPORTED;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  cover::AttnArgs a{q, k_cached, v_cached, k_seedmask, v_seedmask, seed_idx, n_seeds, B, Hq, Hkv, Lk, D, out, lse,
                    Lq, q0};
  a.fault_cta = fault_cta;
  a.fault_entry = fault_entry;
  a.wait_ns = static_cast<uint64_t>(limit_us) * 1000ull;
  return cover::launch_attn_bf16_sm103(a, st, static_cast<cudaStream_t>(stream));
}

int cover_debug_wait_timeout(int limit_us, void* stream) {
  if (limit_us < 1 || limit_us > 2000000) return COVER_ERR_INVALID_ARG;
  int* st = status_block();
  if (st == nullptr) return COVER_ERR_CUDA;
  return cover::launch_wait_timeout(static_cast<uint64_t>(limit_us) * 1000ull, st,
                                    static_cast<cudaStream_t>(stream));
}

}  // extern "C"
