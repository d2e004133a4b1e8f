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
  int B, Hq, Hkv, L, D;   // L: memory length (keys / values)
  void* out;
  float* lse;
  int Lq = 0;             // query rows; query row r sits at memory position q0 + r
  int q0 = 0;
  // self-test only (bf16 kernel): CTA fault_cta leaves out the K load of its KV ring entry
  // fault_entry, and every bounded wait gives up after wait_ns (0: the default limit)
  int fault_cta = -1;
  int fault_entry = -1;
  uint64_t wait_ns = 0;
};

int launch_attn_bf16_sm103(const AttnArgs& a, int* status, cudaStream_t stream);

// Prefix-cache windows of grouped-query heads (attn_window_gqa.cu): the G = Hq / Hkv query heads
// of a KV head packed into common Q tiles, the keys split over a cluster of up to 8 CTAs.
// Supported for a window (Lq != L or q0 != 0) with G >= 2, Lq <= kMaxWindowGqaRows,
// G * Lq <= kMaxWindowGqaPacked and at most 8 * kMaxWindowGqaSteps KV tiles of 128 keys.
// try_launch_attn_window_gqa launches it where it is supported and (unless `force`) predicted to
// be faster than the square kernel's window path, and returns kWindowGqaNotTaken otherwise.
// With `force`, a.fault_cta >= 0 or a.wait_ns > 0 select its self-test instance: CTA fault_cta
// leaves out the K load of its first KV tile, every bounded wait gives up after wait_ns.
constexpr int kMaxWindowGqaRows = 256;
constexpr int kMaxWindowGqaPacked = 1024;
constexpr int kMaxWindowGqaSteps = 8;
constexpr int kWindowGqaNotTaken = 1;
int try_launch_attn_window_gqa(const AttnArgs& a, int* status, cudaStream_t stream, bool force);
// The launch-time choice for a window on a GPU with n_sm SMs, where max_clusters[c - 1] clusters
// of c CTAs of the packed kernel can be resident at once (c = 1 .. 8). Host arithmetic only.
struct WindowChoice {
  bool supported;          // the packed kernel runs this shape
  bool resident;           // a cluster of its nsplit CTAs can be resident
  bool packed;             // it is predicted faster than the square kernel
  int T, nsplit, n_qt;     // KV tiles per CTA, CTAs per cluster, Q tiles per KV head
  long long clusters;
  double packed_us, square_us;
};
WindowChoice window_gqa_model(const AttnArgs& a, int n_sm, const int* max_clusters);
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

// One decoding step's decisions, run by the last CTA of each segment after the
// per-row scoring (a.topk, a.eligible, a.cur_tok, a.topk_idx and a.topk_score
// are unused; a.score receives the seed scores of the updated state).
struct DecideArgs {
  const uint8_t* draft_ok;   // [N] or null (every masked row may be drafted)
  float tau;                 // drafting / Replace threshold on the confidence
  int budget;                // at most this many drafted rows per segment
  int remask_budget;         // rows with this many ReMasks are not selected
  int mask_id;               // token id of [MASK]
  int min_one;               // draft the lowest-entropy masked row when none passes tau
  int pos0;                  // position of a segment's first row
  int max_seeds;             // seed capacity per segment
  int32_t* tok;              // [N] in: current tokens, out: updated tokens
  uint8_t* flags;            // [N] bit 0 in: previous seeds, out: new seeds
  uint8_t* remask_cnt;       // [N] in / out
  int32_t* seed_idx;         // [n_seq, max_seeds] positions, -1 padded
  int32_t* n_seeds;          // [n_seq]
  int32_t* stats;            // [n_seq, 6] or null
  float* ws_u;               // [N] workspace: u of the current token, then of the updated one
  float* ws_lnz;             // [N] workspace: ln Z (= u of the greedy token)
  int phase = 0;             // 0: update and select; 1: update only (flag bit 1 marks drafted rows)
};
constexpr int kDecideStats = 6;   // drafted, kept, replaced, remasked, n_t, n_above
int launch_score_decide(const ScoreArgs& a, const DecideArgs& d, int* status, cudaStream_t stream);
// Section 5.3 selection alone, from the state and workspace an update phase left.
int launch_seed_select(int N, int n_seq, const DecideArgs& d, const float* d_in, const float* d_out, float* score,
                       cudaStream_t stream);

// Same as launch_score, with the counters in a fixed device array of the
// library (a.counters is ignored). Returns -1 if a.n_seq > kNoAllocMaxSegments.
constexpr int kNoAllocMaxSegments = 4096;
int launch_score_noalloc(ScoreArgs a, int* status, cudaStream_t stream);

// d_in / d_out of Section 5.3 for the response rows pos0 .. pos0 + per - 1 of
// every batch row, from the attention pass's q, K', masked-input keys and lse.
struct MassArgs {
  const void* q;             // [B, Hq, L, 128] bf16
  const void* k_cached;      // [B, Hkv, L, 128] bf16 (K')
  const void* k_seedmask;    // [B, Hkv, S, 128] bf16
  const int32_t* seed_idx;   // [B, S]
  int n_seeds;
  const float* lse;          // [B, Hq, L] natural-log lse of the attention pass
  int B, Hq, Hkv, L, pos0, per;
  const int32_t* tok;        // [B * per] updated tokens
  const uint8_t* flags;      // [B * per] bit 1: drafted in this step
  int mask_id;
  void* workspace;           // mass_workspace_bytes(B, Hq, per)
  float* d_in;               // [B * per]
  float* d_out;              // [B * per]
};
constexpr int kMassMaxPer = 16384;   // a response block's per-column data is staged in shared memory
size_t mass_workspace_bytes(int B, int Hq, int per);
int launch_attn_mass(const MassArgs& a, int* status, cudaStream_t stream);

// Seed K/V cache (Section 5.1): gather (override_swap = false) or the override
// swap (true) of rows of row_bytes (a multiple of 16) bytes.
int launch_seed_kv(bool override_swap, void* k, void* v, const int32_t* seed_idx, int n_seeds, int B, int Hkv, int L,
                   int row_bytes, void* k_cache, void* v_cache, cudaStream_t stream);

int launch_umma_tile(const void* a, const void* b, const void* p, const void* v, float* c1, float* c2, int* status,
                     cudaStream_t stream);
int launch_wait_timeout(uint64_t limit_ns, int* status, cudaStream_t stream);

}  // namespace cover
