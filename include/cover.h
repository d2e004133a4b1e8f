/*
 * cover.h - C ABI of the COVER override-attention and seed-scoring kernels
 * (single GB300 GPU, sm_103a).
 *
 * COVER ("Stop the Flip-Flop: Context-Preserving Verification for Fast
 * Revocable Diffusion Decoding") verifies previously decoded "seed" positions
 * in the same forward pass that drafts new tokens. Section 5.1: the seeds are
 * masked in the input, their key/value columns are overridden with the states
 * cached at the previous step (memory K', V'), every query attends once over
 * K', V', and each seed query's own diagonal entry is restored to the pair
 * (k_i, v_i) computed from the masked input (leave-one-out view). Appendix B
 * gives the closed form of that diagonal correction.
 *
 * Conventions for every entry point:
 *  - Pointers are DEVICE pointers owned by the caller, unless stated otherwise.
 *    The library allocates no device memory and keeps no per-call state.
 *  - Calls are asynchronous on `stream` (a cudaStream_t; NULL = legacy default
 *    stream). Argument errors are returned synchronously, before any launch.
 *  - Every kernel is launched as a programmatic dependent of the stream's
 *    previous kernel: its CTAs may start while that kernel finishes, but they
 *    read and write no global memory before it has completed and its writes
 *    are visible, so stream order holds as for plain launches. Work after an
 *    event wait or a copy on the stream is ordered as usual.
 *  - Kernels never trap. A kernel that gives up on an internal wait (bounded at
 *    about one second) records COVER_ERR_DEVICE_TIMEOUT in a per-device status
 *    word; read and clear it with cover_device_status().
 *  - Tensors are dense and contiguous (row-major, last index fastest).
 */
#ifndef COVER_H_
#define COVER_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  COVER_OK = 0,
  COVER_ERR_INVALID_ARG = -1,    /* null required pointer, bad size, misaligned pointer */
  COVER_ERR_UNSUPPORTED = -2,    /* valid request outside what the kernels implement (e.g. head dim) */
  COVER_ERR_CUDA = -3,           /* a CUDA runtime call or launch failed */
  COVER_ERR_DEVICE_TIMEOUT = -4  /* a kernel gave up on a bounded internal wait (status word only) */
} cover_status_t;

/*
 * Two-view override attention, bf16 in / bf16 out, fp32 accumulation.
 * Section 5.1 (Attn(Q, K', V') over the overridden memory, softmax scale
 * 1/sqrt(d)) and Appendix B.1-B.4 (diagonal correction of seed queries).
 *
 *   q          [B, Hq,  L, D] bf16  queries from the masked-seed input
 *   k_cached   [B, Hkv, L, D] bf16  overridden memory K' (seed columns already
 *   v_cached   [B, Hkv, L, D] bf16  hold the previous step's cached states)
 *   k_seedmask [B, Hkv, n_seeds, D] bf16  row s = key   of position seed_idx[b, s]
 *   v_seedmask [B, Hkv, n_seeds, D] bf16  row s = value of position seed_idx[b, s]
 *                                   computed from the masked input (may be NULL
 *                                   when n_seeds == 0)
 *   seed_idx   [B, n_seeds] int32   seed positions per batch row, any order.
 *                                   Entries outside [0, L) are ignored; if a
 *                                   position repeats, the lowest slot s is used.
 *   out        [B, Hq, L, D] bf16   o_i (corrected for seed rows)
 *   lse        [B, Hq, L] fp32      natural-log log-sum-exp of the scaled
 *                                   scores of each row's own view (NULL = skip)
 *
 * Query head hq reads KV head hq / (Hq / Hkv) (contiguous groups). No causal
 * mask. For non-seed rows the result is plain attention over K', V'; for a
 * seed row i the diagonal term uses (k_i, v_i) instead of (k'_i, v'_i).
 *
 * Requirements: D == 128 (else COVER_ERR_UNSUPPORTED); B, Hq, Hkv, L >= 1;
 * Hq % Hkv == 0; 0 <= n_seeds <= L; q, k_cached, v_cached, out, k_seedmask,
 * v_seedmask 16-byte aligned; lse 4-byte aligned. Any L >= 1 is supported.
 * Otherwise COVER_ERR_INVALID_ARG. The inputs must not alias out / lse.
 */
int cover_attn_fwd(const void* q, const void* k_cached, const void* v_cached,
                   const void* k_seedmask, const void* v_seedmask,
                   const int32_t* seed_idx, int n_seeds,
                   int B, int Hq, int Hkv, int L, int D,
                   void* out, float* lse, void* stream);

/*
 * The same operation in fp32 throughout (float tensors, fp32 FMA on CUDA
 * cores, accurate expf). Intended for small fp32 checks. D in {64, 128}.
 * Same layouts, ownership and errors as cover_attn_fwd (4-byte alignment).
 */
int cover_attn_fwd_f32(const float* q, const float* k_cached, const float* v_cached,
                       const float* k_seedmask, const float* v_seedmask,
                       const int32_t* seed_idx, int n_seeds,
                       int B, int Hq, int Hkv, int L, int D,
                       float* out, float* lse, void* stream);

/*
 * Prefix-cache variant (Section 6.6 "Compatibility with Fast-dLLM": only the
 * active block's queries are recomputed while the memory holds every
 * position). The memory k_cached / v_cached is [B, Hkv, Lk, D] (overridden at
 * the seeds, as above); the queries q and the outputs out / lse are
 * [B, Hq, Lq, D] / [B, Hq, Lq], and query row r sits at memory position
 * q0 + r (0 <= q0, q0 + Lq <= Lk). seed_idx holds memory positions in
 * [0, Lk); a seed inside [q0, q0 + Lq) gets its leave-one-out view on the
 * diagonal column q0 + r, a seed outside the window affects only the memory.
 * With Lq = Lk and q0 = 0 this is cover_attn_fwd. Types, layouts, ownership
 * and errors as cover_attn_fwd / cover_attn_fwd_f32, plus
 * COVER_ERR_INVALID_ARG for Lq < 1, Lk < 1, q0 < 0 or q0 + Lq > Lk.
 * The bf16 call may run a window of grouped-query heads (G = Hq / Hkv >= 2,
 * Lq <= 256, G * Lq <= 1024, Lk <= 8192) on a kernel of its own: the G query
 * heads of a KV head packed into common Q tiles, the keys split over a cluster
 * of up to 8 CTAs that combine their partial softmax states. It does so where
 * a launch-time model (the clusters that fit on the GPU at once, the KV steps
 * of each kernel's longest chain) predicts it to be faster than the square
 * kernel. Its rows agree with the square kernel's up to rounding (not bit for
 * bit); any other window runs on the square kernel, whose window rows equal
 * the square launch's.
 */
int cover_attn_fwd_prefix(const void* q, const void* k_cached, const void* v_cached,
                          const void* k_seedmask, const void* v_seedmask,
                          const int32_t* seed_idx, int n_seeds,
                          int B, int Hq, int Hkv, int Lq, int Lk, int q0, int D,
                          void* out, float* lse, void* stream);
int cover_attn_fwd_prefix_f32(const float* q, const float* k_cached, const float* v_cached,
                              const float* k_seedmask, const float* v_seedmask,
                              const int32_t* seed_idx, int n_seeds,
                              int B, int Hq, int Hkv, int Lq, int Lk, int q0, int D,
                              float* out, float* lse, void* stream);

/*
 * Seed routing as the attention kernels see it (seed-set semantics of
 * Sections 3 and 5.1), exported for checking.
 *   slot_out   [B, L] int32: slot s of the seed naming position r, else -1
 *   bitmap_out [B, ceil(L/128), 4] uint32: bit r%32 of word (r%128)/32 of
 *              tile r/128 is set iff slot_out[b, r] >= 0
 *   n_invalid_out [1] int32: entries out of [0, L) plus repeated positions
 * seed_idx may be NULL when n_seeds == 0. Requirements: B, L >= 1,
 * 0 <= n_seeds <= L (else COVER_ERR_INVALID_ARG).
 */
int cover_seed_route(const int32_t* seed_idx, int n_seeds, int B, int L,
                     int32_t* slot_out, uint32_t* bitmap_out, int32_t* n_invalid_out,
                     void* stream);
/* The same function under the name the boundary's specification gives it
 * (cover_seed_route_debug); identical arguments, results and errors. */
int cover_seed_route_debug(const int32_t* seed_idx, int n_seeds, int B, int L,
                           int32_t* slot_out, uint32_t* bitmap_out, int32_t* n_invalid_out,
                           void* stream);

/*
 * Bytes of device workspace cover_score_fwd needs for n_seq segments.
 * The caller allocates it once, fills it with zeros, and may pass the same
 * buffer to every later call (each call leaves it zeroed again). Calls that
 * share one workspace must not run concurrently on the GPU.
 */
size_t cover_score_workspace_bytes(int n_seq);

/*
 * Fused per-position scoring over the vocabulary and top-k seed selection.
 * Section 3 (greedy token y_hat = argmax p, confidence c = max p), Section 6.1
 * (entropy-ordered unmasking: H = -sum p ln p), Section 5.3 (uncertainty
 * u = -log p(y), Score = u (1 + d_in)/(1 + d_out), top-k over eligible rows).
 *
 *   logits  [N, V] bf16   one row per scored position, softmax at temperature 1
 *   n_seq               rows split into n_seq equal consecutive segments
 *                       (sequences); top-k is taken per segment
 *   cur_tok [N] int32   current token y of each row; NULL => y = argmax row
 *   d_in, d_out [N] f32 influence / drift terms of the score; NULL => 0
 *   eligible [N] uint8  nonzero = row may be selected; NULL => all rows
 *   topk                k per segment (0 <= k <= N / n_seq)
 * Outputs (per row): maxprob = c, entropy = H, argmax = y_hat (lowest index
 * among equal maxima), score = Score. Per segment: topk_idx [n_seq, topk]
 * (row offsets within the segment, by score descending then index
 * ascending; -1 where fewer than k rows are eligible) and topk_score
 * [n_seq, topk] (NULL = skip; -inf where idx is -1).
 * workspace: cover_score_workspace_bytes(n_seq) zero-filled bytes (see above).
 *
 * Requirements: N, V >= 1; 1 <= n_seq; N % n_seq == 0; N / n_seq <= 4096;
 * logits 16-byte aligned (any V; rows need not be 16-byte aligned).
 * A cur_tok entry outside [0, V) yields NaN u and score for that row.
 * Non-finite logits give unspecified results. Otherwise COVER_ERR_INVALID_ARG.
 */
int cover_score_fwd(const void* logits, int N, int V, int n_seq,
                    const int32_t* cur_tok, const float* d_in, const float* d_out,
                    const uint8_t* eligible, int topk,
                    float* maxprob, float* entropy, int32_t* argmax, float* score,
                    int32_t* topk_idx, float* topk_score,
                    void* workspace, void* stream);

/*
 * cover_score_fwd without a workspace argument. The paper has no counterpart:
 * this entry point exists for callers that cannot allocate device memory for
 * a workspace - for example a serving loop that reserves all of its GPU
 * memory up front and forbids allocation afterwards, or a plugin interface
 * that hands the library its inputs and outputs but no allocator.
 *
 * Same arguments, layouts, results and errors as cover_score_fwd. The
 * per-sequence counters that cover_score_fwd keeps in the caller's workspace
 * live here in one fixed device array of the library, sized for at most
 * COVER_NOALLOC_MAX_SEQ (4096) sequences; n_seq beyond that returns
 * COVER_ERR_INVALID_ARG. Every device that loads the library holds this
 * 16 KB array until the process exits. The call allocates nothing: no
 * cudaMalloc / cudaFree, no allocating library routine; it clears the
 * counters it uses with an asynchronous memset on `stream`, then launches.
 *
 * The first call on each device looks up the array's device address
 * (cudaGetSymbolAddress, with that device current); make that first call
 * before any stream capture begins. The address is kept per context: after
 * cudaDeviceReset the next call (again outside any capture) looks it up in
 * the new context. All calls share the one array: calls
 * that overlap on the GPU (different streams, or different host threads
 * without ordering) race on it and can return wrong top-k results.
 */
#define COVER_NOALLOC_MAX_SEQ 4096
int cover_score_fwd_noalloc(const void* logits, int N, int V, int n_seq,
                            const int32_t* cur_tok, const float* d_in, const float* d_out,
                            const uint8_t* eligible, int topk,
                            float* maxprob, float* entropy, int32_t* argmax, float* score,
                            int32_t* topk_idx, float* topk_score, void* stream);

/*
 * Seed key/value cache (Section 5.1, "KV cache override yields a stable
 * drafting view"), per layer. k, v: the layer's states [B, Hkv, L, D];
 * k_cache, v_cache: [B, Hkv, n_seeds, D]; seed_idx: int32 [B, n_seeds]
 * positions (the row of the previous step's cover_score_decide_fwd output
 * works as is). Elements are elem_bytes (2 for bf16, 4 for fp32) bytes; a row
 * (D * elem_bytes) must be a multiple of 16 bytes and every pointer 16-byte
 * aligned. All pointers are device pointers owned by the caller.
 *
 * A slot names its position when the position is in [0, L) and no lower slot
 * of the same batch row names it (the lowest slot wins, as in cover_attn_fwd).
 *
 * cover_seed_kv_gather (at selection, step t-1): k_cache[b, h, s] =
 *   k[b, h, seed_idx[b, s]], likewise v; a slot with an out-of-range position
 *   gets zeros (a repeated position is copied again).
 * cover_seed_kv_override (at step t, after the layer's k, v were computed from
 *   the input with the seeds masked): swaps row seed_idx[b, s] of k / v with
 *   row s of k_cache / v_cache for every slot that names a position. Afterwards
 *   k, v hold the overridden memory K', V' and k_cache, v_cache hold the
 *   masked-input pairs (k_i, v_i): exactly cover_attn_fwd's k_cached,
 *   v_cached, k_seedmask, v_seedmask. Slots that name no position leave both
 *   buffers untouched.
 * n_seeds = 0 is a no-op (seed pointers may then be NULL).
 * Errors: COVER_ERR_INVALID_ARG for a NULL required pointer, B, Hkv, L or D
 * < 1, n_seeds < 0, elem_bytes not 2 or 4, a row that is not a multiple of 16
 * bytes or is longer than 64 KB, or a misaligned pointer; COVER_ERR_UNSUPPORTED if B * Hkv > 2^31 - 1 or
 * n_seeds > 1048560; COVER_ERR_CUDA for a launch failure.
 */
int cover_seed_kv_gather(const void* k, const void* v, const int32_t* seed_idx, int n_seeds,
                         int B, int Hkv, int L, int D, int elem_bytes,
                         void* k_cache, void* v_cache, void* stream);
int cover_seed_kv_override(void* k, void* v, const int32_t* seed_idx, int n_seeds,
                           int B, int Hkv, int L, int D, int elem_bytes,
                           void* k_cache, void* v_cache, void* stream);

/*
 * One decoding step's decisions, fused behind the scoring pass
 * (Section 5.2 "Threshold drafting" and the Keep / Replace / ReMask revision
 * rule, Section 3 state update, Section 5.3 stability-aware seed score,
 * adaptive revision rate and seed exclusions).
 *
 * The N rows split into n_seq equal segments (sequences); row i of a segment
 * is response position pos0 + i. Per row the scoring pass computes c = max p,
 * y_hat = argmax p (ties to the lower index) and H exactly as
 * cover_score_fwd, and u = -log p(tok) for the current token. Then, per
 * segment (state arrays updated in place):
 *   1. Drafting: among rows with tok == mask_id and draft_ok != 0 (all such
 *      rows when draft_ok is NULL), those with c > tau_draft; if more than
 *      draft_budget, the largest c are kept (ties to the lower index). If none
 *      is drafted and min_one != 0, the allowed masked row with the lowest H is
 *      drafted (ties to the lower index). Drafted rows take tok = y_hat.
 *   2. Revision of the previous seeds (rows with flag bit COVER_FLAG_SEED set
 *      and tok != mask_id): Keep if y_hat == tok; else Replace (tok = y_hat)
 *      if c > tau_draft; else ReMask (tok = mask_id, remask_cnt + 1, saturating
 *      at 255).
 *   3. Seed score of every unmasked row of the updated state, in fp32:
 *      score = (u * (1 + d_in)) / (1 + d_out), with u = ln Z = -log c for
 *      drafted and replaced rows and the current token's u otherwise (NULL
 *      d_in / d_out = 0). Masked rows and non-finite scores get -INFINITY.
 *   4. Adaptive revision rate: n_t = rows with a finite score, n_above = rows
 *      with n_t * score > sum of the scores (fp64; this is n_t * pi_t),
 *      k = min(ceil(sqrt(n_above)), max_seeds).
 *   5. New seeds: the k highest-scoring rows (ties to the lower index) among
 *      the scored rows that were not previous seeds and have
 *      remask_cnt < remask_budget; fewer if fewer are eligible. Their flag bit
 *      COVER_FLAG_SEED is set and every other row's is cleared (other flag bits
 *      are kept); seed_idx[seg, 0..n_seeds) lists their positions pos0 + i in
 *      order, the rest of the row is -1, so it can be passed to
 *      cover_attn_fwd as the next step's seed_idx with n_seeds = max_seeds.
 *
 * logits   bf16 [N, V] row-major, 16-byte aligned (device).
 * d_in, d_out, draft_ok: [N] or NULL (device).
 * tok      int32 [N] (device, in/out); flags, remask_cnt uint8 [N] (in/out).
 * maxprob, entropy, score float [N]; argmax int32 [N] (device, out).
 * seed_idx int32 [n_seq, max_seeds] (device, out; may be NULL if max_seeds is
 *          0); n_seeds int32 [n_seq] (out); stats int32 [n_seq, 6] or NULL:
 *          drafted, kept, replaced, remasked, n_t, n_above per segment.
 * workspace: cover_decide_workspace_bytes(N, n_seq) bytes of device memory,
 *          16-byte aligned, zero-filled before its first use; it is left ready
 *          for the next call on the same stream.
 * phase COVER_DECIDE_ALL runs steps 1-5 with the given d_in / d_out.
 * phase COVER_DECIDE_UPDATE runs steps 1-2 only: it writes maxprob, entropy,
 *   argmax, the updated tok / remask_cnt, flag bit COVER_FLAG_DRAFTED on the
 *   rows drafted in this step (bit COVER_FLAG_SEED still marks the previous
 *   seeds), stats[.., 0..3], and the uncertainty of every row's updated token
 *   into the workspace; score, seed_idx and n_seeds are not written (they may
 *   be NULL). Then cover_attn_mass_fwd produces d_in / d_out from the updated
 *   state, and cover_seed_select_fwd runs steps 3-5 on the same workspace. This
 *   is the order of Section 5.3, where d_in sums over the masked positions after
 *   the update and d_out over the positions drafted in this step.
 * Errors: COVER_ERR_INVALID_ARG for a NULL required pointer, N, V or n_seq < 1,
 * N % n_seq != 0, N / n_seq > 4096, draft_budget, remask_budget or max_seeds
 * < 0, an unknown phase, or a misaligned pointer. COVER_ERR_CUDA for a launch
 * failure.
 */
#define COVER_FLAG_SEED 1
#define COVER_FLAG_DRAFTED 2
#define COVER_DECIDE_ALL 0
#define COVER_DECIDE_UPDATE 1
size_t cover_decide_workspace_bytes(int N, int n_seq);
int cover_score_decide_fwd(const void* logits, int N, int V, int n_seq,
                           const float* d_in, const float* d_out, const uint8_t* draft_ok,
                           float tau_draft, int draft_budget, int remask_budget, int mask_id,
                           int min_one, int pos0, int max_seeds, int phase,
                           int32_t* tok, uint8_t* flags, uint8_t* remask_cnt,
                           float* maxprob, float* entropy, int32_t* argmax, float* score,
                           int32_t* seed_idx, int32_t* n_seeds, int32_t* stats,
                           void* workspace, void* stream);

/*
 * d_in and d_out of the seed score (Section 5.3) from the attention of the
 * current pass, averaged over the Hq heads: for the response positions
 * pos0 .. pos0 + per - 1 of every batch row (state row b * per + i is
 * position pos0 + i),
 *   d_in(j)  = sum over masked positions q (tok == mask_id) of A[q -> j],
 *   d_out(j) = sum over positions i with flag bit COVER_FLAG_DRAFTED of A[j -> i],
 * where A_h[q -> j] = exp(q_q . k'_j / sqrt(D) - lse_h(q)) and a seed query's
 * diagonal uses its masked-input key (the leave-one-out view; lse is the one
 * cover_attn_fwd wrote, that of the corrected distribution). Only response
 * queries and response keys contribute. Tensor-core recomputation of the
 * per x per block of every head (once per orientation, so that both sums are
 * row sums); partial sums per head are added in a fixed order, so the result
 * is deterministic.
 * q [B, Hq, L, 128], k_cached [B, Hkv, L, 128], k_seedmask [B, Hkv, n_seeds,
 * 128] bf16; seed_idx int32 [B, n_seeds]; lse float [B, Hq, L]; tok int32,
 * flags uint8 [B * per] (cover_score_decide_fwd's state after the update
 * phase); d_in, d_out float [B * per] (out). workspace:
 * cover_attn_mass_workspace_bytes(B, Hq, per) bytes, 16-byte aligned, no
 * initialisation needed. All device pointers, owned by the caller.
 * Errors: COVER_ERR_INVALID_ARG for a NULL required pointer, B, Hq, Hkv, L,
 * per < 1, Hq % Hkv != 0, pos0 < 0 or pos0 + per > L, n_seeds < 0 or > L, or a
 * misaligned pointer; COVER_ERR_UNSUPPORTED for D != 128 or per > 16384 (the
 * per-column data of a response block is staged in shared memory);
 * COVER_ERR_CUDA for a launch failure; COVER_ERR_DEVICE_TIMEOUT via
 * cover_device_status.
 */
size_t cover_attn_mass_workspace_bytes(int B, int Hq, int per);
int cover_attn_mass_fwd(const void* q, const void* k_cached, const void* k_seedmask,
                        const int32_t* seed_idx, int n_seeds, const float* lse,
                        int B, int Hq, int Hkv, int L, int D,
                        const int32_t* tok, const uint8_t* flags, int mask_id, int pos0, int per,
                        void* workspace, float* d_in, float* d_out, void* stream);

/*
 * Steps 3-5 of cover_score_decide_fwd (seed score, adaptive revision rate,
 * selection) after a COVER_DECIDE_UPDATE call on the same workspace and state:
 * score = u * (1 + d_in) / (1 + d_out) with u of the updated token; clears flag
 * bits COVER_FLAG_SEED and COVER_FLAG_DRAFTED, then sets COVER_FLAG_SEED on the
 * new seeds; writes score [N], seed_idx [n_seq, max_seeds], n_seeds [n_seq] and
 * stats[.., 4..5]. Arguments and errors as cover_score_decide_fwd.
 */
int cover_seed_select_fwd(int N, int n_seq, const float* d_in, const float* d_out,
                          int remask_budget, int mask_id, int pos0, int max_seeds,
                          int32_t* tok, uint8_t* flags, uint8_t* remask_cnt, float* score,
                          int32_t* seed_idx, int32_t* n_seeds, int32_t* stats,
                          void* workspace, void* stream);

/*
 * Synchronises `stream`, then returns and clears the current device's status
 * word: COVER_OK, or COVER_ERR_DEVICE_TIMEOUT if a kernel gave up on a
 * bounded wait since the last call. Returns COVER_ERR_CUDA if the
 * synchronisation itself fails.
 */
int cover_device_status(void* stream);

/* Static, human-readable name of a status code. Never NULL. */
const char* cover_status_str(int code);

#ifdef __cplusplus
}
#endif

#endif /* COVER_H_ */
