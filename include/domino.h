/*
 * domino.h -- C ABI of the GB300 (sm_103a) Domino draft-side block step.
 *
 * Method: Domino (arXiv 2605.29707).  Given the parallel draft backbone's hidden states for
 * a K-position draft block and the block's prefix tokens, one call computes, for every
 * sequence b and draft position j:
 *   base logits          L_base = W_lm . hidden[b, j]                 (section 4.1.1, LM-head eq.)
 *   causal state         S_j = GRU(E_0 .. E_j), E_i = emb[prefix_ids[b, i]], h starts at 0
 *                                                                      (section 4.1.2, encoder eq.)
 *   low-rank correction  dL = W2 . SiLU(W1 [hidden[b, j]; S_j] + b1) + b2
 *                                                                      (section 4.1.2, correction eq.)
 *   final logits         L = L_base + dL                               (section 4.1.2, residual)
 *   log-softmax of L, its k best tokens (value descending, then token id ascending), and
 *   the draft tree: the N nodes of highest cumulative log-probability below the anchor,
 *   chosen best-first with ties to the lower token id and then the lower parent index; a
 *   node at depth d takes its token from position d-1's top-k list ("Tree" cost, Fig. 1).
 * prefix_ids[b, 0] is the anchor (last verified token); prefix_ids[b, j >= 1] is the token
 * drafted for position j-1.  Full logits never reach memory.
 *
 * Conventions for every entry point
 *   - All tensors are row-major and contiguous.  bf16 tensors are raw IEEE bfloat16.
 *   - Device pointers are owned by the caller; the library never allocates, frees or keeps
 *     them.  Work is enqueued on `stream` (a cudaStream_t passed as void*; NULL = legacy
 *     default stream).  domino_draft_step does not synchronise.
 *   - Synchronous argument checks return a negative DOMINO_ERR_* code before anything is
 *     enqueued.  Errors found on the device (a prefix id outside [0, V), a device-side wait
 *     that ran out) are written to a status word inside the workspace and read back by
 *     domino_check_status; the device never traps or asserts.
 *   - The library runs on sm_103 devices only (GB300); elsewhere it returns
 *     DOMINO_ERR_UNSUPPORTED.
 */
#ifndef DOMINO_H
#define DOMINO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define DOMINO_ABI_VERSION 2

#if defined(__GNUC__)
#define DOMINO_API __attribute__((visibility("default")))
#else
#define DOMINO_API
#endif

enum domino_status {
  DOMINO_OK = 0,
  DOMINO_ERR_INVALID_ARG = -1, /* NULL required pointer, size <= 0, k > V, N > sum_{d=1..K} k^d,
                                  workspace too small */
  DOMINO_ERR_UNSUPPORTED = -2, /* outside the supported envelope: H, Ds or R not a multiple of 8,
                                  a tensor pointer not 16-byte aligned, k > 32, N > 256, K > 64,
                                  Ds > 2048, V >= 2^22, or not an sm_103 device */
  DOMINO_ERR_CUDA = -3,        /* a CUDA runtime call or kernel launch failed */
  DOMINO_ERR_TIMEOUT = -4,     /* device: a bounded wait (pipeline barrier, grid barrier) ran out */
  DOMINO_ERR_BAD_TOKEN = -5    /* device: a prefix id outside [0, V) */
};

/* The Domino head's weights (section 4.1.2), all device pointers to bf16.
 * GRU: torch.nn.GRU layout, gate blocks r | z | n:
 *   w_ih [3*Ds, H], w_hh [3*Ds, Ds], b_ih [3*Ds] or NULL, b_hh [3*Ds] or NULL.
 *   r = sigmoid(W_ir x + b_ir + W_hr h + b_hr); z = sigmoid(W_iz x + b_iz + W_hz h + b_hz);
 *   n = tanh(W_in x + b_in + r * (W_hn h + b_hn)); h' = (1 - z) * n + z * h.
 * emb [V, H]: the target's token embedding table feeding the GRU (may alias w_lm when the
 *   target ties them); only the rows named by prefix_ids are read.
 * w1 [R, H + Ds]: columns 0..H-1 multiply hidden, columns H..H+Ds-1 multiply S; b1 [R] or NULL.
 * w2 [V, R]; b2 [V] or NULL.
 * Ds = d_s (1024 in the paper), R = r (256 in the paper).  R == 0 or w2 == NULL turns the
 * correction branch off: the step then returns log softmax(W_lm . hidden + b2), the base
 * distribution of the paper's Table 4 "w/o Domino head" (b2 still applies when given), and
 * emb / w_ih / w_hh / w1 / b1 are not read. */
typedef struct domino_head_weights {
  const void* emb;
  const void* w_ih;
  const void* w_hh;
  const void* b_ih;
  const void* b_hh;
  const void* w1;
  const void* b1;
  const void* w2;
  const void* b2;
  int Ds;
  int R;
  /* Optional fp32 [V, 3*Ds] input-projection table, table[t] = W_ih . emb[t] (no bias), made
   * once per set of weights by domino_build_input_table; NULL = the GRU projects emb[t]
   * itself.  When set, every entry point takes the GRU's input-gate sums from it (one row per
   * token) instead of projecting the embedding rows: the block step then launches no X GEMM
   * (domino_launches_per_step_table) and the rollout's steps read one row each.  16-byte
   * aligned, like every tensor (refused as the other pointers are). */
  const float* x_table;
} domino_head_weights;

/* Bytes of the input-projection table (V * 3 * Ds fp32 values); 0 for invalid sizes. */
DOMINO_API size_t domino_input_table_bytes(int V, int Ds);

/* table[t][g] = sum_h emb[t][h] * w_ih[g][h] for every token t < V and gate row g < 3*Ds: the
 * GRU's input projection (section 4.1.2, encoder eq.; b_ih is not included) of every token,
 * computed once on the tensor cores (fp32 accumulation).  emb bf16 [V, H], w_ih bf16 [3*Ds, H],
 * table fp32 [V, 3*Ds] (domino_input_table_bytes), all device pointers, 16-byte aligned; H and
 * Ds multiples of 8.  The table depends on emb and w_ih only: rebuild it when they change.
 * Synchronises the stream; returns DOMINO_OK, DOMINO_ERR_INVALID_ARG / _UNSUPPORTED (nothing
 * enqueued), DOMINO_ERR_CUDA or DOMINO_ERR_TIMEOUT (a device-side wait ran out: the table is
 * not valid). */
DOMINO_API int domino_build_input_table(const void* emb, const void* w_ih, int V, int H, int Ds, float* table,
                                        void* stream);

/* Bytes of device workspace domino_draft_step needs for these sizes on the current device
 * (the split of the work depends on the device's SM count).  Returns 0 when the sizes are
 * invalid or unsupported.  R = 0 (or a head without w2) sizes the correction-off step. */
DOMINO_API size_t domino_workspace_bytes(int B, int K, int H, int V, int Ds, int R, int k, int N);

/* One draft-side block step.
 *   hidden      bf16 [B, K, H]   backbone hidden states of the K draft positions
 *   prefix_ids  int32 [B, K]     anchor then drafted tokens (see above)
 *   w_lm        bf16 [V, H]      frozen target LM head (nn.Linear layout)
 *   head        Domino head weights (host struct holding device pointers); NULL = head off
 *   k           top-k width, 1 <= k <= min(32, V)
 *   N           tree nodes per sequence, 1 <= N <= min(256, sum_{d=1..K} k^d)
 * Outputs (device):
 *   topk_ids    int32 [B, K, k]  per position, log-prob descending, ties to the lower id
 *   topk_logp   fp32  [B, K, k]  refined log-probabilities log softmax(L)[id]
 *   tree_parent int32 [B, N]     parent node index, -1 for a child of the anchor; parent < i
 *   tree_token  int32 [B, N]
 *   tree_depth  int32 [B, N]     1..K
 *   tree_score  fp32  [B, N] or NULL   cumulative log-probability, non-increasing in i
 * workspace: device buffer of at least domino_workspace_bytes(...) bytes, 256-byte aligned,
 * ZERO-FILLED before its first use (once, e.g. cudaMemsetAsync at allocation); every step
 * leaves it ready for the next one, whatever the sizes or the kind of the step before.  Small
 * batches skip a per-step clear: the GRU's state words carry a step count the last kernel
 * advances, and are trusted only over the byte range the control words record as holding state
 * words; when a step of another shape or kind used the workspace last, the GRU first zeroes its
 * own state words behind a grid barrier.  A call that fails part-way with DOMINO_ERR_CUDA zeroes
 * the control words itself; if the CUDA context is broken, zero the whole workspace before
 * reusing it.  One workspace must not be shared by steps that overlap in time.
 * Returns DOMINO_OK once everything is enqueued, or a negative code (nothing enqueued). */
DOMINO_API int domino_draft_step(const void* hidden, const int32_t* prefix_ids, const void* w_lm,
                      const domino_head_weights* head, int B, int K, int H, int V, int k, int N,
                      int32_t* topk_ids, float* topk_logp, int32_t* tree_parent,
                      int32_t* tree_token, int32_t* tree_depth, float* tree_score,
                      void* workspace, size_t workspace_bytes, void* stream);

/* The same step with the per-step inputs and the outputs in HOST memory (pinned memory
 * recommended for the inputs) and the weights on the device.  hidden / prefix_ids are copied
 * into the workspace, the step runs, and every output plus the device status come back in one
 * copy into a pinned staging buffer the library allocates on first use and keeps for the
 * process (calls from several threads take turns on it), from which they are copied to the
 * caller's buffers; the call synchronises the stream before returning.  The workspace must
 * hold domino_workspace_bytes_host(...) bytes and be zero-filled before its first use, as for
 * domino_draft_step.  From the second call with the same arguments (pointers and sizes) on, the
 * library replays a CUDA graph of the whole call that it captured on a stream of its own
 * (launched on `stream`), so that the step's launches need not reach the GPU one by one after
 * the previous call returned; the inputs are read afresh on every call.  Calls it cannot
 * capture (pageable inputs, for instance) run directly.  The graphs hold no device memory of
 * their own; at most 16 are kept.  Returns DOMINO_OK or the first error,
 * including device-side errors (bad prefix id, timeout). */
DOMINO_API size_t domino_workspace_bytes_host(int B, int K, int H, int V, int Ds, int R, int k, int N);
DOMINO_API int domino_draft_step_host(const void* hidden_host, const int32_t* prefix_ids_host,
                           const void* w_lm, const domino_head_weights* head, int B, int K,
                           int H, int V, int k, int N, int32_t* topk_ids_host,
                           float* topk_logp_host, int32_t* tree_parent_host,
                           int32_t* tree_token_host, int32_t* tree_depth_host,
                           float* tree_score_host, void* workspace, size_t workspace_bytes,
                           void* stream);

/* Synchronises `stream` and returns the device status word of the last step that used
 * `workspace`: DOMINO_OK, DOMINO_ERR_BAD_TOKEN or DOMINO_ERR_TIMEOUT (DOMINO_ERR_CUDA if the
 * read itself fails).  Each domino_draft_step clears the word when it starts. */
DOMINO_API int domino_check_status(const void* workspace, void* stream);

/* Failure-detection test hook; the paper has no counterpart.  It lets a test check that a
 * step whose inter-CTA wait can never be satisfied reports DOMINO_ERR_TIMEOUT instead of
 * hanging, without faulting anything.  It arms, on the current device, one withheld event in
 * the next GRU launch that has a CTA numbered gru_cta; the launch's other CTAs wait for that
 * event, their bounded waits run out (about one second of SM clock cycles each), and the step
 * records DOMINO_ERR_TIMEOUT in its device status word (domino_check_status):
 *   DOMINO_HOLD_STATE          CTA gru_cta does not publish its hidden states of position
 *                              `step` (0 <= step < 64; a step >= K withholds nothing);
 *   DOMINO_HOLD_CLEAR_BARRIER  CTA gru_cta does not arrive at the barrier of the state clear
 *                              that a small-batch step (B <= 2 at K = 16) runs when the workspace
 *                              last held another kind or shape of step (or is fresh); `step` is
 *                              ignored, and a step that needs no clear withholds nothing;
 *   DOMINO_HOLD_OFF            disarms the hook.
 * The held CTA disarms the hook when its launch ends, so it affects one step.  Every kernel of
 * the held step still completes (its outputs are undefined) and the workspace stays usable: the
 * next step runs normally.  Synchronous (a copy to a device symbol); not for use while steps
 * run on other threads.  Returns DOMINO_OK, DOMINO_ERR_INVALID_ARG or DOMINO_ERR_CUDA. */
enum domino_hold { DOMINO_HOLD_OFF = 0, DOMINO_HOLD_STATE = 1, DOMINO_HOLD_CLEAR_BARRIER = 2 };
DOMINO_API int domino_debug_hold(int what, int gru_cta, int step);

/* Static, human-readable name of a status code. */
DOMINO_API const char* domino_status_string(int status);

/* DOMINO_ABI_VERSION of the loaded library. */
DOMINO_API int domino_abi_version(void);

/* Number of kernel launches one domino_draft_step makes for these sizes (head on when
 * R > 0), so a caller can count device work: the plan of the current device (of a 152-SM GB300
 * when no device is visible).  3 with the head off, 3 for small batches whose GRU computes its
 * own projections (B <= 2 at K = 16), 6 for other batches of at most 128 positions, 7 above;
 * a negative code for sizes domino_draft_step would reject. */
DOMINO_API int domino_launches_per_step(int B, int K, int H, int V, int Ds, int R, int k, int N);
/* The same count for a head that carries an input-projection table (head->x_table): one launch
 * fewer wherever domino_launches_per_step counts an X GEMM (5 instead of 6, 6 instead of 7). */
DOMINO_API int domino_launches_per_step_table(int B, int K, int H, int V, int Ds, int R, int k, int N);

/* Greedy verification of draft trees against the target model's logits: the step after the
 * draft.  Section 3.1: one target pass checks the whole draft, the draft tokens are kept up to the
 * first one the target rejects, and tau counts them plus the one extra token the target adds.  At
 * temperature 0 a draft token is valid when it equals the target's most likely next token.
 * For each sequence b, from the anchor: a = argmax of the current node's row (equal values: the
 * lowest id); if a child of the current node carries token a (several: the lowest node index),
 * accept it and continue from it; otherwise stop, and a is the bonus token.
 *   target_logits: device fp32 [B, N + 1, V]: the target's next-token logits after the anchor
 *     (row 0) and after tree node i (row i + 1).  Finite values (NaN is not ordered).
 *   tree_parent / tree_token: device int32 [B, N] as domino_draft_step writes them (parent -1 =
 *     the anchor, otherwise an earlier node); may be NULL when N = 0.
 * Outputs (device int32): row_argmax [B, N + 1]; accepted_nodes [B, N] = the accepted nodes in
 *   order, -1 after the last; accepted_count [B] (tau = accepted_count + 1); bonus_token [B].
 * Two kernels on `stream`; no workspace.  Returns DOMINO_OK once enqueued, or a negative code
 * (bad sizes or pointers) with nothing enqueued. */
DOMINO_API int domino_verify_tree_greedy(const float* target_logits, const int32_t* tree_parent,
                                         const int32_t* tree_token, int B, int N, int V, int32_t* row_argmax,
                                         int32_t* accepted_nodes, int32_t* accepted_count,
                                         int32_t* bonus_token, void* stream);

/* Verification of draft trees at temperature T > 0 (section 3.1: the target keeps draft tokens by
 * the speculative sampling rule, which leaves what it emits distributed as its own samples).
 * The tree's children are fixed proposals (chosen best-first, not drawn): against a proposal x
 * that is certain, the rule keeps x with probability p(x) and otherwise draws from p without x,
 * renormalised; tried child after child, that is one draw y from the target's p at the node,
 * kept when a child carries y.  So, for each sequence b, from the anchor: y = the draw of the
 * current node's row; if a child of the current node carries y (several: the lowest node index),
 * accept it and continue from it; otherwise stop, and y is the bonus token.
 *   The draw of row r: p = softmax(target_logits[r] / T); y = the first id v whose cumulative
 *   probability sum_{v' <= v} p(v'), in id order, exceeds u = uniforms[r] (values outside [0, 1)
 *   are clamped to it), computed in fp32: where u falls within rounding of a boundary either
 *   neighbour may be drawn, and past the computed total the last id of non-zero probability is.
 *   Ids of zero probability (logit -inf) are never drawn; a row with no finite logit gives id 0.
 *   target_logits: device fp32 [B, N + 1, V] as for domino_verify_tree_greedy; finite or -inf
 *     (NaN is not ordered).  V <= 8 * 53248 (a row is staged in shared memory once).
 *   uniforms: device fp32 [B, N + 1], the caller's random draws, one per row (only the rows the
 *     walk visits matter).
 *   temperature: T > 0 with 1 / T finite in fp32.
 *   tree_parent / tree_token: as for domino_verify_tree_greedy.
 * Outputs (device int32): row_sample [B, N + 1] = every row's draw; accepted_nodes [B, N],
 *   accepted_count [B] (tau = accepted_count + 1) and bonus_token [B] as for
 *   domino_verify_tree_greedy.
 * Two kernels on `stream`; no workspace.  Returns DOMINO_OK once enqueued, DOMINO_ERR_UNSUPPORTED
 * for a larger V, or another negative code (bad sizes, pointers or temperature) with nothing
 * enqueued. */
DOMINO_API int domino_verify_tree_sample(const float* target_logits, const int32_t* tree_parent,
                                         const int32_t* tree_token, const float* uniforms, float temperature,
                                         int B, int N, int V, int32_t* row_sample, int32_t* accepted_nodes,
                                         int32_t* accepted_count, int32_t* bonus_token, void* stream);

/* The greedy sequential draft loop, the paper's inference loop (section 4.1.2 and Fig. 3: each
 * draft token is chosen from the final logits and becomes the causal encoder's next input), as
 * a variant of domino_draft_step for callers that do not have the prefix (V < 2^22, else
 * DOMINO_ERR_UNSUPPORTED):
 *   t_0 = anchors[b]; for j = 0..K-1: S_j = the GRU state after emb[t_0..t_j];
 *   u_j = SiLU(W1 [hidden_j ; S_j] + b1); L_j = W_lm hidden_j + W2 u_j + b2;
 *   t_{j+1} = argmax L_j (equal values: the lowest id); logp_j = log-softmax(L_j)[t_{j+1}].
 * With the correction branch off (head NULL, R = 0 or w2 NULL) L_j = W_lm hidden_j + b2.
 *   hidden [B, K, H] bf16, anchors [B] int32, w_lm [V, H] bf16, head as for domino_draft_step,
 *   all device pointers, 16-byte aligned.  B <= 8 (a latency path; batches use
 *   domino_draft_step); H, d_s and r multiples of 8; r <= 8192.  The step kernel runs one CTA
 *   per SM; a CTA's shared memory (at most 225 KB) holds u of every sequence (4 B r) and its
 *   share of the base logits (4 B ceil(V / SMs) rows), plus, for r <= 256, as many of its W2
 *   rows as fit (its first 512 W2 rows live in the tensor memory, all of it, of the SM for the
 *   whole call; with the input table, B <= 2 and r a multiple of 64, 128-row W2 blocks in tensor
 *   and shared memory instead, for the tensor cores), or,
 *   for r > 256, a 96 KB ring W2 streams through every step (those shares rounded up to whole
 *   ring chunks).  Sizes whose u and base-logit share alone exceed 225 KB return
 *   DOMINO_ERR_INVALID_ARG.
 * Outputs (device): tokens int32 [B, K] = t_1 .. t_K; logp fp32 [B, K].
 * workspace: device memory of domino_rollout_workspace_bytes(...) bytes (16-byte aligned);
 * its first int32 receives the device status (DOMINO_OK, DOMINO_ERR_BAD_TOKEN,
 * DOMINO_ERR_TIMEOUT; domino_check_status reads it).  Two kernels on `stream`: a tensor-core
 * GEMM for W_lm hidden_j of every position, then one cooperative kernel for the K steps (for
 * r <= 256 it first computes W1[:, :H] hidden_j of every position, which does not depend on the
 * recurrence).  With head->x_table set, a step's GRU input-gate sums are row t_j of that table
 * instead of a product with emb[t_j].
 * Returns DOMINO_OK once enqueued, or a negative code with nothing enqueued. */
DOMINO_API size_t domino_rollout_workspace_bytes(int B, int K, int H, int V, int Ds, int R);

/* The same loop with every draft token SAMPLED from the final distribution (section 4.1.2: each
 * draft token is sampled from the final logits; temperature 1): with u = uniforms[b * K + j],
 * the caller's random draws in [0, 1) (device float [B, K]; values outside are clamped to it),
 * t_{j+1} = the first id v whose cumulative probability sum_{v' <= v} softmax(L_j)[v'], in id
 * order, exceeds u (computed in fp32: where u falls within rounding of a boundary either
 * neighbour may be chosen); logp_j = log-softmax(L_j)[t_{j+1}].  Arguments, outputs, workspace
 * (domino_rollout_workspace_bytes) and errors as domino_rollout_greedy; uniforms NULL or not
 * 4-byte aligned: DOMINO_ERR_INVALID_ARG.  The same grid barriers per step as the greedy loop: every
 * CTA reads the final logits of the CTA whose rows hold the draw and scans them itself. */
DOMINO_API int domino_rollout_sample(const void* hidden, const int32_t* anchors, const float* uniforms,
                                     const void* w_lm, const domino_head_weights* head, int B, int K, int H,
                                     int V, int32_t* tokens, float* logp, void* workspace,
                                     size_t workspace_bytes, void* stream);
DOMINO_API int domino_rollout_greedy(const void* hidden, const int32_t* anchors, const void* w_lm,
                                     const domino_head_weights* head, int B, int K, int H, int V,
                                     int32_t* tokens, float* logp, void* workspace, size_t workspace_bytes,
                                     void* stream);

/* The same loop with every draft token SAMPLED from the final distribution (section 4.1.2: each
 * draft token is sampled from the final logits; temperature 1) by the exponential race (Gumbel-
 * max, the rule serving systems sample with): t_{j+1} = argmax_v L_j[v] + g_{b,j}[v], ties to the
 * lowest id, where g_{b,j}[v] = -log(-log(u)) and u comes from Philox-4x32-10 (Salmon, Moraes,
 * Dror and Shaw, SC 2011), key = seed (low word first), counter (v, j, floor(b / 4), 0), word
 * b mod 4, u = (that word's top 23 bits + 1/2) / 2^23.  This draws t_{j+1} from softmax(L_j);
 * logp_j = log-softmax(L_j)[t_{j+1}].  The perturbations are computed in fp32 on the device, so
 * where two perturbed logits lie within rounding of each other either may win.  The draws depend
 * on (seed, b, j, v) alone, so a call with the same seed repeats them: pass a new seed for every
 * block (a running counter will do).  Unlike
 * domino_rollout_sample it needs no per-step scan after the argmax: it costs what the greedy
 * loop costs (one grid barrier per step on the fast path) plus the generator.  Arguments,
 * outputs, workspace (domino_rollout_workspace_bytes) and errors as domino_rollout_greedy. */
DOMINO_API int domino_rollout_sample_gumbel(const void* hidden, const int32_t* anchors, uint64_t seed,
                                            const void* w_lm, const domino_head_weights* head, int B, int K,
                                            int H, int V, int32_t* tokens, float* logp, void* workspace,
                                            size_t workspace_bytes, void* stream);

/* Draft step for callers that cannot allocate device memory.  Some callers cannot call
 * cudaMalloc or any allocator at all: code running inside a host framework that owns every
 * allocation, a plugin loaded into a process whose memory pool is fixed up front, or a
 * real-time caller that must not risk an allocation failing or blocking.  This entry point
 * takes the same inputs and outputs as domino_draft_step but no workspace: its scratch lives
 * in a file-scope static device array of DOMINO_STATIC_SCRATCH_BYTES (16 MiB) inside the
 * library, which every GPU that loads the library holds until the process exits.  The paper
 * has no counterpart to this; it is a deployment convenience.
 *   - The first call on a device looks up that array's device address (cudaGetSymbolAddress,
 *     with that device current); make the first call on each device before any stream capture.
 *   - Sizes whose step needs more scratch than the array (domino_workspace_bytes(...) >
 *     DOMINO_STATIC_SCRATCH_BYTES; e.g. the B = 32 serving batch) return DOMINO_ERR_UNSUPPORTED
 *     before anything is enqueued.
 *   - Every call on a device shares the one array and it keeps the last call's contents; each
 *     call clears the words that must start at zero (status and counters) itself, and a small
 *     batch whose state words overlap what a call of another shape or kind left there zeroes
 *     them first, as for a caller's workspace.  Calls whose work overlaps on the GPU (other
 *     streams, other host threads) race on the array: serialise them.
 *   - No allocation of any kind is made (no cudaMalloc / cudaFree, no library allocator).
 * device_status: optional device int32; after the step it receives the device status word
 * (DOMINO_OK, DOMINO_ERR_BAD_TOKEN or DOMINO_ERR_TIMEOUT) by an asynchronous copy on `stream`.
 * Returns DOMINO_OK once enqueued, or a negative code with nothing enqueued. */
#define DOMINO_STATIC_SCRATCH_BYTES (16u << 20)
DOMINO_API int domino_draft_step_static_scratch(const void* hidden, const int32_t* prefix_ids,
                                                const void* w_lm, const domino_head_weights* head,
                                                int B, int K, int H, int V, int k, int N,
                                                int32_t* topk_ids, float* topk_logp,
                                                int32_t* tree_parent, int32_t* tree_token,
                                                int32_t* tree_depth, float* tree_score,
                                                int32_t* device_status, void* stream);

/* Per-kernel device timing, for the per-component latency breakdown the paper reports in
 * its Fig. 1 (LM head, Domino head, tree).  After domino_timing_begin(max_launches), every
 * kernel the library enqueues (up to max_launches of them, on any stream) is bracketed by a
 * pair of CUDA events.  domino_timing_end() waits for those events, stops recording and writes
 * for each kernel kind (index = DOMINO_KERNEL_*) the summed device time in milliseconds and
 * the number of launches; kinds beyond nkinds are dropped.  Not thread-safe: one recording at
 * a time per process.  Returns DOMINO_OK or DOMINO_ERR_CUDA / DOMINO_ERR_INVALID_ARG. */
enum domino_kernel_kind {
  DOMINO_KERNEL_GATHER = 0,       /* E_j = emb[prefix id], id range check */
  DOMINO_KERNEL_GRU_INPUT = 1,    /* E . W_ih^T on tensor cores (split-K partials) */
  DOMINO_KERNEL_W1_HIDDEN = 2,    /* W1 projection on tensor cores (split-K partials): the hidden
                                     half before the GRU for M <= 128; both halves after it, plus
                                     the SiLU finalize, for larger M */
  DOMINO_KERNEL_GRU = 3,          /* GRU recurrence over K positions (and u = SiLU(...) for
                                     M <= 128) */
  DOMINO_KERNEL_VOCAB = 4,        /* [hidden | u] . [W_lm | W2]^T with online softmax / top-k */
  DOMINO_KERNEL_TREE = 5,         /* merge to log-probs and top-k; best-first tree */
  DOMINO_KERNEL_ROLLOUT_BASE = 6, /* domino_rollout_*: W_lm hidden_j of every position */
  DOMINO_KERNEL_ROLLOUT = 7,      /* domino_rollout_*: the K sequential steps */
  DOMINO_KERNEL_VERIFY = 8,       /* domino_verify_tree_greedy / _sample: row argmax or draw, and
                                     tree walk */
  DOMINO_KERNEL_KINDS = 9
};
DOMINO_API int domino_timing_begin(int max_launches);
DOMINO_API int domino_timing_end(float* total_ms, int* launches, int nkinds);

#ifdef __cplusplus
}
#endif
#endif /* DOMINO_H */
