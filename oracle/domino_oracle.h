/*
 * domino_oracle.h -- plain fp64 CPU oracle of the Domino draft-side block step.
 *
 * TEST INFRASTRUCTURE ONLY.  This library exists to check the CUDA path; it is
 * called from the tests, from the package smoke check and from the CPU-baseline
 * leg and the reference arm of the benchmark, never from the product path.  It shares no code, header,
 * table or helper with the CUDA library (include/domino.h) and includes nothing
 * from it.
 *
 * Conventions
 *   - bf16 tensors are passed as raw uint16_t bit patterns and widened exactly to
 *     double; every intermediate is double; nothing is rounded in between.
 *   - Row-major everywhere; a weight [rows, cols] has element (r, c) at r*cols + c.
 *   - A NULL bias means a zero bias.
 *   - Return codes: 0 ok, ORACLE_ERR_ARG (-1) for bad sizes or pointers,
 *     ORACLE_ERR_TOKEN (-2) for a prefix id outside [0, V).
 *
 * Notation follows the paper (Domino, arXiv 2605.29707): B sequences, K draft
 * positions, hidden size H, vocabulary V, GRU state size Ds (d_s), correction
 * rank R (r), top-k width k, N tree nodes per sequence.
 */
#ifndef DOMINO_ORACLE_H
#define DOMINO_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ORACLE_ERR_ARG (-1)
#define ORACLE_ERR_TOKEN (-2)

/* Exact bf16 -> double widening. */
double oracle_bf16_to_double(uint16_t b);

/* O1, section 4.1.2 "Causal Encoder": E_j is the token embedding of prefix id j.
 * emb: bf16 [V, H]; ids: [n]; E: double [n, H]. */
int oracle_embed(const uint16_t* emb, int V, int H, const int32_t* ids, int n, double* E);

/* O2, section 4.1.2 causal-encoder equation S_{i-1} = GRU(E_{<=i-1}).
 * GRU with torch.nn.GRU gate conventions (gate blocks r | z | n):
 *   r = sigmoid(W_ir x + b_ir + W_hr h + b_hr)
 *   z = sigmoid(W_iz x + b_iz + W_hz h + b_hz)
 *   n = tanh(W_in x + b_in + r * (W_hn h + b_hn))
 *   h' = (1 - z) * n + z * h,  starting from h = 0.
 * E: double [K, Hin]; w_ih bf16 [3Ds, Hin]; w_hh bf16 [3Ds, Ds]; b_ih, b_hh bf16 [3Ds] or NULL.
 * S: double [K, Ds], S[j] = state after absorbing E_0..E_j. */
int oracle_gru(const double* E, int K, int Hin, int Ds, const uint16_t* w_ih, const uint16_t* w_hh,
               const uint16_t* b_ih, const uint16_t* b_hh, double* S);

/* O3, section 4.1.2 low-rank correction equation: u_j = SiLU(W1 [hidden_j ; S_j] + b1).
 * hidden: double [K, H]; S: double [K, Ds]; w1 bf16 [R, H + Ds] (columns 0..H-1 multiply
 * hidden, H..H+Ds-1 multiply S); b1 bf16 [R] or NULL.  u: double [K, R]. */
int oracle_lowrank(const double* hidden, const double* S, int K, int H, int Ds, int R,
                   const uint16_t* w1, const uint16_t* b1, double* u);

/* O4, section 4.1.1 base-logit equation plus section 4.1.2 residual:
 *   z_j[v] = W_lm[v] . hidden_j + W2[v] . u_j + b2[v].
 * hidden: double [K, H]; u: double [K, R] (ignored when R == 0); w_lm bf16 [V, H];
 * w2 bf16 [V, R] or NULL (no correction); b2 bf16 [V] or NULL.  z: double [K, V].
 * nthreads > 1 splits the (row, vocab) grid across OpenMP threads. */
int oracle_logits(const double* hidden, const double* u, int K, int H, int V, int R,
                  const uint16_t* w_lm, const uint16_t* w2, const uint16_t* b2, double* z,
                  int nthreads);

/* O5: log-softmax of each row: lse = m + log(sum_v exp(z - m)), logp = z - lse. */
int oracle_log_softmax(const double* z, int n, int V, double* logp, double* lse);

/* O6: the k best entries of each row ordered by (value descending, id ascending). */
int oracle_topk(const double* logp, int n, int V, int k, int32_t* ids, double* vals);

/* O7, draft tree: best-first selection of N nodes.  The frontier starts with the k
 * depth-1 candidates of position 0; each pop takes the candidate with the greatest
 * (score, then lower token id, then lower parent index); a popped node of depth d < K
 * pushes its k children from position d's top-k list with score = parent score + logp.
 * topk_ids / topk_logp: [K, k].  Outputs [N]: parent (-1 for the root/anchor), token,
 * depth (1..K), score (cumulative log-probability). */
int oracle_tree(const int32_t* topk_ids, const double* topk_logp, int K, int k, int N,
                int32_t* parent, int32_t* token, int32_t* depth, double* score);

/* The whole step for the sequences listed in seqs (nseq of them; seqs == NULL means
 * all B in order).  Output arrays are indexed by the position in that list.
 *   hidden bf16 [B, K, H], prefix_ids [B, K], w_lm bf16 [V, H], emb bf16 [V, H],
 *   w_ih [3Ds, H], w_hh [3Ds, Ds], b_ih/b_hh [3Ds] or NULL, w1 [R, H+Ds], b1 [R] or NULL,
 *   w2 [V, R] or NULL, b2 [V] or NULL.
 * Outputs: logp_full [nseq, K, V] or NULL, lse [nseq, K] or NULL,
 *   topk_ids/topk_logp [nseq, K, k], tree_* [nseq, N]. */
int oracle_draft_step(const uint16_t* hidden, const int32_t* prefix_ids, const uint16_t* w_lm,
                      const uint16_t* emb, const uint16_t* w_ih, const uint16_t* w_hh,
                      const uint16_t* b_ih, const uint16_t* b_hh, const uint16_t* w1,
                      const uint16_t* b1, const uint16_t* w2, const uint16_t* b2, int B, int K,
                      int H, int V, int Ds, int R, int k, int N, const int32_t* seqs, int nseq,
                      double* logp_full, double* lse, int32_t* topk_ids, double* topk_logp,
                      int32_t* tree_parent, int32_t* tree_token, int32_t* tree_depth,
                      double* tree_score, int nthreads);

/* O8, the step after the draft (section 3.1: one target pass checks the whole draft, the draft
 * tokens are kept up to the first one the target rejects, and tau counts the kept tokens plus
 * the one extra token the target itself contributes).  Greedy verification of one draft tree at temperature 0, where a draft
 * token is valid when it equals the target's most likely next token:
 *   parent/token [N]: the tree (parent -1 = the anchor, otherwise an earlier node), as from
 *     oracle_tree; target [N+1, V] fp32: the target's next-token logits after the anchor
 *     (row 0) and after each node i (row i+1).
 *   Walk from the anchor: a = the argmax of the current node's row (equal values: the lowest
 *   id); if a child of the current node carries token a (several: the lowest node index),
 *   accept it and continue from it; otherwise stop.
 * Outputs: row_argmax [N+1]; nodes [N] = the accepted nodes in order, -1 after the last;
 *   n_acc = their number; bonus = the last argmax (the target's own next token). tau =
 *   n_acc + 1.  The comparisons are on the given fp32 values, exactly. */
int oracle_verify_greedy(const float* target, int N, int V, const int32_t* parent, const int32_t* token,
                         int32_t* row_argmax, int32_t* nodes, int32_t* n_acc, int32_t* bonus);

/* The walk of oracle_verify_greedy for any per-row choice: row_choice [N+1] = the target's token
 * after the anchor (row 0) and after each node i (row i+1); same outputs and tree checks. */
int oracle_tree_walk(int N, const int32_t* parent, const int32_t* token, const int32_t* row_choice,
                     int32_t* nodes, int32_t* n_acc, int32_t* bonus);

/* O11: one draw from softmax(row / T) (temperature T > 0) with the caller's uniform u in [0, 1):
 * the first id whose cumulative probability in id order exceeds u; at or past the total
 * (rounding) the last id of non-zero mass; a row without a finite value gives id 0. */
int oracle_row_sample(const float* row, int V, double T, double u, int32_t* id);

/* O12, verification at temperature T > 0 (section 3.1: the target keeps draft tokens by the
 * speculative sampling rule, so that what it emits is distributed as its own samples).  Reading:
 * the tree's children are fixed proposals (chosen best-first, not drawn), a point mass per
 * child.  Against a point mass at x the rule accepts x with probability p(x) and otherwise draws
 * from p with x removed, renormalised; applied child after child (recursive rejection) that is
 * the same as drawing one token y from p and moving to the child that carries y, or emitting y
 * when no child does.  So, per tree: row_sample[r] = oracle_row_sample(row r, T, uniforms[r]),
 * then oracle_tree_walk on those draws; uniforms [N+1] in [0, 1).  Lossless: the emitted tokens
 * follow the target's own distribution whatever the tree. */
int oracle_verify_sample(const float* target, int N, int V, double T, const float* uniforms,
                         const int32_t* parent, const int32_t* token, int32_t* row_sample, int32_t* nodes,
                         int32_t* n_acc, int32_t* bonus);

/* O9, the sequential draft loop at inference (section 4.1.2 and Fig. 3: each draft token is
 * chosen from the final logits and is the causal encoder's next input), greedy: per sequence,
 * t_0 = anchors[b]; for j = 0..K-1: S_j = the GRU state after E_0..E_j with E_i = emb[t_i];
 * u_j = SiLU(W1 [hidden_j ; S_j] + b1); L_j = W_lm hidden_j + W2 u_j + b2; t_{j+1} = argmax L_j
 * (equal values: the lowest id); logp_j = log-softmax(L_j)[t_{j+1}].  With the correction branch
 * off (w2 NULL or R = 0) L_j = W_lm hidden_j + b2.
 * Outputs for the sequences in seqs (as in oracle_draft_step): tokens [nseq, K] = t_1..t_K,
 * logp [nseq, K]. */
int oracle_rollout_greedy(const uint16_t* hidden, const int32_t* anchors, const uint16_t* w_lm,
                          const uint16_t* emb, const uint16_t* w_ih, const uint16_t* w_hh,
                          const uint16_t* b_ih, const uint16_t* b_hh, const uint16_t* w1,
                          const uint16_t* b1, const uint16_t* w2, const uint16_t* b2, int B, int K,
                          int H, int V, int Ds, int R, const int32_t* seqs, int nseq, int32_t* tokens,
                          double* logp, int nthreads);

/* O10, the same loop with each token sampled from the final distribution (section 4.1.2 and
 * Fig. 3: every draft token is drawn from the refined logits l_i + c_i): with u_j = uniforms[b * K + j] in [0, 1)
 * (the caller's random draws), t_{j+1} = the first id v whose cumulative probability
 * sum_{v' <= v} softmax(L_j)[v'] (in id order) exceeds u_j; a u_j at or past the rounded total
 * takes the last id of non-zero probability.  logp_j = log-softmax(L_j)[t_{j+1}].  Returns
 * ORACLE_ERR_ARG for a uniform outside [0, 1). */
int oracle_rollout_sample(const uint16_t* hidden, const int32_t* anchors, const float* uniforms,
                          const uint16_t* w_lm, const uint16_t* emb, const uint16_t* w_ih,
                          const uint16_t* w_hh, const uint16_t* b_ih, const uint16_t* b_hh,
                          const uint16_t* w1, const uint16_t* b1, const uint16_t* w2, const uint16_t* b2,
                          int B, int K, int H, int V, int Ds, int R, const int32_t* seqs, int nseq,
                          int32_t* tokens, double* logp, int nthreads);

/* O13, the counter-based generator of the exponential-race sampler: Philox-4x32 with ten
 * rounds, as published by Salmon, Moraes, Dror and Shaw ("Parallel random numbers: as easy as
 * 1, 2, 3", SC 2011): ctr (4 words) and key (2 words) in, 4 words out. */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]);

/* O14, the perturbation of vocabulary entry v at step j of sequence b under a 64-bit seed:
 * x = word (b mod 4) of Philox-4x32-10 with counter (v, j, floor(b / 4), 0) and key (seed mod
 * 2^32, floor(seed / 2^32)); u = (floor(x / 512) + 1/2) / 2^23, which lies in [2^-24, 1 - 2^-24];
 * g = -log(-log(u)), a standard Gumbel draw.  Fills g[0 .. V-1] for v = 0 .. V-1. */
int oracle_gumbel_row(uint64_t seed, int b, int j, int V, double* g);

/* O15, the same loop as O10 with each token sampled by the exponential race (Gumbel-max): with
 * g_j[v] the perturbation O14 of (seed, b, j, v), t_{j+1} = argmax_v (L_j[v] + g_j[v]) (equal
 * values: the lowest id), a draw from softmax(L_j); logp_j = log-softmax(L_j)[t_{j+1}].
 * Otherwise as oracle_rollout_greedy. */
int oracle_rollout_sample_gumbel(const uint16_t* hidden, const int32_t* anchors, uint64_t seed,
                                 const uint16_t* w_lm, const uint16_t* emb, const uint16_t* w_ih,
                                 const uint16_t* w_hh, const uint16_t* b_ih, const uint16_t* b_hh,
                                 const uint16_t* w1, const uint16_t* b1, const uint16_t* w2, const uint16_t* b2,
                                 int B, int K, int H, int V, int Ds, int R, const int32_t* seqs, int nseq,
                                 int32_t* tokens, double* logp, int nthreads);

/* Number of OpenMP threads the oracle would use for nthreads <= 0 (all available). */
int oracle_max_threads(void);

#ifdef __cplusplus
}
#endif
#endif
