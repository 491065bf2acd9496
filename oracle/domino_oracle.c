/*
 * domino_oracle.c -- plain, slow, fp64 CPU oracle of the Domino draft-side block step.
 *
 * TEST INFRASTRUCTURE ONLY: used by the tests, the smoke check and the CPU-baseline leg
 * of the benchmark to check the CUDA path.  No product code calls it.  It shares no code
 * with the CUDA library.
 *
 * Every function is the written-out definition of one step, in the paper's order
 * (Domino, arXiv 2605.29707):
 *   section 4.1.1  base logits L_base_i = LMHead(H_i)            -> oracle_logits (W_lm term)
 *   section 4.1.2  E_j token embedding of the preceding tokens   -> oracle_embed
 *                  S_{i-1} = GRU(E_{<=i-1}), d_s = 1024           -> oracle_gru
 *                  dL_i = W2 SiLU(W1 [H_i; S_{i-1}]), r = 256     -> oracle_lowrank + W2 term
 *                  L_i = L_base_i + dL_i                          -> oracle_logits (sum)
 *   Fig. 3 caption: tokens are drawn from the final logits        -> oracle_log_softmax
 *   Fig. 1 caption: the "Tree" construction cost                  -> oracle_topk, oracle_tree
 *   section 3.1, verification of the draft (the step after it)     -> oracle_verify_greedy,
 *                                                                       oracle_verify_sample
 *   section 4.1.2 / Fig. 3, tokens chosen and fed back one by one   -> oracle_rollout_greedy,
 *                                                                       oracle_rollout_sample,
 *                                                                       oracle_rollout_sample_gumbel
 * Readings of points the paper leaves open (GRU gate convention, which ids feed which
 * position, tree tie-breaks) are listed in the design notes; the comments below state the
 * reading each function implements.
 *
 * Floating point: bf16 inputs are widened exactly; all arithmetic is double; dot products
 * are summed in index order.  The only parallelism is an OpenMP split of independent
 * (row, vocab entry) logits in oracle_logits; it does not reorder any sum.
 */
#include "domino_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

double oracle_bf16_to_double(uint16_t b) {
  uint32_t u = ((uint32_t)b) << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static double bf(const uint16_t* p, long i) { return oracle_bf16_to_double(p[i]); }

static double sigmoid(double x) { return 1.0 / (1.0 + exp(-x)); }

static double silu(double x) { return x / (1.0 + exp(-x)); }

int oracle_max_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* O1: E[i] = emb[ids[i]]: the GRU input at a position is the embedding row of the token there
   (section 4.1.2, causal encoder equation). */
int oracle_embed(const uint16_t* emb, int V, int H, const int32_t* ids, int n, double* E) {
  if (!emb || !ids || !E || V <= 0 || H <= 0 || n < 0) return ORACLE_ERR_ARG;
  for (int i = 0; i < n; ++i) {
    if (ids[i] < 0 || ids[i] >= V) return ORACLE_ERR_TOKEN;
    for (int c = 0; c < H; ++c) E[(long)i * H + c] = bf(emb, (long)ids[i] * H + c);
  }
  return 0;
}

/* O2: the GRU recurrence of section 4.1.2 with the torch.nn.GRU gate convention.
 * Reading: the state starts at zero at every block and S[j] is the state after
 * absorbing E_0..E_j, so draft position j sees the anchor and the j tokens drafted
 * before it. */
int oracle_gru(const double* E, int K, int Hin, int Ds, const uint16_t* w_ih, const uint16_t* w_hh,
               const uint16_t* b_ih, const uint16_t* b_hh, double* S) {
  if (!E || !w_ih || !w_hh || !S || K <= 0 || Hin <= 0 || Ds <= 0) return ORACLE_ERR_ARG;
  const int G = 3 * Ds;
  double* h = (double*)calloc((size_t)Ds, sizeof(double));
  double* gi = (double*)malloc((size_t)G * sizeof(double));
  double* gh = (double*)malloc((size_t)G * sizeof(double));
  if (!h || !gi || !gh) {
    free(h); free(gi); free(gh);
    return ORACLE_ERR_ARG;
  }
  for (int j = 0; j < K; ++j) {
    const double* x = E + (long)j * Hin;
    /* the 3Ds gate rows are independent dot products; threads split the rows only */
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (int g = 0; g < G; ++g) {
      double a = b_ih ? bf(b_ih, g) : 0.0;
      for (int c = 0; c < Hin; ++c) a += bf(w_ih, (long)g * Hin + c) * x[c];
      gi[g] = a;
      double b = b_hh ? bf(b_hh, g) : 0.0;
      for (int c = 0; c < Ds; ++c) b += bf(w_hh, (long)g * Ds + c) * h[c];
      gh[g] = b;
    }
    for (int d = 0; d < Ds; ++d) {
      double r = sigmoid(gi[d] + gh[d]);
      double z = sigmoid(gi[Ds + d] + gh[Ds + d]);
      double n = tanh(gi[2 * Ds + d] + r * gh[2 * Ds + d]);
      S[(long)j * Ds + d] = (1.0 - z) * n + z * h[d];
    }
    memcpy(h, S + (long)j * Ds, (size_t)Ds * sizeof(double));
  }
  free(h); free(gi); free(gh);
  return 0;
}

/* O3: u_j = SiLU(W1 [hidden_j ; S_j] + b1) (section 4.1.2, sigma = SiLU, rank r).
 * The concatenation puts hidden first, then the causal state. */
int oracle_lowrank(const double* hidden, const double* S, int K, int H, int Ds, int R,
                   const uint16_t* w1, const uint16_t* b1, double* u) {
  if (!hidden || !S || !w1 || !u || K <= 0 || H <= 0 || Ds <= 0 || R <= 0) return ORACLE_ERR_ARG;
  const long ld = (long)H + Ds;
#ifdef _OPENMP
#pragma omp parallel for collapse(2) schedule(static)
#endif
  for (int j = 0; j < K; ++j) {
    for (int q = 0; q < R; ++q) {
      double a = b1 ? bf(b1, q) : 0.0;
      for (int c = 0; c < H; ++c) a += bf(w1, q * ld + c) * hidden[(long)j * H + c];
      for (int d = 0; d < Ds; ++d) a += bf(w1, q * ld + H + d) * S[(long)j * Ds + d];
      u[(long)j * R + q] = silu(a);
    }
  }
  return 0;
}

/* O4: z_j[v] = W_lm[v] . hidden_j + W2[v] . u_j + b2[v]
 * (section 4.1.1 base logits plus the section 4.1.2 logit-space residual). */
int oracle_logits(const double* hidden, const double* u, int K, int H, int V, int R,
                  const uint16_t* w_lm, const uint16_t* w2, const uint16_t* b2, double* z,
                  int nthreads) {
  if (!hidden || !w_lm || !z || K <= 0 || H <= 0 || V <= 0 || R < 0) return ORACLE_ERR_ARG;
  const int use_head = (w2 != NULL && R > 0);
  if (use_head && !u) return ORACLE_ERR_ARG;
  const long total = (long)K * V;
#ifdef _OPENMP
  int nt = nthreads > 0 ? nthreads : omp_get_max_threads();
#pragma omp parallel for schedule(static) num_threads(nt)
#endif
  for (long e = 0; e < total; ++e) {
    const long j = e / V, v = e % V;
    double a = 0.0;
    for (int c = 0; c < H; ++c) a += bf(w_lm, v * H + c) * hidden[j * H + c];
    if (use_head) {
      double d = 0.0;
      for (int q = 0; q < R; ++q) d += bf(w2, v * R + q) * u[j * R + q];
      a += d;
    }
    if (b2) a += bf(b2, v);
    z[e] = a;
  }
  (void)nthreads;
  return 0;
}

/* O5: per-row log-softmax with the max subtracted before exponentiating. */
int oracle_log_softmax(const double* z, int n, int V, double* logp, double* lse) {
  if (!z || !logp || n < 0 || V <= 0) return ORACLE_ERR_ARG;
  for (int i = 0; i < n; ++i) {
    const double* zi = z + (long)i * V;
    double m = zi[0];
    for (int v = 1; v < V; ++v) m = zi[v] > m ? zi[v] : m;
    double s = 0.0;
    for (int v = 0; v < V; ++v) s += exp(zi[v] - m);
    double l = m + log(s);
    if (lse) lse[i] = l;
    for (int v = 0; v < V; ++v) logp[(long)i * V + v] = zi[v] - l;
  }
  return 0;
}

/* (value, id) ordering: a ranks before b when its value is larger, or equal with a lower id. */
static int ranks_before(double va, int ia, double vb, int ib) {
  return va > vb || (va == vb && ia < ib);
}

/* O6: k passes, each taking the best entry not yet taken under (value desc, id asc). */
int oracle_topk(const double* logp, int n, int V, int k, int32_t* ids, double* vals) {
  if (!logp || !ids || !vals || n < 0 || V <= 0 || k <= 0 || k > V) return ORACLE_ERR_ARG;
  unsigned char* taken = (unsigned char*)malloc((size_t)V);
  if (!taken) return ORACLE_ERR_ARG;
  for (int i = 0; i < n; ++i) {
    const double* row = logp + (long)i * V;
    memset(taken, 0, (size_t)V);
    for (int q = 0; q < k; ++q) {
      int best = -1;
      for (int v = 0; v < V; ++v) {
        if (taken[v]) continue;
        if (best < 0 || ranks_before(row[v], v, row[best], best)) best = v;
      }
      taken[best] = 1;
      ids[(long)i * k + q] = best;
      vals[(long)i * k + q] = row[best];
    }
  }
  free(taken);
  return 0;
}

/* O7: best-first draft tree.  The frontier holds every pushed candidate that has not
 * been popped; each step scans it for the greatest (score, lower token, lower parent). */
int oracle_tree(const int32_t* topk_ids, const double* topk_logp, int K, int k, int N,
                int32_t* parent, int32_t* token, int32_t* depth, double* score) {
  if (!topk_ids || !topk_logp || !parent || !token || !depth || !score) return ORACLE_ERR_ARG;
  if (K <= 0 || k <= 0 || N <= 0) return ORACLE_ERR_ARG;
  /* the tree below the anchor has sum_{d=1..K} k^d nodes; N must not exceed it */
  double cap = 0.0, pw = 1.0;
  for (int d = 1; d <= K; ++d) { pw *= k; cap += pw; }
  if ((double)N > cap) return ORACLE_ERR_ARG;

  const long fcap = (long)k * (N + 1);
  double* f_score = (double*)malloc((size_t)fcap * sizeof(double));
  int32_t* f_tok = (int32_t*)malloc((size_t)fcap * sizeof(int32_t));
  int32_t* f_par = (int32_t*)malloc((size_t)fcap * sizeof(int32_t));
  int32_t* f_dep = (int32_t*)malloc((size_t)fcap * sizeof(int32_t));
  unsigned char* f_live = (unsigned char*)malloc((size_t)fcap);
  if (!f_score || !f_tok || !f_par || !f_dep || !f_live) {
    free(f_score); free(f_tok); free(f_par); free(f_dep); free(f_live);
    return ORACLE_ERR_ARG;
  }
  long nf = 0;
  for (int q = 0; q < k; ++q) { /* depth-1 candidates: children of the anchor */
    f_score[nf] = topk_logp[q];
    f_tok[nf] = topk_ids[q];
    f_par[nf] = -1;
    f_dep[nf] = 1;
    f_live[nf] = 1;
    ++nf;
  }
  for (int i = 0; i < N; ++i) {
    long best = -1;
    for (long c = 0; c < nf; ++c) {
      if (!f_live[c]) continue;
      if (best < 0) { best = c; continue; }
      int better = f_score[c] > f_score[best] ||
                   (f_score[c] == f_score[best] &&
                    (f_tok[c] < f_tok[best] || (f_tok[c] == f_tok[best] && f_par[c] < f_par[best])));
      if (better) best = c;
    }
    f_live[best] = 0;
    parent[i] = f_par[best];
    token[i] = f_tok[best];
    depth[i] = f_dep[best];
    score[i] = f_score[best];
    if (f_dep[best] < K) { /* children of node i come from position depth[i]'s list */
      const int pos = f_dep[best];
      for (int q = 0; q < k; ++q) {
        f_score[nf] = score[i] + topk_logp[(long)pos * k + q];
        f_tok[nf] = topk_ids[(long)pos * k + q];
        f_par[nf] = i;
        f_dep[nf] = f_dep[best] + 1;
        f_live[nf] = 1;
        ++nf;
      }
    }
  }
  free(f_score); free(f_tok); free(f_par); free(f_dep); free(f_live);
  return 0;
}

int oracle_draft_step(const uint16_t* hidden, const int32_t* prefix_ids, const uint16_t* w_lm,
                      const uint16_t* emb, const uint16_t* w_ih, const uint16_t* w_hh,
                      const uint16_t* b_ih, const uint16_t* b_hh, const uint16_t* w1,
                      const uint16_t* b1, const uint16_t* w2, const uint16_t* b2, int B, int K,
                      int H, int V, int Ds, int R, int k, int N, const int32_t* seqs, int nseq,
                      double* logp_full, double* lse, int32_t* topk_ids, double* topk_logp,
                      int32_t* tree_parent, int32_t* tree_token, int32_t* tree_depth,
                      double* tree_score, int nthreads) {
  if (!hidden || !prefix_ids || !w_lm || !topk_ids || !topk_logp || !tree_parent || !tree_token ||
      !tree_depth || !tree_score)
    return ORACLE_ERR_ARG;
  if (B <= 0 || K <= 0 || H <= 0 || V <= 0 || R < 0 || k <= 0 || k > V || N <= 0)
    return ORACLE_ERR_ARG;
  const int use_head = (w2 != NULL && R > 0);
  if (use_head && (!emb || !w_ih || !w_hh || !w1 || Ds <= 0)) return ORACLE_ERR_ARG;
  if (!seqs) nseq = B;
  if (nseq <= 0) return ORACLE_ERR_ARG;

  double* hid = (double*)malloc((size_t)K * H * sizeof(double));
  double* E = (double*)malloc((size_t)K * H * sizeof(double));
  double* S = use_head ? (double*)malloc((size_t)K * Ds * sizeof(double)) : NULL;
  double* u = use_head ? (double*)malloc((size_t)K * R * sizeof(double)) : NULL;
  double* z = (double*)malloc((size_t)K * V * sizeof(double));
  double* lp = (double*)malloc((size_t)K * V * sizeof(double));
  double* ls = (double*)malloc((size_t)K * sizeof(double));
  int rc = 0;
  if (!hid || !E || !z || !lp || !ls || (use_head && (!S || !u))) rc = ORACLE_ERR_ARG;

  for (int si = 0; si < nseq && rc == 0; ++si) {
    const int b = seqs ? seqs[si] : si;
    if (b < 0 || b >= B) { rc = ORACLE_ERR_ARG; break; }
    for (long e = 0; e < (long)K * H; ++e) hid[e] = bf(hidden, (long)b * K * H + e);
    /* the ids are validated even when the correction branch is off */
    for (int j = 0; j < K; ++j) {
      int32_t id = prefix_ids[(long)b * K + j];
      if (id < 0 || id >= V) { rc = ORACLE_ERR_TOKEN; break; }
    }
    if (rc) break;
    if (use_head) {
      rc = oracle_embed(emb, V, H, prefix_ids + (long)b * K, K, E);
      if (!rc) rc = oracle_gru(E, K, H, Ds, w_ih, w_hh, b_ih, b_hh, S);
      if (!rc) rc = oracle_lowrank(hid, S, K, H, Ds, R, w1, b1, u);
      if (rc) break;
    }
    rc = oracle_logits(hid, u, K, H, V, use_head ? R : 0, w_lm, use_head ? w2 : NULL, b2, z, nthreads);
    if (!rc) rc = oracle_log_softmax(z, K, V, lp, ls);
    if (!rc) rc = oracle_topk(lp, K, V, k, topk_ids + (long)si * K * k, topk_logp + (long)si * K * k);
    if (!rc)
      rc = oracle_tree(topk_ids + (long)si * K * k, topk_logp + (long)si * K * k, K, k, N,
                       tree_parent + (long)si * N, tree_token + (long)si * N,
                       tree_depth + (long)si * N, tree_score + (long)si * N);
    if (rc) break;
    if (logp_full) memcpy(logp_full + (long)si * K * V, lp, (size_t)K * V * sizeof(double));
    if (lse) memcpy(lse + (long)si * K, ls, (size_t)K * sizeof(double));
  }
  free(hid); free(E); free(S); free(u); free(z); free(lp); free(ls);
  return rc;
}

/* O8: greedy verification of one tree (section 3.1): the target checks the whole draft at once and
   keeps the draft tokens up to the first one it would not have produced itself. */
int oracle_verify_greedy(const float* target, int N, int V, const int32_t* parent, const int32_t* token,
                         int32_t* row_argmax, int32_t* nodes, int32_t* n_acc, int32_t* bonus) {
  if (!target || !row_argmax || !nodes || !n_acc || !bonus || N < 0 || V <= 0) return ORACLE_ERR_ARG;
  if (N > 0 && (!parent || !token)) return ORACLE_ERR_ARG;
  for (int i = 0; i < N; ++i)
    if (parent[i] < -1 || parent[i] >= i) return ORACLE_ERR_ARG;
  for (int r = 0; r <= N; ++r) {
    const float* row = target + (long)r * V;
    int best = 0;
    for (int v = 1; v < V; ++v)
      if (row[v] > row[best]) best = v; /* strict: an equal value keeps the lower id */
    row_argmax[r] = best;
  }
  return oracle_tree_walk(N, parent, token, row_argmax, nodes, n_acc, bonus);
}

/* The walk shared by both verification rules: from the anchor, the target's choice a for the
   current node's row is kept when a child of that node carries it (the first such child in node
   order), and the walk continues from that child; the first choice that no child carries ends
   the walk and is the token the target adds itself (section 3.1). */
int oracle_tree_walk(int N, const int32_t* parent, const int32_t* token, const int32_t* row_choice,
                     int32_t* nodes, int32_t* n_acc, int32_t* bonus) {
  if (!row_choice || !nodes || !n_acc || !bonus || N < 0) return ORACLE_ERR_ARG;
  if (N > 0 && (!parent || !token)) return ORACLE_ERR_ARG;
  for (int i = 0; i < N; ++i)
    if (parent[i] < -1 || parent[i] >= i) return ORACLE_ERR_ARG;
  for (int i = 0; i < N; ++i) nodes[i] = -1;
  int cur = -1, n = 0;
  for (;;) {
    const int a = row_choice[cur + 1];
    int next = -1;
    for (int c = 0; c < N; ++c)
      if (parent[c] == cur && token[c] == a) { next = c; break; }
    if (next < 0) {
      *bonus = a;
      break;
    }
    nodes[n++] = next;
    cur = next;
  }
  *n_acc = n;
  return 0;
}

/* O11: one draw from the target's distribution at temperature T for one row of logits:
   p(v) = exp(l_v / T) / sum_v' exp(l_v' / T), computed as exp((l_v - max) / T) over its sum;
   the draw is the first id whose cumulative probability, summed in id order, exceeds u.  A u at
   or past the total (rounding) takes the last id of non-zero mass; a row with no finite value
   takes id 0. */
int oracle_row_sample(const float* row, int V, double T, double u, int32_t* id) {
  if (!row || !id || V <= 0 || !(T > 0.0) || !isfinite(T) || !(u >= 0.0 && u < 1.0)) return ORACLE_ERR_ARG;
  double m = -INFINITY;
  for (int v = 0; v < V; ++v)
    if ((double)row[v] > m) m = (double)row[v];
  if (!isfinite(m)) {
    *id = 0;
    return 0;
  }
  double Z = 0.0;
  for (int v = 0; v < V; ++v) Z += exp(((double)row[v] - m) / T);
  const double theta = u * Z;
  double c = 0.0;
  int last = 0;
  for (int v = 0; v < V; ++v) {
    const double w = exp(((double)row[v] - m) / T);
    if (w > 0.0) last = v;
    c += w;
    if (c > theta) {
      *id = v;
      return 0;
    }
  }
  *id = last;
  return 0;
}

/* O12: verification of one tree at temperature T > 0 (section 3.1's rule for sampled decoding,
   applied to a tree whose children are fixed proposals; the reading is in oracle_verify_sample's
   declaration): every row's draw (O11) with its own uniform, then the walk above. */
int oracle_verify_sample(const float* target, int N, int V, double T, const float* uniforms,
                         const int32_t* parent, const int32_t* token, int32_t* row_sample, int32_t* nodes,
                         int32_t* n_acc, int32_t* bonus) {
  if (!target || !uniforms || !row_sample || N < 0 || V <= 0) return ORACLE_ERR_ARG;
  for (int r = 0; r <= N; ++r) {
    const int rc = oracle_row_sample(target + (long)r * V, V, T, (double)uniforms[r], row_sample + r);
    if (rc) return rc;
  }
  return oracle_tree_walk(N, parent, token, row_sample, nodes, n_acc, bonus);
}

/* O13: Philox-4x32-10.  One round multiplies words 0 and 2 by the two round constants (full
   64-bit products), and the new words are (high product of word 2) ^ word 1 ^ key 0, (low product
   of word 2), (high product of word 0) ^ word 3 ^ key 1, (low product of word 0); the key grows
   by the two Weyl constants between rounds. */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  const uint64_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;
  uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += W0;
      k1 += W1;
    }
    const uint64_t p0 = M0 * (uint64_t)c0, p1 = M1 * (uint64_t)c2;
    const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    c0 = hi1 ^ c1 ^ k0;
    c1 = lo1;
    c2 = hi0 ^ c3 ^ k1;
    c3 = lo0;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* O14: u from the top 23 bits of the word, centred in its interval (never 0 or 1), then the
   Gumbel transform of the uniform. */
int oracle_gumbel_row(uint64_t seed, int b, int j, int V, double* g) {
  if (!g || b < 0 || j < 0 || V <= 0) return ORACLE_ERR_ARG;
  const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  for (int v = 0; v < V; ++v) {
    const uint32_t ctr[4] = {(uint32_t)v, (uint32_t)j, (uint32_t)(b / 4), 0u};
    uint32_t x[4];
    oracle_philox4x32_10(ctr, key, x);
    const double u = ((double)(x[b % 4] >> 9) + 0.5) / 8388608.0;
    g[v] = -log(-log(u));
  }
  return 0;
}

/* O9: the greedy sequential draft loop.  Each position is computed from scratch out of the
 * primitives above (the GRU re-run over the whole prefix chosen so far), so the only new step is
 * the feedback: the argmax of position j becomes the input of position j + 1. */
/* The draft loop of section 4.1.2 / Fig. 3 for every selection rule: with `uniforms` NULL and
 * `gumbel` 0 the greedy choice (O9), with `uniforms` the inverse-CDF draw (O10), with `gumbel`
 * the exponential race under `seed` (O15). */
static int rollout(const uint16_t* hidden, const int32_t* anchors, const float* uniforms, int gumbel, uint64_t seed,
                   const uint16_t* w_lm,
                   const uint16_t* emb, const uint16_t* w_ih, const uint16_t* w_hh, const uint16_t* b_ih,
                   const uint16_t* b_hh, const uint16_t* w1, const uint16_t* b1, const uint16_t* w2,
                   const uint16_t* b2, int B, int K, int H, int V, int Ds, int R, const int32_t* seqs, int nseq,
                   int32_t* tokens, double* logp, int nthreads) {
  if (!hidden || !anchors || !w_lm || !tokens || !logp) return ORACLE_ERR_ARG;
  if (B <= 0 || K <= 0 || H <= 0 || V <= 0 || R < 0) return ORACLE_ERR_ARG;
  const int use_head = (w2 != NULL && R > 0);
  if (use_head && (!emb || !w_ih || !w_hh || !w1 || Ds <= 0)) return ORACLE_ERR_ARG;
  if (!seqs) nseq = B;
  if (nseq <= 0) return ORACLE_ERR_ARG;

  int32_t* ids = (int32_t*)malloc((size_t)(K + 1) * sizeof(int32_t));
  double* hid = (double*)malloc((size_t)H * sizeof(double));
  double* E = (double*)malloc((size_t)K * H * sizeof(double));
  double* S = use_head ? (double*)malloc((size_t)K * Ds * sizeof(double)) : NULL;
  double* u = use_head ? (double*)malloc((size_t)R * sizeof(double)) : NULL;
  double* z = (double*)malloc((size_t)V * sizeof(double));
  double* lp = (double*)malloc((size_t)V * sizeof(double));
  double* gv = gumbel ? (double*)malloc((size_t)V * sizeof(double)) : NULL;
  double ls;
  int rc = 0;
  if (!ids || !hid || !E || !z || !lp || (use_head && (!S || !u)) || (gumbel && !gv)) rc = ORACLE_ERR_ARG;

  for (int si = 0; si < nseq && rc == 0; ++si) {
    const int b = seqs ? seqs[si] : si;
    if (b < 0 || b >= B) { rc = ORACLE_ERR_ARG; break; }
    ids[0] = anchors[b];
    if (ids[0] < 0 || ids[0] >= V) { rc = ORACLE_ERR_TOKEN; break; }
    for (int j = 0; j < K && rc == 0; ++j) {
      for (int c = 0; c < H; ++c) hid[c] = bf(hidden, ((long)b * K + j) * H + c);
      if (use_head) {
        /* the causal encoder over the prefix t_0 .. t_j chosen so far */
        rc = oracle_embed(emb, V, H, ids, j + 1, E);
        if (!rc) rc = oracle_gru(E, j + 1, H, Ds, w_ih, w_hh, b_ih, b_hh, S);
        if (!rc) rc = oracle_lowrank(hid, S + (long)j * Ds, 1, H, Ds, R, w1, b1, u);
        if (rc) break;
      }
      rc = oracle_logits(hid, u, 1, H, V, use_head ? R : 0, w_lm, use_head ? w2 : NULL, b2, z, nthreads);
      if (!rc) rc = oracle_log_softmax(z, 1, V, lp, &ls);
      if (rc) break;
      int best = 0;
      if (gumbel) {
        /* O15: the largest perturbed logit; strict, so an equal value keeps the lower id */
        rc = oracle_gumbel_row(seed, b, j, V, gv);
        if (rc) break;
        for (int v = 1; v < V; ++v)
          if (z[v] + gv[v] > z[best] + gv[best]) best = v;
      } else if (!uniforms) {
        for (int v = 1; v < V; ++v)
          if (z[v] > z[best]) best = v; /* strict: an equal value keeps the lower id */
      } else {
        /* O10: the first id whose cumulative probability (in id order) exceeds the uniform;
         * a uniform at or past the total (rounding) takes the last id of non-zero mass */
        const double uu = (double)uniforms[(long)b * K + j];
        double cdf = 0.0;
        int last = 0;
        best = -1;
        for (int v = 0; v < V; ++v) {
          const double pv = exp(lp[v]);
          if (pv > 0.0) last = v;
          cdf += pv;
          if (cdf > uu) { best = v; break; }
        }
        if (best < 0) best = last;
      }
      ids[j + 1] = best;
      tokens[(long)si * K + j] = best;
      logp[(long)si * K + j] = lp[best];
    }
  }
  free(ids); free(hid); free(E); free(S); free(u); free(z); free(lp); free(gv);
  return rc;
}

int oracle_rollout_greedy(const uint16_t* hidden, const int32_t* anchors, const uint16_t* w_lm,
                          const uint16_t* emb, const uint16_t* w_ih, const uint16_t* w_hh,
                          const uint16_t* b_ih, const uint16_t* b_hh, const uint16_t* w1,
                          const uint16_t* b1, const uint16_t* w2, const uint16_t* b2, int B, int K,
                          int H, int V, int Ds, int R, const int32_t* seqs, int nseq, int32_t* tokens,
                          double* logp, int nthreads) {
  return rollout(hidden, anchors, NULL, 0, 0, w_lm, emb, w_ih, w_hh, b_ih, b_hh, w1, b1, w2, b2, B, K, H, V, Ds, R, seqs,
                 nseq, tokens, logp, nthreads);
}

int oracle_rollout_sample(const uint16_t* hidden, const int32_t* anchors, const float* uniforms,
                          const uint16_t* w_lm, const uint16_t* emb, const uint16_t* w_ih,
                          const uint16_t* w_hh, const uint16_t* b_ih, const uint16_t* b_hh,
                          const uint16_t* w1, const uint16_t* b1, const uint16_t* w2, const uint16_t* b2,
                          int B, int K, int H, int V, int Ds, int R, const int32_t* seqs, int nseq,
                          int32_t* tokens, double* logp, int nthreads) {
  if (!uniforms) return ORACLE_ERR_ARG;
  for (long i = 0; i < (long)B * K; ++i)
    if (!(uniforms[i] >= 0.0f && uniforms[i] < 1.0f)) return ORACLE_ERR_ARG;
  return rollout(hidden, anchors, uniforms, 0, 0, w_lm, emb, w_ih, w_hh, b_ih, b_hh, w1, b1, w2, b2, B, K, H, V, Ds,
                 R, seqs, nseq, tokens, logp, nthreads);
}

int oracle_rollout_sample_gumbel(const uint16_t* hidden, const int32_t* anchors, uint64_t seed,
                                 const uint16_t* w_lm, const uint16_t* emb, const uint16_t* w_ih,
                                 const uint16_t* w_hh, const uint16_t* b_ih, const uint16_t* b_hh,
                                 const uint16_t* w1, const uint16_t* b1, const uint16_t* w2, const uint16_t* b2,
                                 int B, int K, int H, int V, int Ds, int R, const int32_t* seqs, int nseq,
                                 int32_t* tokens, double* logp, int nthreads) {
  return rollout(hidden, anchors, NULL, 1, seed, w_lm, emb, w_ih, w_hh, b_ih, b_hh, w1, b1, w2, b2, B, K, H, V, Ds,
                 R, seqs, nseq, tokens, logp, nthreads);
}
