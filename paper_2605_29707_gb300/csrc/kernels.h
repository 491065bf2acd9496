// kernels.h -- internal (C++) interface between the C-ABI host code and the CUDA kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dm {

enum TcMode { kModeSoftmax = 0, kModeStore = 1 };

// Raises a kernel's dynamic shared-memory limit to at least `smem` bytes on the current device
// (with `carveout`, also asks for the largest shared-memory carveout), once per device, kernel
// and size; safe to call from several host threads (api.cu).
cudaError_t ensure_smem_attr(const void* func, size_t smem, bool carveout);

// Most deferred tiles one CTA of the vocabulary GEMM can hold (each has its own completion
// barrier in shared memory).
constexpr int kMaxDefer = 32;

// One tcgen05 GEMM launch: acc[tok, w] = sum over two K segments of
//   seg1: X1[tok, :] . W1[w, :]      (k blocks 0 .. nkb1-1)
//   seg2: X2[tok, :] . W2[w, :]      (k blocks nkb1 .. nkb1+nkb2-1)
// "tok" rows are activations (M of them), "w" rows are weight rows (vocabulary entries or
// output features).  With swap = 1 the weight tile is the 128-row MMA operand A and the
// token tile the N-row operand B (small M); with swap = 0 the token tile is A (128 rows) and
// the weight tile B (N = 256 rows).
struct TcParams {
  int nkb1, nkb2;
  int rows_tok, rows_w;
  int tok_tiles, w_tiles;
  // softmax mode: CTA c handles token tile c % tok_tiles and weight tiles
  // [chunk * w_per_chunk, ...) with chunk = c / tok_tiles
  int nchunks, w_per_chunk;
  // store mode: items (tok tile, w tile, split) round-robin over the CTAs
  int splits, kb_per_split, total_items;
  int w_evict_first;
  int defer;      // softmax + swap only: number of leading tiles whose second segment waits for
                  // the preceding grid (0 = off); see the producer in tc_gemm.cuh
  int pdl_wait;   // launched as a programmatic dependent: 1 = wait for the preceding grid before
                  // the first load, 2 = after the last load, 3 = before the first load of the
                  // second K segment (the pair kernel; 0 = no wait)
  int mcast;      // tokens-on-M orientation: CTAs per cluster sharing each weight box by TMA
                  // multicast (1 = off; 2 or 4, dividing tok_tiles); the weight maps' box is
                  // BN / mcast rows high
  int tmem_cols;  // TMEM columns to allocate (power of two, 32..512)
  const __nv_bfloat16* bias;  // softmax: b2 [V] or nullptr
  float* out;                 // softmax: partial records [M][rec fields][nchunks]; store: [splits][M][ld_out]
  int ld_out;
  int* status;
};

constexpr int kSoftmaxRecWords(int kmax) { return 2 + 2 * kmax; }

// Tensor maps in the order A1, B1, A2, B2 (A = 128-row operand, B = N-row operand).
cudaError_t launch_tc_gemm(int mode, int bn, bool swap, int kmax, const CUtensorMap* maps,
                           const TcParams& p, int grid, cudaStream_t stream);
// The store-mode GEMM for many tokens (bn 256, tokens on M) launched as a programmatic dependent
// of the kernel before it (p.pdl_wait says where it waits for that kernel).
cudaError_t launch_tc_store_dependent(const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t stream);
// Deferred-segment vocabulary GEMM launched as a programmatic dependent of the GRU kernel
// (bn 16 or 32; fewer pipeline stages so that its CTAs fit beside the GRU's on one SM).
cudaError_t launch_tc_softmax_deferred(int bn, int kmax, const CUtensorMap* maps, const TcParams& p, int grid,
                                       cudaStream_t stream);
// Shared memory one deferred-mode CTA uses (for the co-residency budget).
int tc_softmax_deferred_smem(int bn, int kmax);
// The same three for 8-entry top-k lists (kmax = 8; tc_softmax_k8.cu).
cudaError_t launch_tc_softmax_k8(int bn, bool swap, const CUtensorMap* maps, const TcParams& p, int grid,
                                 cudaStream_t stream);
cudaError_t launch_tc_softmax_deferred_k8(int bn, const CUtensorMap* maps, const TcParams& p, int grid,
                                          cudaStream_t stream);
int tc_softmax_deferred_smem_k8(int bn);
// Tokens on M in CTA pairs (mcast = 2, bn 256): the 2-SM MMA variant (tc_pair.cuh); the maps are
// the same as for the multicast kernel (weight boxes 128 rows high).
cudaError_t launch_tc_vocab_pair(int kmax, const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t stream);
cudaError_t launch_tc_vocab_pair_k8(const CUtensorMap* maps, const TcParams& p, int grid, cudaStream_t stream);
// Small-M (swap, bn 16..128) store-mode GEMM with four pipeline stages, launched as a
// programmatic dependent of the preceding kernel (p.pdl_wait says where it waits for it).
cudaError_t launch_tc_store_chained(int bn, const CUtensorMap* maps, const TcParams& p, int grid,
                                   cudaStream_t stream);
// Shared memory one such CTA uses.
int tc_store_chained_smem(int bn);

// ---------------------------------------------------------------- gather / GRU
struct GatherParams {
  const int32_t* ids;       // [M]
  const __nv_bfloat16* emb; // [V, H]
  __nv_bfloat16* E;         // [M, H] or nullptr (validate only)
  uint32_t* hx;             // [M, Ds] tagged GRU states to clear, or nullptr
  int M, H, V, Ds;
  int* status;
};
cudaError_t launch_gather(const GatherParams& p, cudaStream_t stream);

// GRU recurrence.  CTA (cu, cb) of a gu x gb grid owns hidden units [cu*units, cu*units+units)
// (gate rows r|z|n of each) for sequences [cb*bc, cb*bc+bc).  States travel between CTAs as
// tagged words in hx: bf16 value in the high half, a non-zero flag in the low half, one row
// per (sequence, position) written once per step, so a reader polls the data itself.
struct GruParams {
  const float* xpart;  // [xsplits][M][3*Ds]  partial sums of E . W_ih^T
  int xsplits;
  const float* upart;  // [usplits][M][R]     partial sums of hidden . W1[:, :H]^T (u phase only)
  int usplits;
  const __nv_bfloat16* w_hh;  // [3*Ds, Ds]
  const __nv_bfloat16* b_ih;  // [3*Ds] or nullptr
  const __nv_bfloat16* b_hh;  // [3*Ds] or nullptr
  const __nv_bfloat16* w1;    // [R, H + Ds]
  const __nv_bfloat16* b1;    // [R] or nullptr
  int B, K, H, Ds, R;
  int units, gu, gb, bc;      // grid shape: gu unit blocks x gb sequence groups of bc
  float* xs;                  // [M][3*Ds] input-gate sums (scratch)
  uint32_t* hx;               // [M][Ds] tagged states (words of earlier steps carry other tags)
  __nv_bfloat16* s_out;       // [M][Ds] plain bf16 states, or nullptr
  __nv_bfloat16* u;           // [M][R] low-rank code computed in-kernel, or nullptr
  int* status;
  // Fused projections (small batches, u computed in-kernel): with ids set, the kernel computes
  // its own input-gate sums E . W_ih^T (E = emb rows of ids, checked against V) and the hidden
  // half of u, and xpart / upart are unused; hx is not cleared before the launch (see layout).
  const int32_t* ids;         // [M] or nullptr
  const __nv_bfloat16* emb;   // [V, H]
  const __nv_bfloat16* w_ih;  // [3*Ds, H]
  const __nv_bfloat16* hidden;  // [M, H]
  int V;
  const uint32_t* epoch;      // the workspace's step epoch (the state words' tag)
  unsigned int* seq_done;     // [B] merge counters
  int reset_ctrl;             // no clear before the launch: CTA 0 resets the status and seq_done
  // Input-projection table emb . W_ih^T [V, 3*Ds] fp32, or nullptr: when set, each step reads
  // its input-gate sums as b_ih + row x_ids[m] of it, and xpart / xs / the fused path's own
  // product are not used.
  const float* x_table;
  const int32_t* x_ids;       // [M] the prefix ids (read with x_table)
  // No clear before the launch (fused projections): the control word recording which byte range
  // of the workspace held nothing but state words at the end of the last step (lo | hi << 32, 0 =
  // none; every other kind of step zeroes it), this launch's hx range packed the same way, and
  // the grid barrier word (generation << 32 | arrivals) of the clear that runs when the recorded
  // range does not contain this launch's.  layout == nullptr: hx arrives cleared.
  unsigned long long* layout;
  unsigned long long layout_range;
  unsigned long long* clear_bar;
};
// Packs a workspace byte range [lo, hi) the way GruParams::layout holds it.
inline unsigned long long hx_range(size_t lo, size_t hi) {
  return static_cast<unsigned long long>(lo) | (static_cast<unsigned long long>(hi) << 32);
}
// Failure-detection test hook (domino_debug_hold): while armed, GRU CTA `cta` withholds one
// thing its peers wait for -- kHoldPublish: its states of position `step`; kHoldClearBarrier: its
// arrival at the clear barrier -- so their bounded waits run out.  The held CTA disarms it.
constexpr int kHoldOff = 0, kHoldPublish = 1, kHoldClearBarrier = 2;
cudaError_t arm_gru_hold(int what, int cta, int step);
// Largest number of (rank row, position) pairs of u one warp finalises for which the fused
// projections apply (their hidden halves wait in shared memory).
constexpr int kGruMaxUPairs = 8;
struct GruPlan {
  int units, gu, gb, bc;
  size_t smem;  // 0 = unsupported
};
GruPlan gru_plan(int B, int Ds, int num_sms);
// Cooperative launch; with pdl, also as a programmatic dependent of the preceding kernel (the
// kernel waits for that grid before it reads the projections).  wide: the launch shares no SM
// with the vocabulary GEMM (not with fused projections): one CTA's worth of registers per SM.
cudaError_t launch_gru(const GruParams& p, const GruPlan& plan, cudaStream_t stream, bool pdl, bool wide);

// u = bf16(SiLU(b1 + sum over splits of part)) for the large-batch path.
struct UFinalParams {
  const float* part;  // [splits][M][R]
  int splits, M, R;
  const __nv_bfloat16* b1;
  __nv_bfloat16* u;
};
// pdl: launched as a programmatic dependent of the W1 GEMM (it waits for it before reading)
cudaError_t launch_u_finalize(const UFinalParams& p, cudaStream_t stream, bool pdl = false);

// ---------------------------------------------------------------- merge + tree
struct TreeParams {
  const float* partials;  // [M][rec fields][nchunks]
  unsigned int* seq_done; // [B] zeroed counters: rows of each sequence merged so far
  int nchunks, kmax;
  int B, K, k, N;
  int32_t* topk_ids;      // [B, K, k]
  float* topk_logp;       // [B, K, k]
  int32_t* tree_parent;   // [B, N]
  int32_t* tree_token;
  int32_t* tree_depth;
  float* tree_score;      // or nullptr
  const int* status;      // the step's device status word
  int32_t* status_out;    // or nullptr: a copy of it beside the outputs, made once the step is done
  uint32_t* epoch;        // the workspace's step epoch, advanced once the step's GRU is done
};
cudaError_t launch_merge_tree(const TreeParams& p, cudaStream_t stream);

// ---------------------------------------------------------------- sequential draft loop (rollout*.cu)
constexpr int kRollMaxB = 8;  // sequences per rollout launch
constexpr unsigned kGreedyIdMask = 0x3FFFFFu;  // greedy rollout keys: token ids below 2^22
constexpr int kRollComputeWarps = 8;             // compute warps of a rollout CTA
struct RolloutParams {
  const __nv_bfloat16* hidden;  // [B, K, H]
  const int32_t* anchors;       // [B]
  const __nv_bfloat16 *emb, *w_ih, *w_hh, *b_ih, *b_hh, *w1, *b1, *w2, *b2;  // b* may be null
  int head;                     // correction branch on (R > 0 and W2 given)
  int B, K, H, V, Ds, R;
  int smem_rows;                // set by launch_rollout: W2 rows a CTA keeps in shared memory
  const float* base;            // [B*K, V] W_lm hidden (fp32, from the store-mode GEMM)
  float* h;                     // [2][B][Ds] GRU states (cleared: h_{-1} = 0)
  float* u;                     // [B][R]
  float* partials;              // float4 (max, sum exp, argmax bits, 0) per sequence: greedy
                                // [K][grid][kRollComputeWarps][kRollMaxB] (per warp); sampled
                                // [2][grid][kRollMaxB] (per CTA), by step parity
  unsigned long long* best;     // greedy and race: [2][kRollMaxB] keys of each sequence's (perturbed)
                                // argmax by step parity (cleared); nullptr in inverse-CDF mode (every CTA
                                // combines the partials)
  unsigned* barrier;            // grid barrier counter (cleared)
  int32_t* tokens;              // [B, K] t_1 .. t_K
  float* logp;                  // [B, K]
  int* status;
  const float* uniforms;        // [B, K] in [0, 1): sampled mode (inverse CDF); nullptr: greedy or race
  int race;                     // seeded sampled mode: t_{j+1} = argmax_v L_j[v] + Gumbel(seed, b, j, v)
                                // (the exponential race); keys, partials and logp as greedy (best set)
  unsigned long long seed;      // race: the generator's key
  float* lg;                    // [2][B][V] sampled mode: every CTA's final logits, by step parity
  const float* x_table;         // [V, 3 Ds] emb . W_ih^T, or nullptr (phase A projects emb[t] itself)
  float* uh;                    // [B*K][R] scratch for hidden . W1[:, :H]^T (resident kernel), or nullptr
  float* gh;                    // [2][B][3 Ds] W_hh h_j of the next step's gates, by step parity
  int fast_gates;               // set by launch_rollout: one grid barrier per step (resident kernel,
                                // table, h_j of every sequence in each CTA's shared memory)
  unsigned* ucount;             // rows of u finished so far in this launch (cleared), fast_gates only
  unsigned* uhcount;            // warps done with uh before the steps (cleared), fast_gates only
  int mma_tb, mma_sb;           // set by launch_rollout: phase C on the tensor cores over mma_tb
                                // 128-row W2 blocks in tensor memory and mma_sb in shared memory
                                // (both 0: phase C on the CUDA cores)
};
// dynamic shared memory of one rollout CTA (the resident W2 rows or the W2 ring, u of every
// sequence and this CTA's rows of base logits + b2): at most kRollMaxSmem, the 227 KB a CTA may
// hold less 2 KB for the kernels' static shared memory
constexpr size_t kRollMaxSmem = 225 * 1024;
size_t rollout_smem_bytes(int B, int V, int R, bool head, int grid);
// tm_w2: tensor map of W2 [V, r] bf16 (boxes of 64 x 128, 128-byte swizzle), or nullptr; without it
// phase C stays on the CUDA cores.
cudaError_t launch_rollout(const RolloutParams& p, int grid, cudaStream_t stream, const CUtensorMap* tm_w2);

// ---------------------------------------------------------------- tree verification (verify.cu)
cudaError_t launch_verify_greedy(const float* logits, const int32_t* parent, const int32_t* token, int B, int N,
                                 int V, int32_t* row_argmax, int32_t* nodes, int32_t* count, int32_t* bonus,
                                 cudaStream_t stream);
// Row draws from softmax(logits / T) (inv_t = 1 / T) with one uniform per row, then the same walk;
// a row slice of at most kMaxSampleSlice floats is staged in shared memory (V <= 8 of them).
constexpr int kMaxSampleSlice = 53248;
cudaError_t launch_verify_sample(const float* logits, const int32_t* parent, const int32_t* token,
                                 const float* uniforms, int B, int N, int V, float inv_t, int32_t* row_sample,
                                 int32_t* nodes, int32_t* count, int32_t* bonus, cudaStream_t stream);

}  // namespace dm
