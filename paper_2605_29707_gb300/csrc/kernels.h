// kernels.h -- internal (C++) interface between the C-ABI host code and the CUDA kernels.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace dm {

enum TcMode { kModeSoftmax = 0, kModeStore = 1 };

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
  const __nv_bfloat16* bias;  // softmax: b2 [V] or nullptr
  float* out;                 // softmax: partial records [M][rec fields][nchunks]; store: [splits][M][ld_out]
  int ld_out;
  int* status;
};

constexpr int kSoftmaxRecWords(int kmax) { return 2 + 2 * kmax; }

// Tensor maps in the order A1, B1, A2, B2 (A = 128-row operand, B = N-row operand).
cudaError_t launch_tc_gemm(int mode, int bn, bool swap, int kmax, const CUtensorMap* maps,
                           const TcParams& p, int grid, cudaStream_t stream);

// ---------------------------------------------------------------- gather / GRU
struct GatherParams {
  const int32_t* ids;       // [M]
  const __nv_bfloat16* emb; // [V, H]
  __nv_bfloat16* E;         // [M, H] or nullptr (validate only)
  int M, H, V;
  int* status;
};
cudaError_t launch_gather(const GatherParams& p, cudaStream_t stream);

struct GruParams {
  const float* xpart;  // [xsplits][M][3*Ds]  partial sums of E . W_ih^T
  int xsplits;
  const float* upart;  // [usplits][M][R]     partial sums of hidden . W1[:, :H]^T
  int usplits;
  const __nv_bfloat16* w_hh;  // [3*Ds, Ds]
  const __nv_bfloat16* b_ih;  // [3*Ds] or nullptr
  const __nv_bfloat16* b_hh;  // [3*Ds] or nullptr
  const __nv_bfloat16* w1;    // [R, H + Ds]
  const __nv_bfloat16* b1;    // [R] or nullptr
  int B, K, H, Ds, R;
  int units;                  // hidden units owned by one CTA
  float* S;                   // [M][Ds] causal states (fp32)
  __nv_bfloat16* u;           // [M][R] low-rank code
  unsigned int* barrier;      // zeroed grid-barrier counter
  int* status;
};
int gru_grid(int Ds, int num_sms, int* units);
size_t gru_smem_bytes(int Ds, int units, int M, int B);  // 0 = does not fit
cudaError_t launch_gru(const GruParams& p, int grid, cudaStream_t stream);

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
};
cudaError_t launch_merge_tree(const TreeParams& p, cudaStream_t stream);

}  // namespace dm
