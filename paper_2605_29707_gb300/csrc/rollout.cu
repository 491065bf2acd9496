// rollout.cu -- launch of the sequential draft loop (the kernels are in rollout_kernels.cuh): the
// shared-memory and tensor-memory layout a launch takes, and the greedy and inverse-CDF
// instantiations; the exponential race's are in rollout_race.cu.
#include "rollout_kernels.cuh"

namespace dm {

// ================================================================ launch
// Resident kernel: shared-memory W2 rows that fit beside u, the staged base logits and `extra`
// bytes (h_j of every sequence for two-barrier steps); -1 when those alone do not fit.
static int resident_smem_rows(int B, int V, int R, int grid, long long extra = 0) {
  const int rows_cta = resident_rows_per_cta(V, grid);
  const long long fixed =
      static_cast<long long>(B) * R * 4 + static_cast<long long>(B + 1) * rows_cta * 4 + extra;
  const long long avail = static_cast<long long>(kRollMaxSmem) - fixed;
  if (avail < 0) return -1;
  const long long fit = (avail / (2LL * R)) & ~3LL;
  const long long want = rows_cta > kTmemRows ? rows_cta - kTmemRows : 0;
  return static_cast<int>(fit < want ? fit : want);
}

size_t rollout_smem_bytes(int B, int V, int R, bool head, int grid) {
  if (head && R <= kResidentMaxR) {
    const int ns = resident_smem_rows(B, V, R, grid);
    if (ns < 0) return kRollMaxSmem + 1;
    return static_cast<size_t>(ns) * R * 2 + static_cast<size_t>(B) * R * 4 +
           static_cast<size_t>(B + 1) * resident_rows_per_cta(V, grid) * 4;
  }
  return (head ? static_cast<size_t>(kW2Stages) * kW2StageBytes : 0) +
         static_cast<size_t>(B) * (head ? R : 0) * sizeof(float) +
         static_cast<size_t>(B) * rollout_rows_per_cta(V, R, head, grid) * sizeof(float);
}

// Two grid barriers per step (phase A done by every CTA for all units, gates_all / ub_phase):
// the resident kernel with a table, when h_j of every sequence fits in shared memory beside u and
// the base logits (the shared-memory W2 rows give way to it).
static bool use_fast_gates(const RolloutParams& p, int grid) {
  // gates_all reads the biases four at a time (8-byte loads)
  const bool bias_ok = (reinterpret_cast<uintptr_t>(p.b_ih) & 7u) == 0 && (reinterpret_cast<uintptr_t>(p.b_hh) & 7u) == 0;
  return use_resident(p) && p.x_table && p.uh && p.gh && p.ucount && p.uhcount && p.Ds <= 1024 && bias_ok &&
         resident_smem_rows(p.B, p.V, p.R, grid, static_cast<long long>(p.B) * p.Ds * 4 + 16) >= 0;
}

// Phase C on the tensor cores (two-barrier steps, at most two sequences, r a multiple of 64 up to
// 256): the 128-row blocks of a CTA's rows, tb in tensor memory and sb in shared memory, that
// cover the most rows (tensor memory first: an A block there costs r/2 columns and its D 16 more;
// one in shared memory costs 128 r bf16 beside the fixed buffers).  False when the layout does
// not apply or would leave more than kMmaMaxL2Rows rows of a CTA to read through L2 every step.
static bool mma_blocks(const RolloutParams& p, int grid, int* tb, int* sb, size_t* smem) {
  *tb = *sb = 0;
  if (!use_fast_gates(p, grid) || p.B > 2 || p.R % 64 != 0 || p.R > 256) return false;
  const int rows_cta = resident_rows_per_cta(p.V, grid);
  const int need = (rows_cta + 127) / 128;
  const long long fixed = 1024 + static_cast<long long>(p.R / 64) * kMmaBopTileBytes +
                          static_cast<long long>(p.B) * p.R * 4 + static_cast<long long>(p.B + 1) * rows_cta * 4 +
                          static_cast<long long>(p.B) * p.Ds * 4 + 16;
  const long long blk = static_cast<long long>(p.R / 64) * kMmaTileBytes;
  if (fixed > static_cast<long long>(kRollMaxSmem)) return false;
  const int s_max = static_cast<int>((static_cast<long long>(kRollMaxSmem) - fixed) / blk);
  int bt = 0, bs = 0;
  for (int t = 0; t <= need; ++t) {
    const int room = kTmemCols - t * (p.R / 2);  // columns left for the D blocks
    if (room < 16 * t) break;
    const int s = std::min(std::min(s_max, need - t), room / 16 - t);
    if (s < 0) continue;
    if (t + s > bt + bs || (t + s == bt + bs && t > bt)) { bt = t; bs = s; }
  }
  if (bt + bs == 0 || rows_cta - 128 * (bt + bs) > kMmaMaxL2Rows) return false;
  *tb = bt;
  *sb = bs;
  *smem = static_cast<size_t>(fixed + bs * blk);
  return true;
}

cudaError_t launch_rollout(const RolloutParams& p, int grid, cudaStream_t stream, const CUtensorMap* tm_w2) {
  if (p.B < 1 || p.B > kRollMaxB || grid < 1) return cudaErrorInvalidValue;
  if (p.uniforms && (grid > kRollThreads || !p.lg)) return cudaErrorInvalidValue;  // one thread per CTA
  if (p.race && (p.uniforms || !p.best)) return cudaErrorInvalidValue;  // one rule; the race uses the key slots
  size_t smem = rollout_smem_bytes(p.B, p.V, p.R, p.head, grid);
  if (smem > kRollMaxSmem) return cudaErrorInvalidValue;
  RolloutParams pp = p;
  pp.smem_rows = use_resident(p) ? resident_smem_rows(p.B, p.V, p.R, grid) : 0;
  pp.fast_gates = use_fast_gates(p, grid) ? 1 : 0;
  pp.mma_tb = pp.mma_sb = 0;
  if (pp.fast_gates) {
    const long long hbytes = static_cast<long long>(p.B) * p.Ds * 4 + 16;  // + alignment of s_h
    pp.smem_rows = resident_smem_rows(p.B, p.V, p.R, grid, hbytes);
    smem = static_cast<size_t>(pp.smem_rows) * p.R * 2 + static_cast<size_t>(p.B) * p.R * 4 +
           static_cast<size_t>(p.B + 1) * resident_rows_per_cta(p.V, grid) * 4 + static_cast<size_t>(hbytes);
    int tb = 0, sb = 0;
    size_t mma_smem = 0;
    if (tm_w2 != nullptr && mma_blocks(pp, grid, &tb, &sb, &mma_smem)) {
      pp.mma_tb = tb;
      pp.mma_sb = sb;
      pp.smem_rows = 0;
      smem = mma_smem;
    }
    if (smem > kRollMaxSmem) return cudaErrorInvalidValue;
  }
  if (!use_resident(p)) pp.uh = nullptr;  // only the resident kernel computes it before its steps
  CUtensorMap tm;
  if (tm_w2 != nullptr) tm = *tm_w2;
  else memset(&tm, 0, sizeof(tm));  // never read: phase C stays on the CUDA cores
  if (pp.race) return launch_rollout_race(pp, grid, smem, stream, tm);
  return launch_rollout_b<false>(pp, grid, smem, stream, tm);
}

}  // namespace dm
