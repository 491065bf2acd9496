// api.cu -- host side of the C ABI declared in include/domino.h: argument checks, the launch
// plan for the current device, workspace layout, TMA tensor maps and the launch sequence.
//
// Launch sequence of one step (all on the caller's stream).  Small batches (B <= 2 at K = 16):
//   gru      prologue: prefix-id check, E . W_ih^T from the embedding rows by id (or rows of the
//            input-projection table) and hidden . W1[:, :H]^T; then S_j = GRU(E_0..E_j) and
//            u = SiLU(. + S . W1[:, H:]^T + b1)  (cooperative; its first CTA resets the status)
//   tc soft  logits = [hidden | u] . [W_lm | W2]^T + b2, online max / sum-exp / top-k
//            (a programmatic dependent of the GRU: the W_lm segment streams beside it)
//   tree     merge the partials -> lse, top-k log-probs; best-first draft tree
// Other batches: memset (the control words: status, merge counters), gather (id check, state
// words cleared; E = emb[ids] unless a table is given), tc store Xp = E . W_ih^T (not with a
// table), tc store Up = hidden . W1[:, :H]^T, gru, tc soft, tree; large M moves the W1 GEMM
// (both halves) and a SiLU kernel (u_finalize) after the GRU, and launches X, GRU, W1,
// u_finalize and the vocabulary GEMM on CTA pairs each as a programmatic dependent of the kernel
// before it (the pair kernel waits for u only before its W2 segment).  With the correction
// branch off only memset, gather (id check), tc soft and tree run.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <atomic>
#include <cmath>
#include <map>
#include <mutex>
#include <utility>
#include <vector>

#include "domino.h"
#include "kernels.h"

// ---------------------------------------------------------------- kernel attributes
namespace dm {
cudaError_t ensure_smem_attr(const void* func, size_t smem, bool carveout) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, size_t> done;  // (device, kernel) -> limit set
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> lock(mu);
  size_t& have = done[std::make_pair(dev, func)];
  if (have >= smem) return cudaSuccess;
  e = cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  if (carveout) {
    e = cudaFuncSetAttribute(func, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    if (e != cudaSuccess) return e;
  }
  have = smem;
  return cudaSuccess;
}
}  // namespace dm

namespace {

using dm::TcParams;

constexpr int kMaxTopk = 32;
constexpr int kMaxN = 256;
constexpr int kMaxK = 64;
constexpr int kMaxDs = 2048;
constexpr int kMaxV = 1 << 22;
constexpr size_t kAlign = 256;

size_t align_up(size_t x) { return (x + kAlign - 1) & ~(kAlign - 1); }
int ceil_div(int a, int b) { return (a + b - 1) / b; }
int pow2_at_least(int x, int lo) {
  int v = lo;
  while (v < x) v <<= 1;
  return v;
}

struct StorePlan {
  bool swap = false;
  int bn = 0, tok_tiles = 0, w_tiles = 0, nkb = 0, splits = 0, kb_per_split = 0, total_items = 0, grid = 0;
};

struct Plan {
  int B, K, H, V, Ds, R, k, N, M;
  bool head;
  int num_sms;
  // fused vocabulary GEMM
  bool swap;
  int bn, kmax, rec, tok_tiles, w_tiles, nchunks, w_per_chunk, grid;
  StorePlan xg, ug;
  int mcast;   // vocab GEMM, tokens on M: CTAs per cluster sharing each weight box (1 = off)
  bool chain;  // head kernels launched as a programmatic-dependent chain (small M with overlap)
  bool fused;  // chain path whose GRU computes E . W_ih^T and hidden . W1[:, :H] itself (no
               // gather and no projection GEMMs; the step's first kernel is the GRU)
  dm::GruPlan gru;
  bool u_in_gru;  // small M: u finished inside the GRU kernel; large M: W1 GEMM + finalize
  bool overlap;   // vocab GEMM launched as a programmatic dependent of the GRU (deferred W2)
  int defer_tiles;  // leading tiles per CTA whose W2 segment waits for the GRU
  int tmem_cols;  // TMEM columns of the vocab GEMM
  // workspace layout (offsets in bytes)
  size_t ctrl_bytes, clear_bytes;  // clear_bytes from off_ctrl: the control words (+ hx, fused)
  size_t off_ctrl, off_E, off_xpart, off_upart, off_xs, off_hx, off_S, off_u, off_part, dev_total;
  size_t off_hid, off_ids, off_tid, off_tlp, off_tpar, off_ttok, off_tdep, off_tsc, off_ostat, host_total;
};

// Orientation: up to 128 tokens ride on the MMA's N dimension (weights fill the 128-row
// operand); more tokens take the 128-row operand with 256 weight rows per tile.
void choose_orientation(int M, bool* swap, int* bn) {
  if (M <= 128) {
    *swap = true;
    *bn = pow2_at_least(M, 16);
  } else {
    *swap = false;
    *bn = 256;
  }
}

StorePlan plan_store(int M, int rows_w, int nkb, int num_sms) {
  StorePlan s;
  choose_orientation(M, &s.swap, &s.bn);
  s.tok_tiles = s.swap ? ceil_div(M, s.bn) : ceil_div(M, 128);
  s.w_tiles = s.swap ? ceil_div(rows_w, 128) : ceil_div(rows_w, s.bn);
  s.nkb = nkb;
  const int items = s.tok_tiles * s.w_tiles;
  int splits = num_sms / items;
  if (splits < 1) splits = 1;
  if (splits > nkb) splits = nkb;
  s.kb_per_split = ceil_div(nkb, splits);
  s.splits = ceil_div(nkb, s.kb_per_split);
  s.total_items = items * s.splits;
  s.grid = s.total_items < num_sms ? s.total_items : num_sms;
  return s;
}

long long tree_capacity(int K, int k) {  // sum_{d=1..K} k^d, saturated
  long long cap = 0, pw = 1;
  for (int d = 1; d <= K; ++d) {
    pw *= k;
    cap += pw;
    if (cap > (1LL << 40)) return 1LL << 40;
    if (pw > (1LL << 40)) pw = 1LL << 40;
  }
  return cap;
}

int device_sms(int* sms, int* major, int* minor) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (cudaDeviceGetAttribute(major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (cudaDeviceGetAttribute(minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) return DOMINO_ERR_CUDA;
  return DOMINO_OK;
}

// Size checks that do not need pointers.  Returns DOMINO_OK or an error code.
int check_sizes(int B, int K, int H, int V, int Ds, int R, int k, int N, bool head) {
  if (B <= 0 || K <= 0 || H <= 0 || V <= 0 || k <= 0 || N <= 0) return DOMINO_ERR_INVALID_ARG;
  if (k > V) return DOMINO_ERR_INVALID_ARG;
  if (static_cast<long long>(N) > tree_capacity(K, k)) return DOMINO_ERR_INVALID_ARG;
  if (head && (Ds <= 0 || R < 0)) return DOMINO_ERR_INVALID_ARG;
  if (H % 8 != 0 || k > kMaxTopk || N > kMaxN || K > kMaxK || V >= kMaxV) return DOMINO_ERR_UNSUPPORTED;
  if (head && (Ds % 8 != 0 || R % 8 != 0 || Ds > kMaxDs)) return DOMINO_ERR_UNSUPPORTED;
  if (static_cast<long long>(B) * K > (1LL << 24)) return DOMINO_ERR_UNSUPPORTED;
  return DOMINO_OK;
}

// The plan for a GPU with `sms` SMs (sizes already checked).
int make_plan_sms(int B, int K, int H, int V, int Ds, int R, int k, int N, bool head, int sms, Plan* P) {
  Plan& p = *P;
  p = Plan{};  // every member zero (the nested plans' defaults are zero too)
  p.B = B; p.K = K; p.H = H; p.V = V; p.k = k; p.N = N;
  p.head = head;
  p.Ds = head ? Ds : 0;
  p.R = head ? R : 0;
  p.M = B * K;
  p.num_sms = sms;
  const int M = p.M;

  choose_orientation(M, &p.swap, &p.bn);
  // top-k list length per (token, CTA): the merge reads only the first k entries
  p.kmax = k <= 8 ? 8 : (k <= 16 ? 16 : 32);
  p.rec = dm::kSoftmaxRecWords(p.kmax);
  p.tok_tiles = p.swap ? ceil_div(M, p.bn) : ceil_div(M, 128);
  p.w_tiles = p.swap ? ceil_div(V, 128) : ceil_div(V, p.bn);
  int per_tok = sms / p.tok_tiles;
  if (per_tok < 1) per_tok = 1;
  p.w_per_chunk = ceil_div(p.w_tiles, per_tok);
  p.nchunks = ceil_div(p.w_tiles, p.w_per_chunk);
  p.grid = p.tok_tiles * p.nchunks;
  // Tokens on M: pairs of CTAs with consecutive token tiles of one vocabulary chunk share each
  // weight box by TMA multicast (halving the weight traffic from L2; clusters of two still
  // cover every SM).
  p.mcast = (!p.swap && p.tok_tiles % 2 == 0) ? 2 : 1;

  if (head) {
    p.u_in_gru = p.swap;
    p.xg = plan_store(M, 3 * Ds, ceil_div(H, 64), sms);
    // small M: hidden half of W1 before the GRU; large M: both halves of W1 after it
    p.ug = plan_store(M, R, p.u_in_gru ? ceil_div(H, 64) : ceil_div(H, 64) + ceil_div(Ds, 64), sms);
    p.gru = dm::gru_plan(B, Ds, sms);
    if (p.gru.smem == 0) return DOMINO_ERR_UNSUPPORTED;
    // Overlap the GRU with the W_lm stream when a deferred-mode vocab CTA and a GRU CTA fit on
    // one SM (228 KB of shared memory, 1 KB reserved per CTA) and every tile of a CTA can keep
    // its own TMEM accumulator until u is ready.
    const int vsm = dm::tc_softmax_deferred_smem(p.bn, p.kmax);
    // The first D tiles of each CTA wait for u; the rest run whole.  Pass 0 streams only the
    // W_lm segment of those D tiles (128 x H bf16 per CTA and tile, about 6.6 TB/s over the
    // grid), so D covers the GRU's expected time (12 us + K steps of 4.5 + 0.5 B us, generous
    // for a GRU sharing its SMs with the stream) in such tile waves, plus one.  A deferred tile
    // never waits for the epilogue, so a larger D costs only TMEM columns ((D+2) x BN <= 512)
    // and a later epilogue; a short estimate costs a wait at the checkpoint, never correctness.
    {
      const double t_seg1_us = 128.0 * H * 2.0 * p.grid / 6.6e6;
      const double t_gru_us = 12.0 + K * (4.5 + 0.5 * B);
      int d = static_cast<int>(std::ceil(t_gru_us / t_seg1_us)) + 1;
      int dmax = p.w_per_chunk < dm::kMaxDefer ? p.w_per_chunk : dm::kMaxDefer;
      if (512 / p.bn - 2 < dmax) dmax = 512 / p.bn - 2;
      p.defer_tiles = d < 1 ? 1 : (d > dmax ? dmax : d);
    }
    p.overlap = p.u_in_gru && vsm > 0 && (p.defer_tiles + 2) * p.bn <= 512 &&
                static_cast<size_t>(vsm) + p.gru.smem + 2048 <= 228 * 1024;
    // With the overlap, chain the whole head: the gather, both projection GEMMs and the GRU
    // each let the next kernel launch early, so that the GRU's CTAs (and with them the
    // vocabulary stream) start while the projections still run.
    p.chain = p.overlap && p.xg.swap && p.ug.swap && dm::tc_store_chained_smem(p.xg.bn) > 0 &&
              dm::tc_store_chained_smem(p.ug.bn) > 0;
    // Fused projections: 8 units per GRU CTA (one MMA n-tile per gate) and every warp's u pairs
    // (rank row, position) within the kernel's shared-memory slots.
    if (p.chain && p.gru.units == 8) {
      const int total_warps = p.gru.gu * p.gru.gb * 8;
      const int groups = total_warps / R > 1 ? total_warps / R : 1;
      const long long pairs = static_cast<long long>(ceil_div(R * groups, total_warps)) * ceil_div(M, groups);
      p.fused = pairs <= dm::kGruMaxUPairs;
    }
  }
  p.tmem_cols = pow2_at_least(p.overlap ? (p.defer_tiles + 2) * p.bn : 2 * p.bn, 32);

  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes);
    return o;
  };
  p.ctrl_bytes = align_up(256 + static_cast<size_t>(B) * 4);
  p.off_ctrl = take(p.ctrl_bytes);
  // control words: status at 0, the GRU's clear barrier at 64, step epoch at 128, the hx range
  // record at 160, merge counters from 256.  Fused projections need no clear before a step (the
  // GRU resets the status and the counters; its state words carry the epoch as a tag, trusted
  // where the range record covers them, and cleared by the GRU itself where it does not); the
  // workspace must only be zero when first used.  Every other plan clears all control words,
  // the range record with them.
  p.clear_bytes = p.fused ? 0 : p.ctrl_bytes;
  if (head) {
    p.off_hx = take(static_cast<size_t>(M) * Ds * 4);
    p.off_E = take(static_cast<size_t>(M) * H * 2);
    p.off_xpart = take(static_cast<size_t>(p.xg.splits) * M * 3 * Ds * 4);
    p.off_upart = take(static_cast<size_t>(p.ug.splits) * M * R * 4);
    p.off_xs = take(static_cast<size_t>(M) * 3 * Ds * 4);
    p.off_S = take(static_cast<size_t>(M) * Ds * 2);
    p.off_u = take(static_cast<size_t>(M) * R * 2);
  }
  p.off_part = take(static_cast<size_t>(M) * p.nchunks * p.rec * 4);
  p.dev_total = off;
  p.off_hid = take(static_cast<size_t>(M) * H * 2);
  p.off_ids = take(static_cast<size_t>(M) * 4);
  p.off_tid = take(static_cast<size_t>(M) * k * 4);
  p.off_tlp = take(static_cast<size_t>(M) * k * 4);
  p.off_tpar = take(static_cast<size_t>(B) * N * 4);
  p.off_ttok = take(static_cast<size_t>(B) * N * 4);
  p.off_tdep = take(static_cast<size_t>(B) * N * 4);
  p.off_tsc = take(static_cast<size_t>(B) * N * 4);
  p.off_ostat = take(4);  // the status copy: the host entry point reads [off_tid, off_ostat + 4) at once
  p.host_total = off;
  return DOMINO_OK;
}

int make_plan(int B, int K, int H, int V, int Ds, int R, int k, int N, bool head, Plan* P) {
  int rc = check_sizes(B, K, H, V, Ds, R, k, N, head);
  if (rc != DOMINO_OK) return rc;
  int sms = 0, major = 0, minor = 0;
  rc = device_sms(&sms, &major, &minor);
  if (rc != DOMINO_OK) return rc;
  if (major != 10 || minor != 3) return DOMINO_ERR_UNSUPPORTED;
  return make_plan_sms(B, K, H, V, Ds, R, k, N, head, sms, P);
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// 2-D bf16 tensor map: `rows` rows of `inner` elements, `stride_elems` apart; boxes of
// 64 x box_rows with 128-byte swizzling; out-of-range elements read as zero.
bool make_map(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t stride_elems,
              uint32_t box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[2] = {inner, rows};
  cuuint64_t strides[1] = {stride_elems * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, estr,
                  CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                  CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Maps for one GEMM: activations X [M, inner] (row stride xs) and weights W [rows_w, inner]
// (row stride ws), in A/B order for the orientation.  With weight multicast (tokens on M) each
// CTA of a cluster loads 1/mcast of the weight box, so that map's box is bn / mcast rows high.
bool gemm_maps(CUtensorMap* a, CUtensorMap* b, bool swap, int bn, const void* X, int M, int inner, int xs,
               const void* W, int rows_w, int ws, int mcast = 1) {
  if (swap) return make_map(a, W, inner, rows_w, ws, 128) && make_map(b, X, inner, M, xs, bn);
  return make_map(a, X, inner, M, xs, 128) && make_map(b, W, inner, rows_w, ws, bn / (mcast > 1 ? mcast : 1));
}

int cuda_rc(cudaError_t e) { return e == cudaSuccess ? DOMINO_OK : DOMINO_ERR_CUDA; }


// ---------------------------------------------------------------- host staging
// Pinned host buffer the host entry point copies a step's outputs into (one copy), grown on
// demand and kept for the process; callers hold g_stage_mu while they use it.
std::mutex g_stage_mu;
uint8_t* g_stage = nullptr;
size_t g_stage_bytes = 0;

void drop_host_graphs();

uint8_t* stage_buffer(size_t bytes) {
  if (bytes <= g_stage_bytes) return g_stage;
  drop_host_graphs();  // their output copies target the buffer that is about to move
  if (g_stage) cudaFreeHost(g_stage);
  g_stage = nullptr;
  g_stage_bytes = 0;
  void* p = nullptr;
  if (cudaHostAlloc(&p, bytes, cudaHostAllocDefault) != cudaSuccess) return nullptr;
  g_stage = static_cast<uint8_t*>(p);
  g_stage_bytes = bytes;
  return g_stage;
}

// ---------------------------------------------------------------- host entry point: graphs
// domino_draft_step_host returns only once its step is done, so a call's launches reach the GPU
// one by one after the previous call came back.  The second call with the same arguments
// captures the whole call (the input copies, the step's kernels, the output copy into the
// staging buffer) into a CUDA graph on a stream of this library; it and every later call with
// those arguments launch that graph on the caller's stream.  The first call runs directly, so
// that every kernel attribute is set outside a capture.  Guarded by g_stage_mu (every host
// entry call holds it); at most kMaxHostGraphs graphs are kept (all are dropped when full, and
// when the staging buffer moves).
struct HostKey {
  const void* hidden;
  const void* ids;
  const void* w_lm;
  domino_head_weights head;
  int hd, B, K, H, V, k, N, dev;
  void* ws;
  size_t ws_bytes;
  const uint8_t* stage;
};

struct HostKeyLess {
  bool operator()(const HostKey& a, const HostKey& b) const { return memcmp(&a, &b, sizeof(HostKey)) < 0; }
};

struct HostGraph {
  int calls = 0;
  bool failed = false;  // capture or instantiation failed once: this key runs directly
  cudaGraphExec_t exec = nullptr;
};

constexpr size_t kMaxHostGraphs = 16;
std::map<HostKey, HostGraph, HostKeyLess> g_host_graphs;
std::map<int, cudaStream_t> g_capture_streams;  // per device

void drop_host_graphs() {
  for (auto& kv : g_host_graphs)
    if (kv.second.exec) cudaGraphExecDestroy(kv.second.exec);
  g_host_graphs.clear();
}

cudaStream_t capture_stream(int dev) {
  auto it = g_capture_streams.find(dev);
  if (it != g_capture_streams.end()) return it->second;
  cudaStream_t cs = nullptr;
  if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) {
    (void)cudaGetLastError();
    return nullptr;
  }
  g_capture_streams[dev] = cs;
  return cs;
}

// ---------------------------------------------------------------- per-kernel timing
struct Timing {
  std::atomic<bool> on{false};  // read by every launch, on any thread; set by begin / end
  int used = 0;
  std::vector<cudaEvent_t> start, stop;
  std::vector<int> kind;
};
Timing g_timing;

// Brackets one launch with an event pair when timing is on; returns the slot or -1.
int timing_open(int kind, cudaStream_t st) {
  Timing& t = g_timing;
  if (!t.on || t.used >= static_cast<int>(t.start.size())) return -1;
  const int i = t.used++;
  t.kind[i] = kind;
  cudaEventRecord(t.start[i], st);
  return i;
}

void timing_close(int slot, cudaStream_t st) {
  if (slot >= 0) cudaEventRecord(g_timing.stop[slot], st);
}

int run_step_launches(const Plan& P, const void* hidden, const int32_t* ids, const void* w_lm,
                      const domino_head_weights* hw, int32_t* topk_ids, float* topk_logp, int32_t* tpar,
                      int32_t* ttok, int32_t* tdep, float* tsc, uint8_t* ws, cudaStream_t st,
                      int32_t* status_out) {
  const int M = P.M, H = P.H, V = P.V, Ds = P.Ds, R = P.R;
  int* status = reinterpret_cast<int*>(ws + P.off_ctrl);
  unsigned* seq_done = reinterpret_cast<unsigned*>(ws + P.off_ctrl + 256);
  if (P.clear_bytes && cudaMemsetAsync(ws + P.off_ctrl, 0, P.clear_bytes, st) != cudaSuccess) return DOMINO_ERR_CUDA;
  uint32_t* epoch = reinterpret_cast<uint32_t*>(ws + P.off_ctrl + 128);

  // an input-projection table replaces the gathered embeddings and the X GEMM
  const float* x_table = P.head ? hw->x_table : nullptr;
  __nv_bfloat16* E = (P.head && !x_table) ? reinterpret_cast<__nv_bfloat16*>(ws + P.off_E) : nullptr;
  uint32_t* hx = P.head ? reinterpret_cast<uint32_t*>(ws + P.off_hx) : nullptr;
  int ts = -1, rc = DOMINO_OK;
  if (!P.fused) {
    dm::GatherParams gp{ids, P.head ? static_cast<const __nv_bfloat16*>(hw->emb) : nullptr, E, hx, M, H, V, Ds, status};
    ts = timing_open(DOMINO_KERNEL_GATHER, st);
    rc = cuda_rc(dm::launch_gather(gp, st));
    timing_close(ts, st);
    if (rc) return rc;
  }

  __nv_bfloat16* u = nullptr;
  if (P.head) {
    float* xpart = reinterpret_cast<float*>(ws + P.off_xpart);
    float* upart = reinterpret_cast<float*>(ws + P.off_upart);
    u = reinterpret_cast<__nv_bfloat16*>(ws + P.off_u);
    // X partials: E [M, H] . W_ih [3Ds, H]^T
    if (!P.fused && !x_table) {
      const dm::TcParams base{};
      TcParams tp = base;
      const StorePlan& g = P.xg;
      CUtensorMap maps[4];
      if (!gemm_maps(&maps[0], &maps[1], g.swap, g.bn, E, M, H, H, hw->w_ih, 3 * Ds, H)) return DOMINO_ERR_CUDA;
      maps[2] = maps[0];
      maps[3] = maps[1];
      tp.nkb1 = g.nkb; tp.nkb2 = 0;
      tp.rows_tok = M; tp.rows_w = 3 * Ds;
      tp.tok_tiles = g.tok_tiles; tp.w_tiles = g.w_tiles;
      tp.splits = g.splits; tp.kb_per_split = g.kb_per_split; tp.total_items = g.total_items;
      tp.w_evict_first = 0;
      tp.tmem_cols = pow2_at_least(2 * g.bn, 32);
      tp.out = xpart; tp.ld_out = 3 * Ds;
      tp.status = status;
      // E comes from the gather: small M chained, and for many tokens a programmatic dependent
      // of the gather
      const bool dep = !P.chain && !g.swap && g.bn == 256;
      tp.pdl_wait = (P.chain || dep) ? 1 : 0;
      ts = timing_open(DOMINO_KERNEL_GRU_INPUT, st);
      rc = cuda_rc(P.chain ? dm::launch_tc_store_chained(g.bn, maps, tp, g.grid, st)
                   : dep   ? dm::launch_tc_store_dependent(maps, tp, g.grid, st)
                           : dm::launch_tc_gemm(dm::kModeStore, g.bn, g.swap, 16, maps, tp, g.grid, st));
      timing_close(ts, st);
      if (rc) return rc;
    }
    __nv_bfloat16* S = reinterpret_cast<__nv_bfloat16*>(ws + P.off_S);
    // W1 GEMM: hidden [M, H] . W1[:, :H]^T (+ S [M, Ds] . W1[:, H:]^T on the large-M path)
    auto w1_gemm = [&](bool both) -> int {
      const dm::TcParams base{};
      TcParams tp = base;
      const StorePlan& g = P.ug;
      CUtensorMap maps[4];
      if (!gemm_maps(&maps[0], &maps[1], g.swap, g.bn, hidden, M, H, H, hw->w1, R, H + Ds)) return DOMINO_ERR_CUDA;
      if (both) {
        const void* w1b = static_cast<const __nv_bfloat16*>(hw->w1) + H;
        if (!gemm_maps(&maps[2], &maps[3], g.swap, g.bn, S, M, Ds, Ds, w1b, R, H + Ds)) return DOMINO_ERR_CUDA;
      } else {
        maps[2] = maps[0];
        maps[3] = maps[1];
      }
      tp.nkb1 = ceil_div(H, 64);
      tp.nkb2 = both ? ceil_div(Ds, 64) : 0;
      tp.rows_tok = M; tp.rows_w = R;
      tp.tok_tiles = g.tok_tiles; tp.w_tiles = g.w_tiles;
      tp.splits = g.splits; tp.kb_per_split = g.kb_per_split; tp.total_items = g.total_items;
      tp.w_evict_first = 0;
      tp.tmem_cols = pow2_at_least(2 * g.bn, 32);
      tp.out = upart; tp.ld_out = R;
      tp.status = status;
      const bool chained = P.chain && !both;
      // many tokens: both halves after the GRU, a programmatic dependent of it (S is its output)
      const bool dep = both && !g.swap && g.bn == 256;
      tp.pdl_wait = chained ? 2 : (dep ? 1 : 0);  // chained: reads nothing the kernel before it
                                                  // (X GEMM or gather) writes; completes after it
      const int slot = timing_open(DOMINO_KERNEL_W1_HIDDEN, st);
      const int r = cuda_rc(chained ? dm::launch_tc_store_chained(g.bn, maps, tp, g.grid, st)
                            : dep   ? dm::launch_tc_store_dependent(maps, tp, g.grid, st)
                                    : dm::launch_tc_gemm(dm::kModeStore, g.bn, g.swap, 16, maps, tp, g.grid, st));
      timing_close(slot, st);
      return r;
    };
    if (P.u_in_gru && !P.fused) {
      rc = w1_gemm(false);
      if (rc) return rc;
    }
    dm::GruParams gr{};
    gr.xpart = xpart; gr.xsplits = P.xg.splits;
    gr.upart = upart; gr.usplits = P.ug.splits;
    gr.w_hh = static_cast<const __nv_bfloat16*>(hw->w_hh);
    gr.b_ih = static_cast<const __nv_bfloat16*>(hw->b_ih);
    gr.b_hh = static_cast<const __nv_bfloat16*>(hw->b_hh);
    gr.w1 = static_cast<const __nv_bfloat16*>(hw->w1);
    gr.b1 = static_cast<const __nv_bfloat16*>(hw->b1);
    gr.B = P.B; gr.K = P.K; gr.H = H; gr.Ds = Ds; gr.R = R;
    gr.units = P.gru.units; gr.gu = P.gru.gu; gr.gb = P.gru.gb; gr.bc = P.gru.bc;
    gr.xs = reinterpret_cast<float*>(ws + P.off_xs);
    gr.hx = hx;
    gr.s_out = P.u_in_gru ? nullptr : S;
    gr.u = P.u_in_gru ? u : nullptr;
    gr.status = status;
    gr.epoch = epoch;
    gr.seq_done = seq_done;
    gr.reset_ctrl = P.fused ? 1 : 0;
    if (P.fused) {
      gr.layout = reinterpret_cast<unsigned long long*>(ws + P.off_ctrl + 160);
      gr.layout_range = dm::hx_range(P.off_hx, P.off_hx + static_cast<size_t>(M) * Ds * 4);
      gr.clear_bar = reinterpret_cast<unsigned long long*>(ws + P.off_ctrl + 64);
    }
    gr.V = V;
    gr.x_table = x_table;
    gr.x_ids = ids;
    if (P.fused) {
      gr.ids = ids;
      gr.emb = static_cast<const __nv_bfloat16*>(hw->emb);
      gr.w_ih = static_cast<const __nv_bfloat16*>(hw->w_ih);
      gr.hidden = static_cast<const __nv_bfloat16*>(hidden);
      gr.V = V;
    }
    ts = timing_open(DOMINO_KERNEL_GRU, st);
    // no vocabulary CTA shares the GRU's SMs unless the two overlap; for many tokens the GRU is
    // a programmatic dependent of the kernel before it (it waits for it before reading)
    rc = cuda_rc(dm::launch_gru(gr, P.gru, st, (P.chain && !P.fused) || !P.u_in_gru, !P.overlap));
    timing_close(ts, st);
    if (rc) return rc;
    if (!P.u_in_gru) {
      rc = w1_gemm(true);
      if (rc) return rc;
      dm::UFinalParams uf{upart, P.ug.splits, M, R, static_cast<const __nv_bfloat16*>(hw->b1), u};
      ts = timing_open(DOMINO_KERNEL_W1_HIDDEN, st);
      rc = cuda_rc(dm::launch_u_finalize(uf, st, true));
      timing_close(ts, st);
      if (rc) return rc;
    }
  }

  // fused vocabulary GEMM with the online softmax / top-k epilogue
  {
    const dm::TcParams base{};
    TcParams tp = base;
    CUtensorMap maps[4];
    if (!gemm_maps(&maps[0], &maps[1], P.swap, P.bn, hidden, M, H, H, w_lm, V, H, P.mcast)) return DOMINO_ERR_CUDA;
    if (P.head) {
      if (!gemm_maps(&maps[2], &maps[3], P.swap, P.bn, u, M, R, R, hw->w2, V, R, P.mcast)) return DOMINO_ERR_CUDA;
    } else {
      maps[2] = maps[0];
      maps[3] = maps[1];
    }
    tp.nkb1 = ceil_div(H, 64);
    tp.nkb2 = P.head ? ceil_div(R, 64) : 0;
    tp.rows_tok = M; tp.rows_w = V;
    tp.tok_tiles = P.tok_tiles; tp.w_tiles = P.w_tiles;
    tp.nchunks = P.nchunks; tp.w_per_chunk = P.w_per_chunk;
    tp.w_evict_first = P.tok_tiles == 1 ? 1 : 0;
    tp.defer = P.overlap ? P.defer_tiles : 0;
    tp.mcast = P.mcast;
    tp.tmem_cols = P.tmem_cols;
    tp.bias = hw ? static_cast<const __nv_bfloat16*>(hw->b2) : nullptr;
    tp.out = reinterpret_cast<float*>(ws + P.off_part);
    tp.status = status;
    // large M on CTA pairs: a programmatic dependent of u_finalize, waiting for it only before
    // the W2 segment (the first tile's W_lm segment streams meanwhile)
    if (P.head && !P.u_in_gru && !P.swap && P.mcast == 2) tp.pdl_wait = 3;
    ts = timing_open(DOMINO_KERNEL_VOCAB, st);
    if (P.overlap)
      rc = cuda_rc(dm::launch_tc_softmax_deferred(P.bn, P.kmax, maps, tp, P.grid, st));
    else
      rc = cuda_rc(dm::launch_tc_gemm(dm::kModeSoftmax, P.bn, P.swap, P.kmax, maps, tp, P.grid, st));
    timing_close(ts, st);
    if (rc) return rc;
  }

  dm::TreeParams tr{};
  tr.partials = reinterpret_cast<const float*>(ws + P.off_part);
  tr.seq_done = seq_done;
  tr.nchunks = P.nchunks;
  tr.kmax = P.kmax;
  tr.B = P.B; tr.K = P.K; tr.k = P.k; tr.N = P.N;
  tr.topk_ids = topk_ids; tr.topk_logp = topk_logp;
  tr.tree_parent = tpar; tr.tree_token = ttok; tr.tree_depth = tdep; tr.tree_score = tsc;
  tr.status = status;
  tr.status_out = status_out;
  tr.epoch = P.head ? epoch : nullptr;
  ts = timing_open(DOMINO_KERNEL_TREE, st);
  rc = cuda_rc(dm::launch_merge_tree(tr, st));
  timing_close(ts, st);
  return rc;
}

// One step.  A launch that fails part-way leaves the step's later kernels (among them the one
// that advances the step epoch) unlaunched; the control words are then zeroed, as in a fresh
// workspace, so the next step neither trusts this one's state words nor counts from its barrier.
int run_step(const Plan& P, const void* hidden, const int32_t* ids, const void* w_lm, const domino_head_weights* hw,
             int32_t* topk_ids, float* topk_logp, int32_t* tpar, int32_t* ttok, int32_t* tdep, float* tsc,
             uint8_t* ws, cudaStream_t st, int32_t* status_out = nullptr) {
  const int rc = run_step_launches(P, hidden, ids, w_lm, hw, topk_ids, topk_logp, tpar, ttok, tdep, tsc, ws, st,
                                   status_out);
  if (rc != DOMINO_OK) {
    (void)cudaGetLastError();
    (void)cudaMemsetAsync(ws + P.off_ctrl, 0, P.ctrl_bytes, st);
  }
  return rc;
}

bool head_active(const domino_head_weights* hw) { return hw != nullptr && hw->w2 != nullptr && hw->R > 0; }

int check_pointers(const void* hidden, const int32_t* ids, const void* w_lm, const domino_head_weights* hw,
                   bool head) {
  if (!hidden || !ids || !w_lm) return DOMINO_ERR_INVALID_ARG;
  if (head && (!hw->emb || !hw->w_ih || !hw->w_hh || !hw->w1 || !hw->w2)) return DOMINO_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(w_lm)) return DOMINO_ERR_UNSUPPORTED;
  if (head && (!aligned16(hw->emb) || !aligned16(hw->w_ih) || !aligned16(hw->w_hh) || !aligned16(hw->w1) ||
               !aligned16(hw->w2) || !aligned16(hw->x_table)))
    return DOMINO_ERR_UNSUPPORTED;
  return DOMINO_OK;
}

}  // namespace

extern "C" {

size_t domino_workspace_bytes(int B, int K, int H, int V, int Ds, int R, int k, int N) {
  Plan P;
  if (make_plan(B, K, H, V, Ds, R, k, N, R > 0, &P) != DOMINO_OK) return 0;
  return P.dev_total;
}

size_t domino_workspace_bytes_host(int B, int K, int H, int V, int Ds, int R, int k, int N) {
  Plan P;
  if (make_plan(B, K, H, V, Ds, R, k, N, R > 0, &P) != DOMINO_OK) return 0;
  return P.host_total;
}

int domino_draft_step(const void* hidden, const int32_t* prefix_ids, const void* w_lm,
                      const domino_head_weights* head, int B, int K, int H, int V, int k, int N,
                      int32_t* topk_ids, float* topk_logp, int32_t* tree_parent, int32_t* tree_token,
                      int32_t* tree_depth, float* tree_score, void* workspace, size_t workspace_bytes,
                      void* stream) {
  const bool hd = head_active(head);
  if (!topk_ids || !topk_logp || !tree_parent || !tree_token || !tree_depth || !workspace)
    return DOMINO_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1)) != 0) return DOMINO_ERR_INVALID_ARG;
  int rc = check_pointers(hidden, prefix_ids, w_lm, head, hd);
  if (rc) return rc;
  Plan P;
  rc = make_plan(B, K, H, V, hd ? head->Ds : 0, hd ? head->R : 0, k, N, hd, &P);
  if (rc) return rc;
  if (workspace_bytes < P.dev_total) return DOMINO_ERR_INVALID_ARG;
  return run_step(P, hidden, prefix_ids, w_lm, head, topk_ids, topk_logp, tree_parent, tree_token, tree_depth,
                  tree_score, static_cast<uint8_t*>(workspace), static_cast<cudaStream_t>(stream));
}

int domino_draft_step_host(const void* hidden_host, const int32_t* prefix_ids_host, const void* w_lm,
                           const domino_head_weights* head, int B, int K, int H, int V, int k, int N,
                           int32_t* topk_ids_host, float* topk_logp_host, int32_t* tree_parent_host,
                           int32_t* tree_token_host, int32_t* tree_depth_host, float* tree_score_host,
                           void* workspace, size_t workspace_bytes, void* stream) {
  const bool hd = head_active(head);
  if (!hidden_host || !prefix_ids_host || !w_lm || !topk_ids_host || !topk_logp_host || !tree_parent_host ||
      !tree_token_host || !tree_depth_host || !workspace)
    return DOMINO_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & (kAlign - 1)) != 0) return DOMINO_ERR_INVALID_ARG;
  Plan P;
  int rc = make_plan(B, K, H, V, hd ? head->Ds : 0, hd ? head->R : 0, k, N, hd, &P);
  if (rc) return rc;
  if (workspace_bytes < P.host_total) return DOMINO_ERR_INVALID_ARG;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t M = P.M;
  void* d_hid = ws + P.off_hid;
  int32_t* d_ids = reinterpret_cast<int32_t*>(ws + P.off_ids);
  rc = check_pointers(d_hid, d_ids, w_lm, head, hd);
  if (rc) return rc;
  int32_t* d_tid = reinterpret_cast<int32_t*>(ws + P.off_tid);
  float* d_tlp = reinterpret_cast<float*>(ws + P.off_tlp);
  int32_t* d_par = reinterpret_cast<int32_t*>(ws + P.off_tpar);
  int32_t* d_tok = reinterpret_cast<int32_t*>(ws + P.off_ttok);
  int32_t* d_dep = reinterpret_cast<int32_t*>(ws + P.off_tdep);
  float* d_sc = reinterpret_cast<float*>(ws + P.off_tsc);
  int32_t* d_ostat = reinterpret_cast<int32_t*>(ws + P.off_ostat);
  // every output and the status in one copy, through a pinned staging buffer of this library
  const size_t lo = P.off_tid, bytes = P.off_ostat + 4 - lo;
  std::lock_guard<std::mutex> lock(g_stage_mu);
  uint8_t* h = stage_buffer(bytes);
  if (!h) return DOMINO_ERR_CUDA;
  // the whole call on stream s: input copies, the step, the output copy
  auto enqueue = [&](cudaStream_t s) -> int {
    if (cudaMemcpyAsync(d_hid, hidden_host, M * H * 2, cudaMemcpyHostToDevice, s) != cudaSuccess) return DOMINO_ERR_CUDA;
    if (cudaMemcpyAsync(d_ids, prefix_ids_host, M * 4, cudaMemcpyHostToDevice, s) != cudaSuccess) return DOMINO_ERR_CUDA;
    const int r = run_step(P, d_hid, d_ids, w_lm, head, d_tid, d_tlp, d_par, d_tok, d_dep, d_sc, ws, s, d_ostat);
    if (r) return r;
    return cuda_rc(cudaMemcpyAsync(h, ws + lo, bytes, cudaMemcpyDeviceToHost, s));
  };
  cudaGraphExec_t exec = nullptr;
  int dev = 0;
  if (!g_timing.on && cudaGetDevice(&dev) == cudaSuccess) {
    HostKey key;
    memset(&key, 0, sizeof(key));  // padding included: keys compare as bytes
    key.hidden = hidden_host;
    key.ids = prefix_ids_host;
    key.w_lm = w_lm;
    if (hd) key.head = *head;
    key.hd = hd ? 1 : 0;
    key.B = B; key.K = K; key.H = H; key.V = V; key.k = k; key.N = N; key.dev = dev;
    key.ws = workspace;
    key.ws_bytes = workspace_bytes;
    key.stage = h;
    if (g_host_graphs.size() >= kMaxHostGraphs && g_host_graphs.find(key) == g_host_graphs.end()) drop_host_graphs();
    HostGraph& g = g_host_graphs[key];
    if (!g.exec && !g.failed && g.calls >= 1) {
      // capture on this library's stream (the caller's may be the legacy default stream, which
      // cannot be captured); a capture that fails leaves this key on the direct path
      cudaStream_t cs = capture_stream(dev);
      cudaGraph_t graph = nullptr;
      g.failed = true;
      if (cs && cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) == cudaSuccess) {
        const int r = enqueue(cs);
        const cudaError_t e = cudaStreamEndCapture(cs, &graph);
        if (r == DOMINO_OK && e == cudaSuccess && graph &&
            cudaGraphInstantiate(&g.exec, graph, 0) == cudaSuccess)
          g.failed = false;
        if (graph) cudaGraphDestroy(graph);
      }
      if (g.failed) {  // nothing captured ran: the workspace is as the last call left it
        g.exec = nullptr;
        (void)cudaGetLastError();
      }
    }
    ++g.calls;
    exec = g.exec;
  }
  if (exec) {
    if (cudaGraphLaunch(exec, st) != cudaSuccess) return DOMINO_ERR_CUDA;
  } else {
    rc = enqueue(st);
    if (rc) return rc;
  }
  if (cudaStreamSynchronize(st) != cudaSuccess) return DOMINO_ERR_CUDA;
  const size_t BN = static_cast<size_t>(P.B) * N;
  memcpy(topk_ids_host, h + (P.off_tid - lo), M * k * 4);
  memcpy(topk_logp_host, h + (P.off_tlp - lo), M * k * 4);
  memcpy(tree_parent_host, h + (P.off_tpar - lo), BN * 4);
  memcpy(tree_token_host, h + (P.off_ttok - lo), BN * 4);
  memcpy(tree_depth_host, h + (P.off_tdep - lo), BN * 4);
  if (tree_score_host) memcpy(tree_score_host, h + (P.off_tsc - lo), BN * 4);
  int32_t status = 0;
  memcpy(&status, h + (P.off_ostat - lo), 4);
  return status;
}

int domino_check_status(const void* workspace, void* stream) {
  if (!workspace) return DOMINO_ERR_INVALID_ARG;
  int h = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(&h, workspace, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return DOMINO_ERR_CUDA;
  return h;
}

const char* domino_status_string(int status) {
  switch (status) {
    case DOMINO_OK: return "DOMINO_OK";
    case DOMINO_ERR_INVALID_ARG: return "DOMINO_ERR_INVALID_ARG";
    case DOMINO_ERR_UNSUPPORTED: return "DOMINO_ERR_UNSUPPORTED";
    case DOMINO_ERR_CUDA: return "DOMINO_ERR_CUDA";
    case DOMINO_ERR_TIMEOUT: return "DOMINO_ERR_TIMEOUT";
    case DOMINO_ERR_BAD_TOKEN: return "DOMINO_ERR_BAD_TOKEN";
    default: return "DOMINO_ERR_UNKNOWN";
  }
}

int domino_abi_version(void) { return DOMINO_ABI_VERSION; }

int domino_debug_hold(int what, int gru_cta, int step) {
  if (what == DOMINO_HOLD_OFF) return cuda_rc(dm::arm_gru_hold(dm::kHoldOff, -1, -1));
  if (what != DOMINO_HOLD_STATE && what != DOMINO_HOLD_CLEAR_BARRIER) return DOMINO_ERR_INVALID_ARG;
  if (gru_cta < 0 || (what == DOMINO_HOLD_STATE && (step < 0 || step >= kMaxK))) return DOMINO_ERR_INVALID_ARG;
  const int kind = what == DOMINO_HOLD_STATE ? dm::kHoldPublish : dm::kHoldClearBarrier;
  return cuda_rc(dm::arm_gru_hold(kind, gru_cta, what == DOMINO_HOLD_STATE ? step : -1));
}

int domino_timing_begin(int max_launches) {
  if (max_launches <= 0) return DOMINO_ERR_INVALID_ARG;
  Timing& t = g_timing;
  while (static_cast<int>(t.start.size()) < max_launches) {
    cudaEvent_t a, b;
    if (cudaEventCreate(&a) != cudaSuccess) return DOMINO_ERR_CUDA;
    if (cudaEventCreate(&b) != cudaSuccess) return DOMINO_ERR_CUDA;
    t.start.push_back(a);
    t.stop.push_back(b);
    t.kind.push_back(0);
  }
  t.used = 0;
  t.on = true;
  return DOMINO_OK;
}

int domino_timing_end(float* total_ms, int* launches, int nkinds) {
  Timing& t = g_timing;
  t.on = false;
  if (nkinds < 0 || (nkinds > 0 && (!total_ms || !launches))) return DOMINO_ERR_INVALID_ARG;
  for (int i = 0; i < nkinds; ++i) {
    total_ms[i] = 0.f;
    launches[i] = 0;
  }
  for (int i = 0; i < t.used; ++i) {
    if (cudaEventSynchronize(t.stop[i]) != cudaSuccess) return DOMINO_ERR_CUDA;
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, t.start[i], t.stop[i]) != cudaSuccess) return DOMINO_ERR_CUDA;
    if (t.kind[i] < nkinds) {
      total_ms[t.kind[i]] += ms;
      launches[t.kind[i]] += 1;
    }
  }
  t.used = 0;
  return DOMINO_OK;
}

int domino_verify_tree_greedy(const float* target_logits, const int32_t* tree_parent, const int32_t* tree_token,
                              int B, int N, int V, int32_t* row_argmax, int32_t* accepted_nodes,
                              int32_t* accepted_count, int32_t* bonus_token, void* stream) {
  if (B < 1 || N < 0 || V < 1 || N > (1 << 20)) return DOMINO_ERR_INVALID_ARG;
  if (static_cast<long long>(B) * (N + 1) > 0x7fffffffLL) return DOMINO_ERR_INVALID_ARG;
  if (!target_logits || !row_argmax || !accepted_count || !bonus_token) return DOMINO_ERR_INVALID_ARG;
  if (N > 0 && (!tree_parent || !tree_token || !accepted_nodes)) return DOMINO_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int ts = timing_open(DOMINO_KERNEL_VERIFY, st);
  const int rc = cuda_rc(dm::launch_verify_greedy(target_logits, tree_parent, tree_token, B, N, V, row_argmax,
                                                  accepted_nodes, accepted_count, bonus_token, st));
  timing_close(ts, st);
  return rc;
}

int domino_verify_tree_sample(const float* target_logits, const int32_t* tree_parent, const int32_t* tree_token,
                              const float* uniforms, float temperature, int B, int N, int V, int32_t* row_sample,
                              int32_t* accepted_nodes, int32_t* accepted_count, int32_t* bonus_token, void* stream) {
  if (B < 1 || N < 0 || V < 1 || N > (1 << 20)) return DOMINO_ERR_INVALID_ARG;
  if (static_cast<long long>(B) * (N + 1) > 0x7fffffffLL) return DOMINO_ERR_INVALID_ARG;
  if (!target_logits || !uniforms || !row_sample || !accepted_count || !bonus_token) return DOMINO_ERR_INVALID_ARG;
  if (N > 0 && (!tree_parent || !tree_token || !accepted_nodes)) return DOMINO_ERR_INVALID_ARG;
  const float inv_t = 1.0f / temperature;
  if (!(temperature > 0.f) || !std::isfinite(temperature) || !std::isfinite(inv_t)) return DOMINO_ERR_INVALID_ARG;
  if (((V + 7) / 8 + 3) / 4 * 4 > dm::kMaxSampleSlice) return DOMINO_ERR_UNSUPPORTED;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int ts = timing_open(DOMINO_KERNEL_VERIFY, st);
  const int rc = cuda_rc(dm::launch_verify_sample(target_logits, tree_parent, tree_token, uniforms, B, N, V, inv_t,
                                                  row_sample, accepted_nodes, accepted_count, bonus_token, st));
  timing_close(ts, st);
  return rc;
}

// ---------------------------------------------------------------- input-projection table
namespace {
__device__ int g_table_status;  // device status of domino_build_input_table's GEMM
std::mutex g_table_mu;          // one build at a time uses it
}  // namespace

size_t domino_input_table_bytes(int V, int Ds) {
  if (V <= 0 || Ds <= 0) return 0;
  return static_cast<size_t>(V) * 3 * Ds * sizeof(float);
}

int domino_build_input_table(const void* emb, const void* w_ih, int V, int H, int Ds, float* table, void* stream) {
  if (!emb || !w_ih || !table || V <= 0 || H <= 0 || Ds <= 0) return DOMINO_ERR_INVALID_ARG;
  if (H % 8 != 0 || Ds % 8 != 0 || Ds > kMaxDs || V >= kMaxV) return DOMINO_ERR_UNSUPPORTED;
  if (!aligned16(emb) || !aligned16(w_ih) || !aligned16(table)) return DOMINO_ERR_UNSUPPORTED;
  int sms = 0, major = 0, minor = 0;
  int rc = device_sms(&sms, &major, &minor);
  if (rc != DOMINO_OK) return rc;
  if (major != 10 || minor != 3) return DOMINO_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_table_mu);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int* status = nullptr;
  if (cudaGetSymbolAddress(reinterpret_cast<void**>(&status), g_table_status) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (cudaMemsetAsync(status, 0, sizeof(int), st) != cudaSuccess) return DOMINO_ERR_CUDA;
  // emb [V, H] . W_ih [3 Ds, H]^T, every token a GEMM row, one split (finished sums)
  StorePlan g = plan_store(V, 3 * Ds, ceil_div(H, 64), sms);
  g.splits = 1;
  g.kb_per_split = g.nkb;
  g.total_items = g.tok_tiles * g.w_tiles;
  g.grid = g.total_items < sms ? g.total_items : sms;
  CUtensorMap maps[4];
  if (!gemm_maps(&maps[0], &maps[1], g.swap, g.bn, emb, V, H, H, w_ih, 3 * Ds, H)) return DOMINO_ERR_CUDA;
  maps[2] = maps[0];
  maps[3] = maps[1];
  const dm::TcParams b0{};
  TcParams tp = b0;
  tp.nkb1 = g.nkb; tp.nkb2 = 0;
  tp.rows_tok = V; tp.rows_w = 3 * Ds;
  tp.tok_tiles = g.tok_tiles; tp.w_tiles = g.w_tiles;
  tp.splits = 1; tp.kb_per_split = g.kb_per_split; tp.total_items = g.total_items;
  tp.w_evict_first = 0;
  tp.tmem_cols = pow2_at_least(2 * g.bn, 32);
  tp.out = table; tp.ld_out = 3 * Ds;
  tp.status = status;
  rc = cuda_rc(dm::launch_tc_gemm(dm::kModeStore, g.bn, g.swap, 16, maps, tp, g.grid, st));
  if (rc) return rc;
  int h = 0;
  if (cudaMemcpyAsync(&h, status, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return DOMINO_ERR_CUDA;
  return h;
}

// ---------------------------------------------------------------- sequential rollout (greedy, sampled)
namespace {
struct RollPlan {
  int B, K, H, V, Ds, R, M, grid;
  bool head;
  StorePlan g;  // base-logit GEMM, no split
  size_t off_h, off_u, off_part, off_lg, off_base, off_uh, off_gh, clear_bytes, total;
};

int make_roll_plan(int B, int K, int H, int V, int Ds, int R, bool head, RollPlan* P) {
  if (B < 1 || B > dm::kRollMaxB || K < 1 || H < 8 || (H & 7) || V < 1) return DOMINO_ERR_INVALID_ARG;
  // head on: a W2 row must fit one 16 KB stage of the rollout's ring
  if (head && (Ds < 8 || (Ds & 7) || R < 8 || (R & 7) || R > 8192)) return DOMINO_ERR_INVALID_ARG;
  if (static_cast<long long>(B) * K * V > (1LL << 33)) return DOMINO_ERR_UNSUPPORTED;
  if (V > static_cast<int>(dm::kGreedyIdMask)) return DOMINO_ERR_UNSUPPORTED;  // token ids below 2^22
  int sms = 0, major = 0, minor = 0;
  int rc = device_sms(&sms, &major, &minor);
  if (rc != DOMINO_OK) return rc;
  if (major != 10 || minor != 3) return DOMINO_ERR_UNSUPPORTED;
  RollPlan& p = *P;
  p.B = B; p.K = K; p.H = H; p.V = V; p.head = head;
  p.Ds = head ? Ds : 0;
  p.R = head ? R : 0;
  p.M = B * K;
  p.grid = sms;  // one CTA per SM, all resident (cooperative launch)
  // the ring, u and the CTA's rows of base logits must fit one CTA's shared memory
  if (dm::rollout_smem_bytes(B, V, p.R, head, sms) > dm::kRollMaxSmem) return DOMINO_ERR_INVALID_ARG;
  p.g = plan_store(p.M, V, ceil_div(H, 64), sms);
  // one split: the GEMM writes finished logits
  p.g.splits = 1;
  p.g.kb_per_split = p.g.nkb;
  p.g.total_items = p.g.tok_tiles * p.g.w_tiles;
  p.g.grid = p.g.total_items < sms ? p.g.total_items : sms;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off = align_up(off + bytes);
    return o;
  };
  // status (offset 0, as for domino_check_status), the grid barrier counter (64), the u-row
  // counter (128), the count of warps done with uh (192), the greedy argmax keys (256)
  take(512);
  p.off_h = take(static_cast<size_t>(2) * B * (p.Ds > 0 ? p.Ds : 1) * 4);
  p.clear_bytes = off;
  p.off_u = take(static_cast<size_t>(B) * (p.R > 0 ? p.R : 1) * 4);
  // greedy and race: every step's, per warp (the log-probabilities are merged at the end);
  // inverse-CDF sampled: two, by step parity, per CTA
  p.off_part = take(static_cast<size_t>(K > 2 ? K : 2) * p.grid * dm::kRollComputeWarps * dm::kRollMaxB * 16);
  p.off_lg = take(static_cast<size_t>(2) * B * V * 4);  // inverse-CDF sampling: final logits, by step parity
  p.off_base = take(static_cast<size_t>(p.M) * V * 4);
  p.off_uh = take(static_cast<size_t>(p.M) * (p.R > 0 ? p.R : 1) * 4);  // hidden . W1[:, :H]^T
  p.off_gh = take(static_cast<size_t>(2) * B * 3 * (p.Ds > 0 ? p.Ds : 1) * 4);  // W_hh h_j, by step parity
  p.total = off;
  return DOMINO_OK;
}
}  // namespace

size_t domino_rollout_workspace_bytes(int B, int K, int H, int V, int Ds, int R) {
  RollPlan P;
  if (make_roll_plan(B, K, H, V, Ds, R, R > 0, &P) != DOMINO_OK) return 0;
  return P.total;
}

namespace {
// The greedy (uniforms NULL, race false), the inverse-CDF sampled (uniforms) and the seeded
// exponential-race sampled (race) rollout.
int rollout_entry(const void* hidden, const int32_t* anchors, const float* uniforms, bool race, uint64_t seed,
                  const void* w_lm, const domino_head_weights* head, int B, int K, int H, int V, int32_t* tokens,
                  float* logp, void* workspace, size_t workspace_bytes, void* stream) {
  const bool hd = head_active(head);
  if (!hidden || !anchors || !w_lm || !tokens || !logp || !workspace) return DOMINO_ERR_INVALID_ARG;
  if (hd && (!head->emb || !head->w_ih || !head->w_hh || !head->w1)) return DOMINO_ERR_INVALID_ARG;
  if (!aligned16(hidden) || !aligned16(w_lm)) return DOMINO_ERR_INVALID_ARG;
  if (hd && (!aligned16(head->w2) || !aligned16(head->w1) || !aligned16(head->w_ih) || !aligned16(head->w_hh) ||
             !aligned16(head->emb) || !aligned16(head->x_table)))  // x_table: NULL passes
    return DOMINO_ERR_INVALID_ARG;
  RollPlan P;
  int rc = make_roll_plan(B, K, H, V, hd ? head->Ds : 0, hd ? head->R : 0, hd, &P);
  if (rc) return rc;
  if (workspace_bytes < P.total) return DOMINO_ERR_INVALID_ARG;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  if (cudaMemsetAsync(ws, 0, P.clear_bytes, st) != cudaSuccess) return DOMINO_ERR_CUDA;
  int* status = reinterpret_cast<int*>(ws);
  float* base = reinterpret_cast<float*>(ws + P.off_base);
  // base logits W_lm hidden_j for every position (tensor cores, fp32 out)
  {
    const dm::TcParams b0{};
    TcParams tp = b0;
    const StorePlan& g = P.g;
    CUtensorMap maps[4];
    if (!gemm_maps(&maps[0], &maps[1], g.swap, g.bn, hidden, P.M, H, H, w_lm, V, H)) return DOMINO_ERR_CUDA;
    maps[2] = maps[0];
    maps[3] = maps[1];
    tp.nkb1 = g.nkb; tp.nkb2 = 0;
    tp.rows_tok = P.M; tp.rows_w = V;
    tp.tok_tiles = g.tok_tiles; tp.w_tiles = g.w_tiles;
    tp.splits = 1; tp.kb_per_split = g.kb_per_split; tp.total_items = g.total_items;
    tp.w_evict_first = 1;
    tp.tmem_cols = pow2_at_least(2 * g.bn, 32);
    tp.out = base; tp.ld_out = V;
    tp.status = status;
    const int ts = timing_open(DOMINO_KERNEL_ROLLOUT_BASE, st);
    rc = cuda_rc(dm::launch_tc_gemm(dm::kModeStore, g.bn, g.swap, 16, maps, tp, g.grid, st));
    timing_close(ts, st);
    if (rc) return rc;
  }
  dm::RolloutParams rp{};
  rp.hidden = static_cast<const __nv_bfloat16*>(hidden);
  rp.anchors = anchors;
  if (hd) {
    rp.emb = static_cast<const __nv_bfloat16*>(head->emb);
    rp.w_ih = static_cast<const __nv_bfloat16*>(head->w_ih);
    rp.w_hh = static_cast<const __nv_bfloat16*>(head->w_hh);
    rp.b_ih = static_cast<const __nv_bfloat16*>(head->b_ih);
    rp.b_hh = static_cast<const __nv_bfloat16*>(head->b_hh);
    rp.w1 = static_cast<const __nv_bfloat16*>(head->w1);
    rp.b1 = static_cast<const __nv_bfloat16*>(head->b1);
    rp.w2 = static_cast<const __nv_bfloat16*>(head->w2);
    rp.x_table = head->x_table;
    rp.uh = reinterpret_cast<float*>(ws + P.off_uh);
    rp.gh = reinterpret_cast<float*>(ws + P.off_gh);
  }
  rp.b2 = head ? static_cast<const __nv_bfloat16*>(head->b2) : nullptr;
  rp.head = hd ? 1 : 0;
  rp.B = B; rp.K = K; rp.H = H; rp.V = V; rp.Ds = P.Ds; rp.R = P.R;
  rp.base = base;
  rp.h = reinterpret_cast<float*>(ws + P.off_h);
  rp.u = reinterpret_cast<float*>(ws + P.off_u);
  rp.partials = reinterpret_cast<float*>(ws + P.off_part);
  rp.barrier = reinterpret_cast<unsigned*>(ws + 64);
  rp.ucount = reinterpret_cast<unsigned*>(ws + 128);  // cleared with the status and the barrier
  rp.uhcount = reinterpret_cast<unsigned*>(ws + 192);
  // greedy and race: the (perturbed) argmax keys of the sequences (cleared with them)
  rp.best = uniforms ? nullptr : reinterpret_cast<unsigned long long*>(ws + 256);
  rp.race = race ? 1 : 0;
  rp.seed = seed;
  rp.tokens = tokens;
  rp.logp = logp;
  rp.status = status;
  rp.uniforms = uniforms;
  rp.lg = reinterpret_cast<float*>(ws + P.off_lg);
  // W2 as 64 x 128 swizzled tiles, for phase C on the tensor cores (r a multiple of 64 up to 256)
  CUtensorMap tm_w2;
  const bool have_tm = hd && P.R % 64 == 0 && P.R <= 256 && make_map(&tm_w2, head->w2, P.R, V, P.R, 128);
  const int ts = timing_open(DOMINO_KERNEL_ROLLOUT, st);
  rc = cuda_rc(dm::launch_rollout(rp, P.grid, st, have_tm ? &tm_w2 : nullptr));
  timing_close(ts, st);
  return rc;
}
}  // namespace

int domino_rollout_greedy(const void* hidden, const int32_t* anchors, const void* w_lm,
                          const domino_head_weights* head, int B, int K, int H, int V, int32_t* tokens,
                          float* logp, void* workspace, size_t workspace_bytes, void* stream) {
  return rollout_entry(hidden, anchors, nullptr, false, 0, w_lm, head, B, K, H, V, tokens, logp, workspace,
                       workspace_bytes, stream);
}

int domino_rollout_sample(const void* hidden, const int32_t* anchors, const float* uniforms, const void* w_lm,
                          const domino_head_weights* head, int B, int K, int H, int V, int32_t* tokens,
                          float* logp, void* workspace, size_t workspace_bytes, void* stream) {
  if (!uniforms || (reinterpret_cast<uintptr_t>(uniforms) & 3u) != 0) return DOMINO_ERR_INVALID_ARG;
  return rollout_entry(hidden, anchors, uniforms, false, 0, w_lm, head, B, K, H, V, tokens, logp, workspace,
                       workspace_bytes, stream);
}

int domino_rollout_sample_gumbel(const void* hidden, const int32_t* anchors, uint64_t seed, const void* w_lm,
                                 const domino_head_weights* head, int B, int K, int H, int V, int32_t* tokens,
                                 float* logp, void* workspace, size_t workspace_bytes, void* stream) {
  return rollout_entry(hidden, anchors, nullptr, true, seed, w_lm, head, B, K, H, V, tokens, logp, workspace,
                       workspace_bytes, stream);
}

int domino_launches_per_step(int B, int K, int H, int V, int Ds, int R, int k, int N) {
  const bool head = R > 0;
  if (check_sizes(B, K, H, V, Ds, R, k, N, head) != DOMINO_OK) return -1;
  if (!head) return 3;  // gather (id check), vocab GEMM, merge + tree
  // the plan of this device, or of a 152-SM GB300 when none is visible
  int sms = 0, major = 0, minor = 0;
  if (device_sms(&sms, &major, &minor) != DOMINO_OK || sms <= 0) sms = 152;
  Plan P;
  if (make_plan_sms(B, K, H, V, Ds, R, k, N, head, sms, &P) != DOMINO_OK) return -1;
  // fused small M: GRU (+ its projections and u), vocab GEMM, merge + tree; other small M:
  // gather, X GEMM, W1-hidden GEMM, GRU (+u), vocab GEMM, merge + tree; large M: gather, X GEMM,
  // GRU, W1 GEMM, u finalize, vocab GEMM, merge + tree
  if (P.fused) return 3;
  return P.u_in_gru ? 6 : 7;
}

int domino_launches_per_step_table(int B, int K, int H, int V, int Ds, int R, int k, int N) {
  const int n = domino_launches_per_step(B, K, H, V, Ds, R, k, N);
  if (n < 0 || R <= 0) return n;
  // the table replaces the X GEMM (the fused path has none)
  return n == 3 ? 3 : n - 1;
}

}  // extern "C"

// ---------------------------------------------------------------- static-scratch entry point
// Scratch of domino_draft_step_static_scratch, for callers that cannot allocate device memory.
// Host code only sees a stand-in for this symbol; its device address comes from
// cudaGetSymbolAddress, looked up once per device with that device current.
static __device__ __align__(256) unsigned char g_static_scratch[DOMINO_STATIC_SCRATCH_BYTES];

namespace {

constexpr int kMaxScratchDevices = 256;
std::mutex g_static_scratch_mu;
void* g_static_scratch_addr[kMaxScratchDevices] = {};

int static_scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return DOMINO_ERR_CUDA;
  if (dev < 0 || dev >= kMaxScratchDevices) return DOMINO_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_static_scratch_mu);
  if (g_static_scratch_addr[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || p == nullptr) return DOMINO_ERR_CUDA;
    g_static_scratch_addr[dev] = p;
  }
  *out = g_static_scratch_addr[dev];
  return DOMINO_OK;
}

}  // namespace

extern "C" int domino_draft_step_static_scratch(const void* hidden, const int32_t* prefix_ids, const void* w_lm,
                                                const domino_head_weights* head, int B, int K, int H, int V, int k,
                                                int N, int32_t* topk_ids, float* topk_logp, int32_t* tree_parent,
                                                int32_t* tree_token, int32_t* tree_depth, float* tree_score,
                                                int32_t* device_status, void* stream) {
  const bool hd = head_active(head);
  if (!topk_ids || !topk_logp || !tree_parent || !tree_token || !tree_depth) return DOMINO_ERR_INVALID_ARG;
  int rc = check_pointers(hidden, prefix_ids, w_lm, head, hd);
  if (rc) return rc;
  Plan P;
  rc = make_plan(B, K, H, V, hd ? head->Ds : 0, hd ? head->R : 0, k, N, hd, &P);
  if (rc) return rc;
  if (P.dev_total > DOMINO_STATIC_SCRATCH_BYTES) return DOMINO_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  rc = static_scratch_address(&scratch);
  if (rc) return rc;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // run_step clears the status word and the counters at the start of the scratch itself
  rc = run_step(P, hidden, prefix_ids, w_lm, head, topk_ids, topk_logp, tree_parent, tree_token, tree_depth,
                tree_score, static_cast<uint8_t*>(scratch), st);
  if (rc) return rc;
  if (device_status != nullptr &&
      cudaMemcpyAsync(device_status, static_cast<uint8_t*>(scratch) + P.off_ctrl, sizeof(int32_t),
                      cudaMemcpyDeviceToDevice, st) != cudaSuccess)
    return DOMINO_ERR_CUDA;
  return DOMINO_OK;
}
