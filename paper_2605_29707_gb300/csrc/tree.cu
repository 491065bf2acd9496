// tree.cu -- merge of the per-CTA softmax partials into log-probabilities and top-k lists,
// then the best-first draft tree (the "Tree" cost of the paper's Fig. 1).
//
// Merge: one CTA per draft row (sequence b, position j).  Thread c reads chunk c's record
// (running max, sum of exp, the head of its top-KMAX list; field-major, so the loads are
// coalesced).  The CTA reduces lse = max + log(sum); the k best (value desc, id asc) tokens
// come from a bitonic merge of the chunks' sorted lists, first across the lanes of each warp
// (butterfly), then across the warps.  logp = logit - lse.
// Tree: the CTA that merges the last row of a sequence (atomic counter) selects N nodes
// best-first with one warp.  The frontier is every child (from its position's top-k list) of
// the anchor or of an already selected node that is not selected yet; the next node is the
// frontier entry with the greatest (score, lower token id, lower parent index).  Each expanded
// node ("slot") caches its best remaining child; after a pop only the popped slot and the new
// node need a new best child.  A slot's children have non-increasing scores (its position's
// sorted log-probs plus one parent score), so that child is the first unselected entry unless
// a later unselected entry has exactly the same score and a lower token; every lane computes
// it the same way, and one ballot finds such ties.
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"
#include "topk.cuh"

#ifndef DOMINO_TREE_PDL
#define DOMINO_TREE_PDL 1  // launch the merge kernel as a programmatic dependent of the vocab GEMM
#endif

namespace dm {

// Threads per merge CTA: 256, or 64 when a row has at most 64 chunk records and lists of at most
// 16 entries (tokens-on-M launches, where the rows are many and 256-thread CTAs at their register
// use would need several waves).
constexpr int kMergeThreadsWide = 256;
constexpr int kMergeThreadsNarrow = 64;
constexpr int kMaxK = 64;
constexpr int kMaxTopk = 32;
constexpr int kMaxN = 256;

__device__ __forceinline__ void warp_argmax2(uint32_t hi, uint32_t lo, uint32_t& mhi, uint32_t& mlo, int& src) {
  mhi = __reduce_max_sync(0xffffffffu, hi);
  mlo = __reduce_max_sync(0xffffffffu, hi == mhi ? lo : 0u);
  const unsigned ball = __ballot_sync(0xffffffffu, hi == mhi && lo == mlo);
  src = __ffs(ball) - 1;
}

// Butterfly over lanes l ^ o for o = span/2 .. 1: every lane of each span-wide group ends with
// the best KK entries of the group's lists.
template <int KK>
__device__ __forceinline__ void butterfly_lists(float (&v)[KK], int (&id)[KK], int span) {
  for (int o = span >> 1; o; o >>= 1) {
    float w[KK];
    int iw[KK];
#pragma unroll
    for (int q = 0; q < KK; ++q) {
      w[q] = __shfl_xor_sync(0xffffffffu, v[q], o);
      iw[q] = __shfl_xor_sync(0xffffffffu, id[q], o);
    }
    merge_lists<KK>(v, id, w, iw);
  }
}

__device__ __forceinline__ void lse_merge(float& mx, float& se, float om, float os) {
  const float nm = fmaxf(mx, om);
  if (nm == -INFINITY) return;
  se = (mx == -INFINITY ? 0.f : se * __expf(mx - nm)) + (om == -INFINITY ? 0.f : os * __expf(om - nm));
  mx = nm;
}

// Tree slots.  Slot 0 is the anchor, slot i + 1 the i-th selected node.  Slot s belongs to
// lane s % 32 of the tree warp: slots 0..31 live in that lane's registers, later ones in these
// arrays, which only the owner lane reads and writes.
struct TreeSlots {
  float score[kMaxN + 1];
  int depth[kMaxN + 1];
  unsigned mask[kMaxN + 1];  // children already selected (bit j: entry j of the top-k list)
  unsigned hi[kMaxN + 1];    // cached best child: f32_ord(score), 0 when the slot has none left
  unsigned lo[kMaxN + 1];    // (0x3FFFFF - token) << 10 | (0x3FF - slot): lower token, then slot
  int j[kMaxN + 1];          // the cached child's index in its position's top-k list
  int parent[kMaxN + 1];
  int token[kMaxN + 1];
};

struct SlotState {
  float score;
  int depth;
  unsigned mask;
  uint32_t hi, lo;
  int j, parent, token;
};

__device__ __forceinline__ void slot_put(TreeSlots& S, SlotState& reg, int slot, const SlotState& v) {
  if (slot < 32) {
    reg = v;
  } else {
    S.score[slot] = v.score;
    S.depth[slot] = v.depth;
    S.mask[slot] = v.mask;
    S.hi[slot] = v.hi;
    S.lo[slot] = v.lo;
    S.j[slot] = v.j;
    S.parent[slot] = v.parent;
    S.token[slot] = v.token;
  }
}

__device__ __forceinline__ SlotState slot_get(const TreeSlots& S, const SlotState& reg, int slot) {
  if (slot < 32) return reg;
  SlotState v;
  v.score = S.score[slot];
  v.depth = S.depth[slot];
  v.mask = S.mask[slot];
  v.hi = S.hi[slot];
  v.lo = S.lo[slot];
  v.j = S.j[slot];
  v.parent = S.parent[slot];
  v.token = S.token[slot];
  return v;
}

// Cached best child of a slot from its first unselected entry j0 (score s0) and the entries
// that tie it (bit mask `ties`): the lowest token among them.  (0, 0) when j0 < 0.
__device__ __forceinline__ void child_key(int j0, float s0, unsigned ties, const int* row_ids, int slot,
                                          uint32_t& hi, uint32_t& lo, int& jb) {
  hi = 0u;
  lo = 0u;
  jb = 0;
  if (j0 < 0) return;
  int tb = row_ids[j0];
  jb = j0;
  for (unsigned t = ties; t; t &= t - 1u) {  // rare: an exact tie in fp32
    const int j = __ffs(t) - 1;
    const int tt = row_ids[j];
    if (tt < tb) { tb = tt; jb = j; }
  }
  hi = f32_ord(s0);
  lo = ((0x3FFFFFu - static_cast<unsigned>(tb)) << 10) | (0x3FFu - static_cast<unsigned>(slot));
}

// Best remaining children of two slots a and b (available-entry masks av*, 0 for none; rows
// r* of the top-k lists, clamped to a loaded row; parent scores b*), identical on every lane.
// The tie test runs one entry per lane: half a warp per slot when k <= 16.
__device__ __forceinline__ void best_children(const float* lp, const int* ids, int k, int lane, int ra, float ba,
                                              unsigned ava, int sa, int rb, float bb, unsigned avb, int sb,
                                              uint32_t& ha, uint32_t& la, int& ja, uint32_t& hb, uint32_t& lb,
                                              int& jb) {
  const float* pa = lp + ra * k;
  const float* pb = lp + rb * k;
  const int a0 = ava ? __ffs(ava) - 1 : -1;
  const int b0 = avb ? __ffs(avb) - 1 : -1;
  const float sa0 = ba + pa[a0 < 0 ? 0 : a0];
  const float sb0 = bb + pb[b0 < 0 ? 0 : b0];
  unsigned ta, tb;
  if (k <= 16) {
    const bool up = lane >= 16;
    const int j = lane & 15;
    const float x = (up ? bb : ba) + (up ? pb : pa)[j];  // j < 16 <= row stride bound of the array
    const unsigned av = up ? avb : ava;
    const int j0 = up ? b0 : a0;
    const bool tie = j0 >= 0 && j > j0 && ((av >> j) & 1u) && x == (up ? sb0 : sa0);
    const unsigned t = __ballot_sync(0xffffffffu, tie);
    ta = t & 0xffffu;
    tb = t >> 16;
  } else {
    const float xa = ba + pa[lane], xb = bb + pb[lane];
    ta = __ballot_sync(0xffffffffu, a0 >= 0 && lane > a0 && ((ava >> lane) & 1u) && xa == sa0);
    tb = __ballot_sync(0xffffffffu, b0 >= 0 && lane > b0 && ((avb >> lane) & 1u) && xb == sb0);
  }
  child_key(a0, sa0, ta, ids + ra * k, sa, ha, la, ja);
  child_key(b0, sb0, tb, ids + rb * k, sb, hb, lb, jb);
}

// Best remaining child of a slot, computed by its owner lane: the first available entry j0 of
// row `row` (a best-first top-k list) and, among the available entries whose score
// parent + logp ties it exactly in fp32, the lowest token (scores fall along the row, so the
// scan stops at the first lower one).  The key is child_key's; (0, 0) when nothing is available.
__device__ __forceinline__ void own_best_child(const float* lp, const int* ids, int k, int row, float parent,
                                               unsigned avail, int slot, uint32_t& hi, uint32_t& lo, int& jb) {
  hi = 0u;
  lo = 0u;
  jb = 0;
  if (avail == 0u) return;
  const int j0 = __ffs(avail) - 1;
  const float* pl = lp + row * k;
  const int* pi = ids + row * k;
  const float s0 = parent + pl[j0];
  int tb = pi[j0];
  jb = j0;
  for (int j = j0 + 1; j < k; ++j) {
    if (parent + pl[j] != s0) break;
    if (((avail >> j) & 1u) && pi[j] < tb) { tb = pi[j]; jb = j; }
  }
  hi = f32_ord(s0);
  lo = ((0x3FFFFFu - static_cast<unsigned>(tb)) << 10) | (0x3FFu - static_cast<unsigned>(slot));
}

__device__ __forceinline__ float f32_from_ord(uint32_t o) {
  return __uint_as_float((o & 0x80000000u) ? (o & 0x7FFFFFFFu) : ~o);
}

// The best-first tree for N <= 31 (every slot in its own lane's registers): the same selection,
// keys and tie rules as the general warp version below, with a short dependency chain per pop.
// The popped child's score and token come out of the winning key itself; only the parent's depth
// crosses lanes; the two slots that change (the popped one and the new node) each compute their
// next best child in their own lane, on the same instruction path.
__device__ void tree_lanes(const float* lp, const int* ids, int K, int k, int N, unsigned all, int lane,
                           int32_t* tpar, int32_t* ttok, int32_t* tdep, float* tsc) {
  // slot `lane`: score, depth, mask of selected entries, cached best child (hi, lo, j), and the
  // node it is (parent index, token)
  float score = 0.f;
  int depth = 0, j = 0, par = -1, tok = -1;
  unsigned mask = 0u;
  uint32_t hi = 0u, lo = 0u;
  own_best_child(lp, ids, k, 0, 0.f, lane == 0 ? all : 0u, 0, hi, lo, j);
  int n_sel = 0;
  for (int i = 0; i < N; ++i) {
    const bool live = lane <= i;
    const uint32_t mhi = __reduce_max_sync(0xffffffffu, live ? hi : 0u);
    if (mhi == 0u) break;  // no frontier left (the host keeps N within the tree's capacity)
    const uint32_t mlo = __reduce_max_sync(0xffffffffu, (live && hi == mhi) ? lo : 0u);
    const int src = __ffs(__ballot_sync(0xffffffffu, live && hi == mhi && lo == mlo)) - 1;
    const int d = __shfl_sync(0xffffffffu, depth, src);
    const float sc = f32_from_ord(mhi);
    const int t = static_cast<int>(0x3FFFFFu - (mlo >> 10));
    const bool is_new = lane == i + 1, is_src = lane == src;
    if (is_new) {
      score = sc;
      depth = d + 1;
      mask = 0u;
      par = src - 1;
      tok = t;
    }
    if (is_src) mask |= 1u << j;
    // the two changed slots: the new node's children come from row d + 1 (none past the last
    // position), the popped slot's from its own row without the entries taken
    const int row = is_new ? (d + 1 < K ? d + 1 : K - 1) : depth;
    const unsigned avail = is_new ? (d + 1 < K ? all : 0u) : (~mask & all);
    if (is_new || is_src) own_best_child(lp, ids, k, row, score, avail, lane, hi, lo, j);
    n_sel = i + 1;
  }
  if (lane >= 1 && lane <= n_sel) {  // node lane - 1
    tpar[lane - 1] = par;
    ttok[lane - 1] = tok;
    tdep[lane - 1] = depth;
    if (tsc) tsc[lane - 1] = score;
  }
}

template <int KM, int KK, int NT>
__global__ void __launch_bounds__(NT, NT == kMergeThreadsNarrow ? 8 : 1) merge_tree_kernel(const TreeParams p) {
  constexpr int F = 2 + 2 * KM;
  constexpr int kWarps = NT / 32;
  static_assert(KK <= KM && kWarps <= 32, "list and warp counts");
  __shared__ float s_mx[kWarps], s_se[kWarps];
  __shared__ int s_last;
  __shared__ float s_cv[kWarps * KK];
  __shared__ int s_ci[kWarps * KK];
  __shared__ float s_lp[kMaxK * kMaxTopk];
  __shared__ int s_id[kMaxK * kMaxTopk];
  __shared__ TreeSlots S;

  const int m = blockIdx.x;
  const int K = p.K, k = p.k, N = p.N, nch = p.nchunks;
  const int b = m / K;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // launched as a programmatic dependent of the vocabulary GEMM: wait for its partials
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // every earlier kernel of the step has completed: its status is final
  if (m == 0 && tid == 0) {
    if (p.status_out) *p.status_out = *p.status;
    if (p.epoch) *p.epoch += 1u;  // the next step's GRU tags its state words differently
  }
  const float* base = p.partials + static_cast<size_t>(m) * F * nch;
  const int* ibase = reinterpret_cast<const int*>(base);

  // ------------------------------------------------------------ this thread's chunks
  // Only the first k entries of each chunk's (sorted) list can reach the row's top k.
  float mx = -INFINITY, se = 0.f;
  float tv[KK];
  int ti[KK];
#pragma unroll
  for (int q = 0; q < KK; ++q) { tv[q] = -INFINITY; ti[q] = -1; }
  for (int c = tid; c < nch; c += NT) {
    const float cm = __ldg(base + c), cs = __ldg(base + nch + c);
    float v[KK];
    int id[KK];
#pragma unroll
    for (int q = 0; q < KK; ++q) {
      v[q] = q < k ? __ldg(base + (2 + q) * nch + c) : -INFINITY;
      id[q] = q < k ? __ldg(ibase + (2 + KM + q) * nch + c) : -1;
    }
    lse_merge(mx, se, cm, cs);
    if (c == tid) {
#pragma unroll
      for (int q = 0; q < KK; ++q) { tv[q] = v[q]; ti[q] = id[q]; }
    } else {
      merge_lists<KK>(tv, ti, v, id);
    }
  }

  // ------------------------------------------------------------ lse over the CTA
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float om = __shfl_xor_sync(0xffffffffu, mx, o);
    const float os = __shfl_xor_sync(0xffffffffu, se, o);
    lse_merge(mx, se, om, os);
  }
  if (lane == 0) { s_mx[warp] = mx; s_se[warp] = se; }

  // ------------------------------------------------------------ k best: per warp, then across warps
  butterfly_lists<KK>(tv, ti, 32);
  if (lane == 0) {
#pragma unroll
    for (int q = 0; q < KK; ++q) { s_cv[warp * KK + q] = tv[q]; s_ci[warp * KK + q] = ti[q]; }
  }
  __syncthreads();
  if (warp == 0) {
    mx = -INFINITY;
    se = 0.f;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) lse_merge(mx, se, s_mx[w], s_se[w]);
    const float lse = mx + logf(se);
    const int src = lane < kWarps ? lane : 0;
#pragma unroll
    for (int q = 0; q < KK; ++q) {
      tv[q] = lane < kWarps ? s_cv[src * KK + q] : -INFINITY;
      ti[q] = lane < kWarps ? s_ci[src * KK + q] : -1;
    }
    butterfly_lists<KK>(tv, ti, kWarps);
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < KK; ++q) {
        if (q < k) {
          p.topk_ids[static_cast<size_t>(m) * k + q] = ti[q];
          p.topk_logp[static_cast<size_t>(m) * k + q] = tv[q] - lse;
        }
      }
    }
  }

  // ------------------------------------------------------------ last row of the sequence?
  __threadfence();
  __syncthreads();
  if (tid == 0) s_last = (atomicAdd(p.seq_done + b, 1u) == static_cast<unsigned>(K - 1));
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  const size_t rows = static_cast<size_t>(b) * K * k;
  for (int e = tid; e < K * k; e += NT) {
    s_id[e] = __ldcg(p.topk_ids + rows + e);
    s_lp[e] = __ldcg(p.topk_logp + rows + e);
  }
  __syncthreads();
  if (warp != 0) return;
  if (N <= 31) {
    const size_t ob1 = static_cast<size_t>(b) * N;
    tree_lanes(s_lp, s_id, K, k, N, (k == 32) ? 0xffffffffu : ((1u << k) - 1u), lane, p.tree_parent + ob1,
               p.tree_token + ob1, p.tree_depth + ob1, p.tree_score ? p.tree_score + ob1 : nullptr);
    return;
  }

  // ------------------------------------------------------------ tree (warp 0)
  // Row reads below stay inside s_lp / s_id: rows are clamped to K - 1 and entries to
  // j < max(k, 16) <= 32, and (K - 1) * k + 31 < kMaxK * kMaxTopk; what a clamped read returns
  // is discarded by the masks.
  const size_t ob = static_cast<size_t>(b) * N;
  const unsigned all = (k == 32) ? 0xffffffffu : ((1u << k) - 1u);
  SlotState mine;  // slot `lane`
  mine.hi = 0u;
  mine.lo = 0u;
  {
    uint32_t ha, la, hb, lb;
    int ja, jb;
    best_children(s_lp, s_id, k, lane, 0, 0.f, all, 0, 0, 0.f, 0u, 0, ha, la, ja, hb, lb, jb);
    if (lane == 0) {
      mine.score = 0.f;
      mine.depth = 0;
      mine.mask = 0u;
      mine.hi = ha;
      mine.lo = la;
      mine.j = ja;
      mine.parent = -1;
      mine.token = -1;
    }
  }
  int n_sel = 0;
  for (int i = 0; i < N; ++i) {
    // best cached child over this lane's slots, with that slot's state
    uint32_t hi = 0u, lo = 0u;
    int sb = -1;
    SlotState w;
    w.depth = 0;
    w.score = 0.f;
    w.mask = 0u;
    w.j = 0;
    if (lane <= i && mine.hi != 0u) { hi = mine.hi; lo = mine.lo; sb = lane; w = mine; }
    for (int s2 = lane + 32; s2 <= i; s2 += 32) {
      const uint32_t h = S.hi[s2], l = S.lo[s2];
      if (h > hi || (h == hi && h != 0u && l > lo)) {
        hi = h;
        lo = l;
        sb = s2;
        w = slot_get(S, mine, s2);
      }
    }
    uint32_t mhi, mlo;
    int src;
    warp_argmax2(hi, lo, mhi, mlo, src);
    if (mhi == 0u) break;  // no frontier left (the host keeps N within the tree's capacity)
    const int s = __shfl_sync(0xffffffffu, sb, src);
    const int jj = __shfl_sync(0xffffffffu, w.j, src);
    const int d = __shfl_sync(0xffffffffu, w.depth, src);
    const float base_s = __shfl_sync(0xffffffffu, w.score, src);
    const unsigned mask_s = __shfl_sync(0xffffffffu, w.mask, src) | (1u << jj);
    const int tok = s_id[d * k + jj];
    const float sc = base_s + s_lp[d * k + jj];
    // new best children of the popped slot s (row d) and of the new node i + 1 (row d + 1)
    const int rn = d + 1 < K ? d + 1 : K - 1;
    uint32_t ha, la, hb, lb;
    int ja, jb;
    best_children(s_lp, s_id, k, lane, d, base_s, ~mask_s & all, s, rn, sc, d + 1 < K ? all : 0u, i + 1, ha, la,
                  ja, hb, lb, jb);
    if (lane == src) {
      w.mask = mask_s;
      w.hi = ha;
      w.lo = la;
      w.j = ja;
      slot_put(S, mine, s, w);
    }
    if (lane == ((i + 1) & 31)) {
      SlotState v;
      v.score = sc;
      v.depth = d + 1;
      v.mask = 0u;
      v.hi = hb;
      v.lo = lb;
      v.j = jb;
      v.parent = s - 1;
      v.token = tok;
      slot_put(S, mine, i + 1, v);
    }
    n_sel = i + 1;
  }
  // each owner writes its nodes: output i is slot i + 1
  for (int sl = lane; sl <= n_sel; sl += 32) {
    if (sl == 0) continue;
    const SlotState v = slot_get(S, mine, sl);
    const int i = sl - 1;
    p.tree_parent[ob + i] = v.parent;
    p.tree_token[ob + i] = v.token;
    p.tree_depth[ob + i] = v.depth;
    if (p.tree_score) p.tree_score[ob + i] = v.score;
  }
}

template <int NT>
static cudaError_t launch_merge_nt(cudaLaunchConfig_t& cfg, const TreeParams& p) {
  cfg.blockDim = dim3(NT);
  if constexpr (NT == kMergeThreadsWide) {
    if (p.kmax == 32) return cudaLaunchKernelEx(&cfg, merge_tree_kernel<32, 32, NT>, p);
  }
  if (p.kmax == 8)
    return p.k <= 4 ? cudaLaunchKernelEx(&cfg, merge_tree_kernel<8, 4, NT>, p)
                    : cudaLaunchKernelEx(&cfg, merge_tree_kernel<8, 8, NT>, p);
  if (p.kmax != 16) return cudaErrorInvalidValue;
  if (p.k <= 4) return cudaLaunchKernelEx(&cfg, merge_tree_kernel<16, 4, NT>, p);
  if (p.k <= 8) return cudaLaunchKernelEx(&cfg, merge_tree_kernel<16, 8, NT>, p);
  return cudaLaunchKernelEx(&cfg, merge_tree_kernel<16, 16, NT>, p);
}

cudaError_t launch_merge_tree(const TreeParams& p, cudaStream_t stream) {
  if (p.K > kMaxK || p.k > kMaxTopk || p.k > p.kmax || p.N > kMaxN) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.B * p.K);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = DOMINO_TREE_PDL ? 1 : 0;
  // 32-entry lists keep the wide CTA (their registers do not fit the narrow one's budget)
  const bool narrow = p.nchunks <= kMergeThreadsNarrow && p.kmax <= 16;
  const cudaError_t e = narrow ? launch_merge_nt<kMergeThreadsNarrow>(cfg, p) : launch_merge_nt<kMergeThreadsWide>(cfg, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dm
