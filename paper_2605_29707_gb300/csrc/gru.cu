// gru.cu -- embedding gather (E_j, section 4.1.2), the GRU causal encoder
// S_{i-1} = GRU(E_{<=i-1}) and the low-rank code u = SiLU(W1 [H_i; S_{i-1}] + b1).
//
// The recurrence is the only sequential part of the step: K dependent steps, each needing the
// full previous state of a sequence.  One cooperative launch keeps the W_hh rows of a block of
// hidden units resident in shared memory for all K steps and computes W_hh . h_{t-1} on the
// tensor cores (mma.sync, bf16 operands, fp32 accumulation).  States cross CTAs through L2 as
// tagged words (bf16 value in the high half, the step's 16-bit tag in the low half; one row per
// (sequence, position)), so a CTA waits for exactly the data it reads: no grid barrier and no
// release fence.  Every wait is bounded.
#include <math.h>

#include <atomic>

#include "kernels.h"
#include "ptx.cuh"

#ifndef DOMINO_GRU_BACKOFF_NS
#define DOMINO_GRU_BACKOFF_NS 64  // pause between re-reads of a state word that is not ready
#endif

namespace dm {

constexpr int kGruThreads = 256;
constexpr int kGatePairsPerThread = 2;  // (sequence, unit) gate evaluations per thread and chunk
constexpr int kGruWarps = kGruThreads / 32;
constexpr int kChunkSeqs = 32;  // sequences staged per MMA pass (4 n-tiles of 8)
constexpr int kGsmLd = kChunkSeqs + 1;  // padded row stride of the W_hh . h tile (bank spread)
constexpr int kMaxMt = 3;  // 16-row gate tiles per CTA (up to 16 units x 3 gates)
constexpr int kMaxNt = 4;  // 8-sequence tiles per staged chunk

// ---------------------------------------------------------------------------- gather
__global__ void __launch_bounds__(128) gather_kernel(const GatherParams p) {
  // the input projection launched after this kernel may start its setup now; it waits for
  // this grid before it reads E
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int m = blockIdx.x;
  const int id = p.ids[m];
  const bool ok = id >= 0 && id < p.V;
  if (!ok && threadIdx.x == 0) set_status(p.status, kStatusBadToken);
  if (p.hx != nullptr) {
    uint4* hrow = reinterpret_cast<uint4*>(p.hx + static_cast<size_t>(m) * p.Ds);
    for (int c = threadIdx.x; c < p.Ds / 4; c += blockDim.x) hrow[c] = make_uint4(0, 0, 0, 0);
  }
  if (p.E == nullptr) return;
  uint4* dst = reinterpret_cast<uint4*>(p.E + static_cast<size_t>(m) * p.H);
  const uint4* src = reinterpret_cast<const uint4*>(p.emb + static_cast<size_t>(ok ? id : 0) * p.H);
  for (int c = threadIdx.x; c < p.H / 8; c += blockDim.x) dst[c] = ok ? __ldg(src + c) : make_uint4(0, 0, 0, 0);
}

cudaError_t launch_gather(const GatherParams& p, cudaStream_t stream) {
  gather_kernel<<<p.M, 128, 0, stream>>>(p);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------- helpers
__device__ __forceinline__ uint4 ld_relaxed_v4(const uint32_t* p) {
  uint4 v;
  asm volatile("ld.relaxed.gpu.global.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p)
               : "memory");
  return v;
}

// Four state words all written in this step: their low halves equal the step's tag.
__device__ __forceinline__ bool all_tagged(const uint4& v, uint32_t tag) {
  return (((v.x ^ tag) | (v.y ^ tag) | (v.z ^ tag) | (v.w ^ tag)) & 0xFFFFu) == 0u;
}

// Reads 4 tagged state words, re-reading until all four carry this step's tag.  Returns false
// if that takes longer than kWaitCycles (the caller reports DOMINO_ERR_TIMEOUT).
__device__ __forceinline__ bool poll_v4(const uint32_t* p, uint4& v, uint32_t tag) {
  v = ld_relaxed_v4(p);
  if (all_tagged(v, tag)) return true;
  const long long t0 = clock64();
  while (true) {
    if (DOMINO_GRU_BACKOFF_NS > 0) __nanosleep(DOMINO_GRU_BACKOFF_NS);  // spare L2 while waiting
    v = ld_relaxed_v4(p);
    if (all_tagged(v, tag)) return true;
    if (clock64() - t0 > kWaitCycles) return false;
  }
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long* p) {
  unsigned long long v;
  asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
  return v;
}

// Does the recorded range `have` (lo | hi << 32; 0 = none) contain the range `want`?
__device__ __forceinline__ bool range_contains(unsigned long long have, unsigned long long want) {
  const uint32_t hl = static_cast<uint32_t>(have), hh = static_cast<uint32_t>(have >> 32);
  const uint32_t wl = static_cast<uint32_t>(want), wh = static_cast<uint32_t>(want >> 32);
  return have != 0ull && hl <= wl && wh <= hh;
}

// Test hook state (domino_debug_hold): what to withhold, from which CTA, at which position.
__device__ int3 g_gru_hold = {kHoldOff, -1, -1};

cudaError_t arm_gru_hold(int what, int cta, int step) {
  const int3 v = make_int3(what, cta, step);
  return cudaMemcpyToSymbol(g_gru_hold, &v, sizeof(v));
}

// Grid barrier of a cooperative launch that needs no reset: the word holds the generation in its
// high half and the arrivals of that generation in its low half; the first arrival of a new
// generation restarts the count.  Every generation is used by one launch only (the step epoch),
// so a word another launch left behind never counts.  Called by every thread of the CTA; false
// when the wait ran past kWaitCycles (or the hook withheld this CTA's arrival and its peers').
__device__ bool grid_barrier_gen(unsigned long long* bar, uint32_t gen, uint32_t count, bool skip_arrival) {
  __syncthreads();
  int ok = 1;
  if (threadIdx.x == 0) {
    __threadfence();  // this CTA's writes before its arrival
    if (!skip_arrival) {
      unsigned long long old = ld_relaxed_u64(bar), assumed;
      int tries = 0;
      do {
        assumed = old;
        const unsigned long long next = static_cast<uint32_t>(assumed >> 32) == gen
                                            ? assumed + 1ull
                                            : (static_cast<unsigned long long>(gen) << 32) | 1ull;
        old = atomicCAS(bar, assumed, next);
      } while (old != assumed && ++tries < (1 << 20));
      if (old != assumed) ok = 0;
    }
    const unsigned long long want = (static_cast<unsigned long long>(gen) << 32) | count;
    const long long t0 = clock64();
    while (ok && ld_acquire_u64(bar) != want) {
      __nanosleep(64);
      if (clock64() - t0 > kWaitCycles) ok = 0;
    }
    __threadfence();
  }
  return __syncthreads_and(ok) != 0;
}

__device__ __forceinline__ uint32_t tagged(float h, uint32_t tag) {
  const uint32_t b = static_cast<uint32_t>(__bfloat16_as_ushort(__float2bfloat16_rn(h)));
  return (b << 16) | tag;
}

// two tagged words -> packed bf16x2 (low element first)
__device__ __forceinline__ uint32_t pack_hi_halves(uint32_t lo_word, uint32_t hi_word) {
  return (lo_word >> 16) | (hi_word & 0xFFFF0000u);
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gmem_src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(smem_u32(p)));
}

__device__ __forceinline__ void ldmatrix_x2(uint32_t (&r)[2], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0,%1}, [%2];" : "=r"(r[0]), "=r"(r[1]) : "r"(smem_u32(p)));
}

// D (16x8, f32) += A (16x16 bf16, row-major) * B (16x8 bf16, column-major)
__device__ __forceinline__ void mma_16816(float (&c)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float bf_or0(const __nv_bfloat16* p, int i) {
  return p ? __bfloat162float(p[i]) : 0.f;
}

__device__ __forceinline__ float sigmoidf_(float x) { return 1.f / (1.f + expf(-x)); }

// ---------------------------------------------------------------------------- smem layout
// whh   [mt*16 rows][Ds + 8] bf16  this CTA's W_hh rows (gate g, unit jl) at row g*U + jl;
//                                  rows past 3U are zero
// hsm   [chunk][Ds + 8] bf16       h_{t-1} of up to 32 sequences (the MMA's n operand)
// gsm   [mt*16][33] f32            W_hh . h_{t-1} (padded rows)
// red   [8 warps][tiles][16][8] f32  k-range partial tiles of each warp
// hprev [bc][U] f32                this CTA's own previous states (fp32)
struct GruSmem {
  size_t whh, hsm, gsm, red, hprev, total;
  int ldw, mt, chunk;
};

__host__ __device__ inline GruSmem gru_layout(int Ds, int U, int bc) {
  GruSmem L;
  L.ldw = Ds + 8;
  L.mt = (3 * U + 15) / 16;
  L.chunk = ((bc < kChunkSeqs ? bc : kChunkSeqs) + 7) / 8 * 8;  // staged sequences, whole n-tiles
  size_t o = 0;
  L.whh = o;
  o += static_cast<size_t>(L.mt) * 16 * L.ldw * 2;
  L.hsm = o;
  o += static_cast<size_t>(L.chunk) * L.ldw * 2;
  L.gsm = o;
  o += static_cast<size_t>(L.mt) * 16 * kGsmLd * 4;
  L.red = o;  // [warp][tile][16][8] partials of each warp's k-range
  o += static_cast<size_t>(kGruWarps) * L.mt * (L.chunk / 8) * 128 * 4;
  L.hprev = o;
  o += static_cast<size_t>(bc) * U * 4;
  L.total = (o + 15) & ~static_cast<size_t>(15);
  return L;
}

// ---------------------------------------------------------------------------- fused projections
__device__ __forceinline__ void ldg_words8(const __nv_bfloat16* row, int k0, int H, bool valid, uint32_t (&w)[8]) {
  // elements k0 .. k0 + 15 of a row (two 16-byte halves; zero past H or for an invalid row)
  const uint4 lo = (valid && k0 < H) ? __ldg(reinterpret_cast<const uint4*>(row + k0)) : make_uint4(0, 0, 0, 0);
  const uint4 hi = (valid && k0 + 8 < H) ? __ldg(reinterpret_cast<const uint4*>(row + k0 + 8)) : make_uint4(0, 0, 0, 0);
  w[0] = lo.x; w[1] = lo.y; w[2] = lo.z; w[3] = lo.w;
  w[4] = hi.x; w[5] = hi.y; w[6] = hi.z; w[7] = hi.w;
}

// Small batches, u computed in-kernel: this CTA's input-gate sums xs = b_ih + E . W_ih^T for its
// units (E = emb rows of the prefix ids, which are checked here) on the tensor cores, and the
// hidden half of u, hidden_m . W1[q, :H], for the (q, m) pairs each warp finalises after the
// recurrence.  The MMA (m16n8k16, positions on M, the 3 x 8 gate rows of the units on N) sums k
// in an order of its own: in each 64-element chunk, lane l = 4 g + t loads elements
// 16 t .. 16 t + 15 of its A rows (g, g + 8) and B row (g), and MMA step s of the chunk takes
// words 2 s and 2 s + 1 of those, the same columns in A and B.  The warps split k; their partial
// tiles meet in `red` (one 16 x 8 tile per warp at a time).
template <bool kTable>
__device__ void fused_projections(const GruParams& p, int j0, int Uc, int b0, int nbc, float* red,
                                  float (*s_uh)[kGruMaxUPairs]) {
  const int H = p.H, Ds = p.Ds, K = p.K, R = p.R, M = p.B * p.K;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t = lane & 3;
  __syncthreads();  // CTA 0: the status reset comes first
  if (blockIdx.x == 0) {
    for (int m = tid; m < M; m += kGruThreads) {
      const int id = p.ids[m];
      if (id < 0 || id >= p.V) set_status(p.status, kStatusBadToken);
    }
  }
  const int rows = nbc * K;  // this CTA's positions: m = b0 * K + r
  const int nchunk = (H + 63) / 64;
  const int c_lo = (nchunk * warp) / kGruWarps, c_hi = (nchunk * (warp + 1)) / kGruWarps;
  // B rows of n-tile nt: gate nt, unit g (8 units per CTA on this path)
  const __nv_bfloat16* brow[3];
  bool bvalid[3];
#pragma unroll
  for (int nt = 0; nt < 3; ++nt) {
    bvalid[nt] = g < Uc;
    brow[nt] = p.w_ih + static_cast<size_t>(nt * Ds + j0 + (g < Uc ? g : 0)) * H;
  }
  for (int mt = 0; !kTable && mt * 16 < rows; ++mt) {  // with a table the steps read its rows
    const int ra = mt * 16 + g, rb = ra + 8;
    const int ida = ra < rows ? p.ids[b0 * K + ra] : 0, idb = rb < rows ? p.ids[b0 * K + rb] : 0;
    const bool va = ra < rows && ida >= 0 && ida < p.V, vb = rb < rows && idb >= 0 && idb < p.V;
    const __nv_bfloat16* arow = p.emb + static_cast<size_t>(va ? ida : 0) * H;
    const __nv_bfloat16* brow2 = p.emb + static_cast<size_t>(vb ? idb : 0) * H;
    float acc[3][4];
#pragma unroll
    for (int nt = 0; nt < 3; ++nt) acc[nt][0] = acc[nt][1] = acc[nt][2] = acc[nt][3] = 0.f;
    for (int c = c_lo; c < c_hi; ++c) {
      const int k0 = c * 64 + 16 * t;
      uint32_t wa[8], wb[8], wn[3][8];
      ldg_words8(arow, k0, H, va, wa);
      ldg_words8(brow2, k0, H, vb, wb);
#pragma unroll
      for (int nt = 0; nt < 3; ++nt) ldg_words8(brow[nt], k0, H, bvalid[nt], wn[nt]);
#pragma unroll
      for (int st = 0; st < 4; ++st) {
        const uint32_t a[4] = {wa[2 * st], wb[2 * st], wa[2 * st + 1], wb[2 * st + 1]};
#pragma unroll
        for (int nt = 0; nt < 3; ++nt) {
          const uint32_t b[2] = {wn[nt][2 * st], wn[nt][2 * st + 1]};
          mma_16816(acc[nt], a, b);
        }
      }
    }
    // sum the warps' tiles, one gate (n-tile) at a time: entry (row, col) of the 16 x 8 tile
#pragma unroll
    for (int nt = 0; nt < 3; ++nt) {
      float* out = red + warp * 128;
      out[g * 8 + 2 * t] = acc[nt][0];
      out[g * 8 + 2 * t + 1] = acc[nt][1];
      out[(g + 8) * 8 + 2 * t] = acc[nt][2];
      out[(g + 8) * 8 + 2 * t + 1] = acc[nt][3];
      __syncthreads();
      if (tid < 128) {
        const int row = tid / 8, jl = tid % 8, r = mt * 16 + row;
        if (r < rows && jl < Uc) {
          float sum = bf_or0(p.b_ih, nt * Ds + j0 + jl);
#pragma unroll
          for (int w = 0; w < kGruWarps; ++w) sum += red[w * 128 + tid];
          p.xs[static_cast<size_t>(b0 * K + r) * 3 * Ds + nt * Ds + j0 + jl] = sum;
        }
      }
      __syncthreads();
    }
  }
  // hidden halves of u for this warp's (q, m) pairs, in the tail's order
  const int total_warps = gridDim.x * kGruWarps;
  const int gw = blockIdx.x * kGruWarps + warp;
  const int groups = max(1, total_warps / R);
  int np = 0;
  for (int pi = gw; pi < R * groups; pi += total_warps) {
    const int q = pi % R, mg = pi / R;
    const __nv_bfloat16* w1row = p.w1 + static_cast<size_t>(q) * (H + Ds);
    for (int m = mg; m < M; m += groups, ++np) {
      const __nv_bfloat16* hrow = p.hidden + static_cast<size_t>(m) * H;
      float acc = 0.f;
#pragma unroll 4
      for (int c = lane * 8; c < H; c += 256) {
        const uint4 wv = __ldg(reinterpret_cast<const uint4*>(w1row + c));
        const uint4 hv = __ldg(reinterpret_cast<const uint4*>(hrow + c));
        const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&wv);
        const __nv_bfloat162* h2 = reinterpret_cast<const __nv_bfloat162*>(&hv);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float2 wf = __bfloat1622float2(w2[i]), hf = __bfloat1622float2(h2[i]);
          acc = fmaf(wf.x, hf.x, acc);
          acc = fmaf(wf.y, hf.y, acc);
        }
      }
      acc = warp_sum(acc);
      if (lane == 0 && np < kGruMaxUPairs) s_uh[warp][np] = acc;
    }
  }
}

// At most 128 registers per thread (two CTAs' worth per SM), so that a GRU CTA and a vocabulary
// GEMM CTA (at most 168 registers x 192 threads) fit in one SM's register file.
// kTable: the input-gate sums come from the input-projection table (p.x_table) rather than
// from xs (a separate instantiation, so that the path without a table keeps its registers).
// kWide: a launch that shares no SM with the vocabulary GEMM (large batches): the register
// budget of one CTA per SM, so that a lane issues all 16 of its state loads of a step at once
// (one L2 round trip instead of two at 16 sequences per CTA), and the steps read the input-gate
// sums as split-K partial sums of the X GEMM directly (prefetched before each step's wait)
// instead of a prologue pass that first sums them into xs.
template <bool kTable, bool kWide>
__global__ void __launch_bounds__(kGruThreads, kWide ? 1 : 2) gru_kernel(const GruParams p) {
  constexpr int kPollBatch = kWide ? 16 : 8;  // state loads a lane issues before checking tags
  extern __shared__ __align__(16) uint8_t gsmem[];
  const int U = p.units, Ds = p.Ds, K = p.K, B = p.B, R = p.R, H = p.H;
  const int M = B * K;
  const int cu = blockIdx.x % p.gu, cb = blockIdx.x / p.gu;
  const int j0 = cu * U;
  const int Uc = max(0, min(U, Ds - j0));
  const int b0 = cb * p.bc;
  const int nbc = max(0, min(p.bc, B - b0));  // sequences of this CTA
  const GruSmem L = gru_layout(Ds, U, p.bc);
  __nv_bfloat16* whh = reinterpret_cast<__nv_bfloat16*>(gsmem + L.whh);
  __nv_bfloat16* hsm = reinterpret_cast<__nv_bfloat16*>(gsmem + L.hsm);
  float* gsm = reinterpret_cast<float*>(gsmem + L.gsm);
  float* red = reinterpret_cast<float*>(gsmem + L.red);
  float* hprev = reinterpret_cast<float*>(gsmem + L.hprev);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ldw = L.ldw;
  // This step's tag for the state words (low half): the workspace's step epoch, advanced by
  // the merge kernel at the end of every step, so that words a previous step wrote never pass
  // for this step's; 0 (a cleared word) is never a tag.
  const uint32_t tag = (*p.epoch % 0xFFFFu) + 1u;
  // Without a clear before the launch (fused projections) the first CTA resets the step's
  // status and the merge counters; only it then checks the ids (after the barrier below), so a
  // reset can never hide an error of this step.
  if (p.reset_ctrl && blockIdx.x == 0 && tid == 0) {
    *p.status = 0;
    for (int b = 0; b < B; ++b) p.seq_done[b] = 0u;
  }
  // the vocabulary GEMM that follows may start now: its first K segment does not read
  // anything this kernel writes, and it waits for this grid before reading u
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  const int3 hold = g_gru_hold;
  const bool held = hold.x != kHoldOff && hold.y == static_cast<int>(blockIdx.x);

  // ---- no clear before the launch: a stale word passes for this step's only if its low half
  //      equals the tag, which words of earlier steps never do (the epoch advances every step) but
  //      other data may.  So the tags are trusted only where the workspace held nothing but state
  //      words at the end of the last step: the range recorded in the control words (written by
  //      the last step of this kind, zeroed by any other step).  When it does not cover this
  //      launch's hx, every CTA zeroes the words it will itself write and the grid meets at a
  //      barrier before any CTA reads a state.
  if (p.layout != nullptr) {
    const unsigned long long have = ld_relaxed_u64(p.layout);
    if (!range_contains(have, p.layout_range)) {
      const int Ucl = Uc;
      for (int e = tid; e < nbc * K * Ucl; e += kGruThreads) {
        const size_t m = static_cast<size_t>(b0) * K + e / Ucl;
        p.hx[m * Ds + j0 + e % Ucl] = 0u;
      }
      const bool skip = held && hold.x == kHoldClearBarrier;
      if (!grid_barrier_gen(p.clear_bar, *p.epoch + 1u, gridDim.x, skip)) {
        if (tid == 0) set_status(p.status, kStatusTimeout);
        if (held && tid == 0) g_gru_hold = make_int3(kHoldOff, -1, -1);
        return;
      }
    }
    // every CTA has read the record (before the barrier, or it already covered this range)
    if (blockIdx.x == 0 && tid == 0 && have != p.layout_range) *p.layout = p.layout_range;
  }

  // ---- W_hh rows of this CTA's units (asynchronous); zero rows past 3U and the state tile
  const int rowlen8 = Ds / 8;
  for (int e = tid; e < 3 * Uc * rowlen8; e += kGruThreads) {
    const int c8 = e % rowlen8, r = e / rowlen8;
    const int g = r / Uc, jl = r % Uc;
    cp_async16(whh + static_cast<size_t>(g * U + jl) * ldw + c8 * 8,
               p.w_hh + (static_cast<size_t>(g) * Ds + j0 + jl) * Ds + c8 * 8);
  }
  for (int e = tid; e < L.mt * 16 * (ldw / 8); e += kGruThreads) {
    const int r = e / (ldw / 8);
    const int jl = r % U;
    if (r >= 3 * U || jl >= Uc) reinterpret_cast<uint4*>(whh)[e] = make_uint4(0, 0, 0, 0);
  }
  for (int r = tid; r < L.mt * 16; r += kGruThreads)  // padding columns Ds .. Ds+7 (k tail)
    *reinterpret_cast<uint4*>(whh + static_cast<size_t>(r) * ldw + Ds) = make_uint4(0, 0, 0, 0);
  for (int e = tid; e < L.chunk * (ldw / 8); e += kGruThreads) reinterpret_cast<uint4*>(hsm)[e] = make_uint4(0, 0, 0, 0);
  __shared__ float s_uh[kGruWarps][kGruMaxUPairs];  // fused: hidden halves of this warp's u pairs
  if (p.ids != nullptr) {
    fused_projections<kTable>(p, j0, Uc, b0, nbc, red, s_uh);
  } else {
  // Launched as a programmatic dependent of the projection GEMMs: everything below reads
  // what they (and, through their own waits, the gather) wrote -- X partials, u partials and
  // the cleared state words.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // ---- input-gate sums b_ih + E . W_ih^T for this CTA's rows and units, spread over all
  //      threads (made visible to the CTA by the barrier below)
  // with a table the steps read its rows; wide launches read the partial sums at each step
  const int xs_count = (kTable || kWide) ? 0 : nbc * K * 3 * Uc;
  for (int e0 = tid; e0 < xs_count; e0 += 4 * kGruThreads) {
    float a[4];
    size_t at[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int e = e0 + i * kGruThreads;
      a[i] = 0.f;
      at[i] = 0;
      if (e < xs_count) {
        const int jl = e % Uc, g = (e / Uc) % 3, bt = e / (3 * Uc);
        const int col = g * Ds + j0 + jl;
        const size_t m = static_cast<size_t>(b0) * K + bt;
        at[i] = m * 3 * Ds + col;
        a[i] = bf_or0(p.b_ih, col);
      }
    }
    for (int s = 0; s < p.xsplits; ++s) {
      const float* base = p.xpart + static_cast<size_t>(s) * M * 3 * Ds;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (e0 + i * kGruThreads < xs_count) a[i] += __ldg(base + at[i]);
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
      if (e0 + i * kGruThreads < xs_count) p.xs[at[i]] = a[i];
  }
  }
  for (int e = tid; e < nbc * U; e += kGruThreads) hprev[e] = 0.f;
  cp_async_wait_all();
  __syncthreads();

  const int nk = (Ds + 15) / 16;  // a k tail of 8 reads the zero padding columns
  bool ok = true;
  // The biases of this thread's gate pairs do not change from step to step (pair e of a chunk is
  // unit e % Uc).  b_ih is already in xs except when the steps read a table row or X partials.
  float bih[kGatePairsPerThread][3], bhh[kGatePairsPerThread][3];
#pragma unroll
  for (int r = 0; r < kGatePairsPerThread; ++r) {
    const int j = j0 + (Uc > 0 ? (tid + r * kGruThreads) % Uc : 0);
#pragma unroll
    for (int g = 0; g < 3; ++g) {
      bih[r][g] = (kTable || kWide) ? bf_or0(p.b_ih, g * Ds + j) : 0.f;
      bhh[r][g] = bf_or0(p.b_hh, g * Ds + j);
    }
  }

  for (int t = 0; t < K && ok; ++t) {
    for (int c0 = 0; c0 < nbc; c0 += L.chunk) {
      const int nb = min(L.chunk, nbc - c0);
      const int nt_count = (nb + 7) / 8;
      const int tiles = L.mt * nt_count;
      // gate inputs of this step: issued as loads now and summed only at the gates, after the
      // wait for h_{t-1}, so that no instruction stalls on them before the wait
      constexpr int kXr = kWide ? 3 : 1;  // X partial sums held per gate (more are summed at once)
      float gx[kGatePairsPerThread][3][kXr];
#pragma unroll
      for (int r = 0; r < kGatePairsPerThread; ++r) {
        const int e = tid + r * kGruThreads;
#pragma unroll
        for (int g = 0; g < 3; ++g)
#pragma unroll
          for (int s = 0; s < kXr; ++s) gx[r][g][s] = 0.f;
        if (e < nb * Uc) {
          const int bb = e / Uc, jl = e % Uc;
          const int j = j0 + jl;
          const size_t m = static_cast<size_t>(b0 + c0 + bb) * K + t;
          // b_ih + W_i{r,z,n} E_m: summed into xs before the steps, or a row of the table (an id
          // outside [0, V), reported by the id check, reads row 0), or the X GEMM's split-K partial
          // sums (wide launches)
          const float* x = p.xs + m * 3 * Ds;  // written by this kernel: plain loads
          int nsplit = 1;
          size_t split_stride = 0;
          if (kTable) {
            const int id = p.x_ids[m];
            x = p.x_table + static_cast<size_t>(id >= 0 && id < p.V ? id : 0) * 3 * Ds;
          } else if (kWide) {
            x = p.xpart + m * 3 * Ds;
            nsplit = p.xsplits;
            split_stride = static_cast<size_t>(M) * 3 * Ds;
          }
#pragma unroll
          for (int g = 0; g < 3; ++g) {
#pragma unroll
            for (int s = 0; s < kXr; ++s)
              if (s < nsplit) gx[r][g][s] = x[s * split_stride + g * Ds + j];
            for (int s = kXr; s < nsplit; ++s) gx[r][g][0] += x[s * split_stride + g * Ds + j];  // rare
          }
        }
      }
      if (t > 0) {
        // ---- each warp owns k-range [kw0, kw1) of W_hh . h_{t-1} (one k16 block is the state
        //      of 16 consecutive units, i.e. of one or two writer CTAs): it polls exactly those
        //      state words, stages them and multiplies them at once, so the tensor work on early
        //      k-ranges overlaps the wait for late writers
        const int kw0 = (nk * warp) / kGruWarps, kw1 = (nk * (warp + 1)) / kGruWarps;
        const int q0 = kw0 * 4, q1 = min(kw1 * 4, Ds / 4);  // 4-word columns of the range
        const int ncq = max(0, q1 - q0);
        const int total = nb * ncq;
        bool got = true;
        for (int e0 = lane; e0 < total && got; e0 += kPollBatch * 32) {
          uint4 v[kPollBatch];
#pragma unroll
          for (int i = 0; i < kPollBatch; ++i) {  // issue every load first, then check the flags
            const int e = e0 + i * 32;
            if (e < total) {
              const size_t m = static_cast<size_t>(b0 + c0 + e / ncq) * K + (t - 1);
              v[i] = ld_relaxed_v4(p.hx + m * Ds + (q0 + e % ncq) * 4);
            }
          }
#pragma unroll
          for (int i = 0; i < kPollBatch; ++i) {
            const int e = e0 + i * 32;
            if (e < total && got) {
              const int bb = e / ncq, cq = q0 + e % ncq;
              if (!all_tagged(v[i], tag)) {
                const size_t m = static_cast<size_t>(b0 + c0 + bb) * K + (t - 1);
                got = poll_v4(p.hx + m * Ds + cq * 4, v[i], tag);
              }
              *reinterpret_cast<uint2*>(hsm + static_cast<size_t>(bb) * ldw + cq * 4) =
                  make_uint2(pack_hi_halves(v[i].x, v[i].y), pack_hi_halves(v[i].z, v[i].w));
            }
          }
        }
        got = __all_sync(0xffffffffu, got);
        __syncwarp();
        if (got) {
          float acc[kMaxMt][kMaxNt][4];
#pragma unroll
          for (int a = 0; a < kMaxMt; ++a)
#pragma unroll
            for (int b = 0; b < kMaxNt; ++b) acc[a][b][0] = acc[a][b][1] = acc[a][b][2] = acc[a][b][3] = 0.f;
          const __nv_bfloat16* abase = whh + static_cast<size_t>(lane & 15) * ldw + (lane >> 4) * 8;
          const __nv_bfloat16* bbase = hsm + static_cast<size_t>(lane & 7) * ldw + ((lane >> 3) & 1) * 8;
          for (int kb = kw0; kb < kw1; ++kb) {
            uint32_t bf[kMaxNt][2];
#pragma unroll
            for (int nt = 0; nt < kMaxNt; ++nt)
              if (nt < nt_count) ldmatrix_x2(bf[nt], bbase + static_cast<size_t>(nt * 8) * ldw + kb * 16);
#pragma unroll
            for (int mt = 0; mt < kMaxMt; ++mt) {
              if (mt >= L.mt) break;
              uint32_t af[4];
              ldmatrix_x4(af, abase + static_cast<size_t>(mt * 16) * ldw + kb * 16);
#pragma unroll
              for (int nt = 0; nt < kMaxNt; ++nt)
                if (nt < nt_count) mma_16816(acc[mt][nt], af, bf[nt]);
            }
          }
          const int g = lane >> 2, tq = lane & 3;
#pragma unroll
          for (int mt = 0; mt < kMaxMt; ++mt) {
            if (mt >= L.mt) break;
#pragma unroll
            for (int nt = 0; nt < kMaxNt; ++nt) {
              if (nt >= nt_count) continue;
              float* out = red + (static_cast<size_t>(warp) * tiles + mt * nt_count + nt) * 128;
              out[g * 8 + 2 * tq] = acc[mt][nt][0];
              out[g * 8 + 2 * tq + 1] = acc[mt][nt][1];
              out[(g + 8) * 8 + 2 * tq] = acc[mt][nt][2];
              out[(g + 8) * 8 + 2 * tq + 1] = acc[mt][nt][3];
            }
          }
        }
        if (__syncthreads_or(!got)) {
          set_status(p.status, kStatusTimeout);
          ok = false;
          break;
        }
        // ---- sum the eight k-range partials of every tile
        for (int e = tid; e < tiles * 128; e += kGruThreads) {
          const int tile = e / 128, w = e % 128;
          float sum = 0.f;
#pragma unroll
          for (int ww = 0; ww < kGruWarps; ++ww) sum += red[(static_cast<size_t>(ww) * tiles + tile) * 128 + w];
          const int mt = tile / nt_count, nt = tile % nt_count;
          gsm[static_cast<size_t>(mt * 16 + w / 8) * kGsmLd + nt * 8 + (w % 8)] = sum;
        }
        __syncthreads();
      }
      // ---- gates and the new state (torch.nn.GRU convention); publish the tagged state
#pragma unroll
      for (int rr = 0; rr < kGatePairsPerThread; ++rr) {
        const int e = tid + rr * kGruThreads;
        if (e >= nb * Uc) break;
        const int bb = e / Uc, jl = e % Uc;
        const int j = j0 + jl;
        const int bl = c0 + bb;  // sequence index within this CTA
        const size_t m = static_cast<size_t>(b0 + bl) * K + t;
        float hr = bhh[rr][0], hz = bhh[rr][1], hn = bhh[rr][2];
        if (t > 0) {
          hr += gsm[static_cast<size_t>(jl) * kGsmLd + bb];
          hz += gsm[static_cast<size_t>(U + jl) * kGsmLd + bb];
          hn += gsm[static_cast<size_t>(2 * U + jl) * kGsmLd + bb];
        }
        float xin[3];
#pragma unroll
        for (int g = 0; g < 3; ++g) {
          float s = gx[rr][g][0];
#pragma unroll
          for (int q = 1; q < kXr; ++q) s += gx[rr][g][q];
          xin[g] = s + bih[rr][g];
        }
        const float hp = hprev[bl * U + jl];
        const float r = sigmoidf_(xin[0] + hr);
        const float z = sigmoidf_(xin[1] + hz);
        const float n = tanhf(xin[2] + r * hn);
        const float h = (1.f - z) * n + z * hp;
        hprev[bl * U + jl] = h;
        if (held && hold.x == kHoldPublish && hold.z == t) continue;  // test hook: withheld
        p.hx[m * Ds + j] = tagged(h, tag);
        if (p.s_out) p.s_out[m * Ds + j] = __float2bfloat16_rn(h);
      }
      __syncthreads();
    }
  }
  if (held && tid == 0) g_gru_hold = make_int3(kHoldOff, -1, -1);  // the hook holds one launch
  if (!ok || p.u == nullptr) return;

  // ---- u[m, q] = SiLU(b1[q] + hidden_m . W1[q, :H] + S_m . W1[q, H:]) (small batches): the
  //      hidden half arrives as split-K partial sums, the state half is a warp dot over the
  //      tagged states (polled: other CTAs may still be publishing their last step)
  const int total_warps = gridDim.x * kGruWarps;
  const int gw = blockIdx.x * kGruWarps + warp;
  const int groups = max(1, total_warps / R);
  int np = 0;  // this warp's pair counter (the fused prologue's order)
  for (int pi = gw; pi < R * groups; pi += total_warps) {
    const int q = pi % R, mg = pi / R;
    const __nv_bfloat16* w1row = p.w1 + static_cast<size_t>(q) * (H + Ds) + H;
    const float bq = bf_or0(p.b1, q);
    for (int m = mg; m < M; m += groups) {
      const uint32_t* srow = p.hx + static_cast<size_t>(m) * Ds;
      float acc = 0.f;
      bool got = true;
      for (int c0 = lane * 8; c0 < Ds && got; c0 += 4 * 256) {
        uint4 wv[4], sv[8];
#pragma unroll
        for (int i = 0; i < 4; ++i) {  // issue every load of this slice first
          const int c = c0 + i * 256;
          if (c < Ds) {
            wv[i] = __ldg(reinterpret_cast<const uint4*>(w1row + c));
            sv[2 * i] = ld_relaxed_v4(srow + c);
            sv[2 * i + 1] = ld_relaxed_v4(srow + c + 4);
          }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int c = c0 + i * 256;
          if (c >= Ds || !got) continue;
          for (int h = 0; h < 2; ++h) {
            uint4& x = sv[2 * i + h];
            if (!all_tagged(x, tag)) got = got && poll_v4(srow + c + 4 * h, x, tag);
          }
          const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&wv[i]);
          const uint32_t sw[8] = {sv[2 * i].x, sv[2 * i].y, sv[2 * i].z, sv[2 * i].w,
                                  sv[2 * i + 1].x, sv[2 * i + 1].y, sv[2 * i + 1].z, sv[2 * i + 1].w};
#pragma unroll
          for (int q2 = 0; q2 < 4; ++q2) {
            const float2 wf = __bfloat1622float2(w2[q2]);
            acc = fmaf(wf.x, __uint_as_float(sw[2 * q2] & 0xFFFF0000u), acc);
            acc = fmaf(wf.y, __uint_as_float(sw[2 * q2 + 1] & 0xFFFF0000u), acc);
          }
        }
      }
      if (__any_sync(0xffffffffu, !got)) {
        if (lane == 0) set_status(p.status, kStatusTimeout);
        return;
      }
      if (p.ids != nullptr) {
        if (lane == 0 && np < kGruMaxUPairs) acc += s_uh[warp][np];
        ++np;
      } else {
        for (int s = lane; s < p.usplits; s += 32) acc += __ldg(p.upart + (static_cast<size_t>(s) * M + m) * R + q);
      }
      acc = warp_sum(acc);
      if (lane == 0) {
        const float a = acc + bq;
        p.u[static_cast<size_t>(m) * R + q] = __float2bfloat16_rn(a / (1.f + expf(-a)));
      }
    }
  }
}

GruPlan gru_plan(int B, int Ds, int num_sms) {
  GruPlan g{};
  // 8 units (2 gate tiles) per CTA for small batches, 16 (3 gate tiles) otherwise
  g.units = B <= 8 ? 8 : 16;
  g.gu = (Ds + g.units - 1) / g.units;
  if (g.gu > num_sms) {
    g.units = 16;
    g.gu = (Ds + g.units - 1) / g.units;
    if (g.gu > num_sms) return g;  // smem == 0: unsupported
  }
  g.gb = B <= 8 ? 1 : (num_sms / g.gu >= 2 ? 2 : 1);
  g.bc = (B + g.gb - 1) / g.gb;
  g.gb = (B + g.bc - 1) / g.bc;
  const GruSmem L = gru_layout(Ds, g.units, g.bc);
  g.smem = L.total <= 220 * 1024 ? L.total : 0;
  if (static_cast<long long>(L.chunk) * g.units > static_cast<long long>(kGatePairsPerThread) * kGruThreads) g.smem = 0;
  if (L.mt > kMaxMt || L.chunk / 8 > kMaxNt) g.smem = 0;
  return g;
}

template <bool kTable, bool kWide>
static cudaError_t launch_gru_t(const GruParams& p, const GruPlan& plan, cudaStream_t stream, bool pdl) {
  {
    const cudaError_t e =
        ensure_smem_attr(reinterpret_cast<const void*>(gru_kernel<kTable, kWide>), plan.smem, true);
    if (e != cudaSuccess) return e;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(plan.gu * plan.gb);
  cfg.blockDim = dim3(kGruThreads);
  cfg.dynamicSmemBytes = plan.smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeCooperative;  // every CTA resident at once (state exchange)
  attr[0].val.cooperative = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  // A runtime that refuses the pair gets the cooperative launch alone from then on.
  static std::atomic<bool> pdl_refused{false};
  cfg.numAttrs = (pdl && !pdl_refused) ? 2 : 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, gru_kernel<kTable, kWide>, p);
  if (e != cudaSuccess && cfg.numAttrs == 2) {
    (void)cudaGetLastError();
    pdl_refused = true;
    cfg.numAttrs = 1;
    e = cudaLaunchKernelEx(&cfg, gru_kernel<kTable, kWide>, p);
  }
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_gru(const GruParams& p, const GruPlan& plan, cudaStream_t stream, bool pdl, bool wide) {
  if (plan.smem == 0) return cudaErrorInvalidValue;
  if (wide && p.ids != nullptr) return cudaErrorInvalidValue;  // fused projections share SMs
  if (wide)
    return p.x_table ? launch_gru_t<true, true>(p, plan, stream, pdl) : launch_gru_t<false, true>(p, plan, stream, pdl);
  return p.x_table ? launch_gru_t<true, false>(p, plan, stream, pdl) : launch_gru_t<false, false>(p, plan, stream, pdl);
}

// ---------------------------------------------------------------------------- u finalize
__global__ void __launch_bounds__(256) u_finalize_kernel(const UFinalParams p) {
  // the vocabulary GEMM launched after this kernel may start now: it streams its W_lm segment
  // first and waits for this grid before it loads u
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
  // launched as a programmatic dependent of the W1 GEMM: its partial sums are read below (a
  // no-op otherwise)
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const size_t n = static_cast<size_t>(p.M) * p.R;
  for (size_t e = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < n;
       e += static_cast<size_t>(gridDim.x) * blockDim.x) {
    const int q = static_cast<int>(e % p.R);
    float a = bf_or0(p.b1, q);
    for (int s = 0; s < p.splits; ++s) a += __ldg(p.part + static_cast<size_t>(s) * n + e);
    p.u[e] = __float2bfloat16_rn(a / (1.f + expf(-a)));
  }
}

cudaError_t launch_u_finalize(const UFinalParams& p, cudaStream_t stream, bool pdl) {
  const size_t n = static_cast<size_t>(p.M) * p.R;
  const size_t want = (n + 255) / 256;
  const int blocks = static_cast<int>(want < 1024 ? want : 1024);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(blocks);
  cfg.blockDim = dim3(256);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, u_finalize_kernel, p);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dm
