// rollout_kernels.cuh -- the kernels of the sequential draft loop and the launch helpers that
// instantiate them; included by rollout.cu (greedy and inverse-CDF sampling) and rollout_race.cu
// (the seeded exponential race), so that the two sets of instantiations compile in parallel.
// The sequential draft loop, greedy or sampled (section 4.1.2 and Fig. 3: at inference each
// draft token is chosen from the final logits L_j = L_base_j + W2 u_j + b2 and becomes the
// causal encoder's next input).  The base logits W_lm hidden_j of every position come first from
// the tensor-core GEMM (store mode, fp32); a persistent cooperative kernel then runs the K
// dependent steps, each in three phases separated by grid barriers:
//   A  GRU step: h_j = GRU(emb[t_j], h_{j-1}), one warp per hidden unit (torch.nn.GRU gates);
//   B  u_j = SiLU(W1 [hidden_j ; h_j] + b1), one warp per rank row;
//   C  L_j = base_j + W2 u_j + b2 over the CTA's slice of the vocabulary, with a running max,
//      sum of exp and argmax (equal values: the lowest id) per sequence, reduced per CTA;
// after the third barrier every CTA combines the per-CTA partials itself (the same result
// everywhere), so t_{j+1} needs no fourth barrier.  The sampled loop (t_{j+1} by inverse CDF
// from the caller's uniform) keeps the same barriers: every CTA reads the final logits of the
// CTA whose rows hold the draw and scans them itself.  The seeded sampled loop (kRace, the
// exponential race) takes t_{j+1} = argmax_v L_j[v] + g_j[v] with Gumbel perturbations g from a
// counter-based generator, a draw from softmax(L_j) that runs on the greedy loop's packed keys
// and single barrier per step.  With an input-projection table
// (emb . W_ih^T) phase A reads one row of it instead of projecting emb[t_j]; the resident
// kernel computes u's hidden half W1[:, :H] hidden_j for all positions before the steps.
// Every wait is bounded.
//
// W2 (V x r bf16, 78 MB at the Qwen3 vocabulary) is the operand phase C reads every step.  With
// r <= 256 the resident kernel keeps each CTA's slice of it on chip for the whole block: 512
// rows in the SM's tensor memory (used as storage: written once with tcgen05.st, read with
// tcgen05.ld), as many rows as fit in shared memory, and the few rows left read through L2.
// Wider r uses the streamed kernel, which feeds W2 through a shared-memory ring every step.
#pragma once

#include <math.h>
#include <string.h>

#include <algorithm>

#include "kernels.h"
#include "ptx.cuh"

namespace dm {

constexpr int kRollThreads = 256;                   // the compute warps
constexpr int kRollWarps = kRollThreads / 32;
static_assert(kRollWarps == kRollComputeWarps, "the greedy partials are sized per compute warp");
constexpr int kRollThreadsAll = kRollThreads + 32;  // streamed kernel: + one warp feeding the W2 ring
constexpr int kW2Stages = 6;                        // shared-memory ring of W2 chunks
constexpr int kW2StageBytes = 16 * 1024;            // one chunk: kW2StageBytes / (2 r) rows of W2
constexpr int kRowsPerPass = 4;                     // W2 rows one warp takes at a time
constexpr int kResidentMaxR = 256;                  // r one lane's 8 columns x 32 lanes cover
constexpr int kTmemCols = 512;                      // the whole tensor memory of an SM
// W2 rows in tensor memory: lane quarter q (warps q and q + 4) holds rows 128 q .. 128 q + 127,
// TMEM lane 32 q + l holding columns 8 l .. 8 l + 7 of each (4 32-bit columns per row)
constexpr int kTmemRows = 4 * (kTmemCols / 4);

// ---- tcgen05 forms the phase-C MMA path uses (the GEMM kernels need none of them)
// D[tmem] (+)= A[tmem] * B[smem]^T, bf16 inputs, fp32 accumulation (kind::f16), with A read from
// tensor memory: row m of A in lane m, its K elements packed two to a 32-bit column (the lower
// index in the low half), so one K step of 16 elements spans 8 columns.
__device__ __forceinline__ void tc_mma_bf16_ta(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                               uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Makes this thread's ordinary shared-memory writes visible to the tensor core (async proxy);
// a thread barrier must follow before the MMA that reads them is issued.
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Each thread of the warp reads 4 consecutive 32-bit columns of its TMEM lane.
__device__ __forceinline__ void tc_ld_x4(uint32_t taddr, float (&v)[4]) {
  uint32_t r[4];
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(taddr));
#pragma unroll
  for (int i = 0; i < 4; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ float bf2f(__nv_bfloat16 x) { return __bfloat162float(x); }

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8]) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

__device__ __forceinline__ void bf8(const __nv_bfloat16* p, float (&f)[8]) {
  unpack8(__ldg(reinterpret_cast<const uint4*>(p)), f);
}

// 16 bytes of global memory with an L2 eviction-priority hint
__device__ __forceinline__ uint4 ld16_hint(const void* p, uint64_t pol) {
  uint4 v;
  asm("ld.global.nc.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "l"(p), "l"(pol));
  return v;
}

__device__ __forceinline__ void bf8_hint(const __nv_bfloat16* p, float (&f)[8], uint64_t pol) {
  unpack8(ld16_hint(p, pol), f);
}

// Columns cc .. cc + 7 of rows r0 .. r0 + 3 of a row-major W2 block in shared memory (rows past
// `rows` read as zero).
__device__ __forceinline__ void load_rows(const __nv_bfloat16* sw, int r0, int rows, int R, int cc,
                                          float (&wv)[kRowsPerPass][8]) {
#pragma unroll
  for (int r = 0; r < kRowsPerPass; ++r) {
    if (r0 + r < rows) {
      unpack8(*reinterpret_cast<const uint4*>(sw + static_cast<size_t>(r0 + r) * R + cc), wv[r]);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) wv[r][e] = 0.f;
    }
  }
}

// tensor memory: each thread of the warp writes 16 consecutive 32-bit columns of its lane
__device__ __forceinline__ void tc_st_x16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]), "r"(r[8]),
      "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

__device__ __forceinline__ void tc_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// 4-byte asynchronous copy global -> shared (completes at cp_async_wait_all)
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_all;" ::: "memory");
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// Sums N per-lane values over the warp, N a power of two <= 32, in N - 1 + 5 - log2 N
// shuffles: each round halves the values a lane holds (a lane keeps the upper half when its
// lane bit O is set and receives its partner's matching half).  Lane l ends with the sum of
// value (l >> (5 - log2 N)).
template <int N, int O>
struct ReduceScatter {
  static __device__ __forceinline__ float run(const float (&v)[N]) {
    const bool up = (threadIdx.x & O) != 0;
    float w[N / 2];
#pragma unroll
    for (int i = 0; i < N / 2; ++i) {
      const float send = up ? v[i] : v[i + N / 2];
      const float keep = up ? v[i + N / 2] : v[i];
      w[i] = keep + __shfl_xor_sync(0xffffffffu, send, O);
    }
    return ReduceScatter<N / 2, O / 2>::run(w);
  }
};
template <int O>
struct ReduceScatter<1, O> {
  static __device__ __forceinline__ float run(const float (&v)[1]) {
    float x = v[0];
#pragma unroll
    for (int o = O; o; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
  }
};

__host__ __device__ constexpr int ilog2(int n) { return n <= 1 ? 0 : 1 + ilog2(n / 2); }

// Streamed kernel: rows of the vocabulary one CTA covers, a contiguous run of chunks of `ch`
// rows (ch = the rows of W2 in one ring stage with the head on, 1024 without it).
__host__ __device__ inline int rollout_chunk_rows(int R, int head) {
  return head ? max(1, kW2StageBytes / (2 * R)) : 1024;
}
__host__ __device__ inline int rollout_rows_per_cta(int V, int R, int head, int grid) {
  const int ch = rollout_chunk_rows(R, head);
  const int nchunk_all = (V + ch - 1) / ch;
  return ((nchunk_all + grid - 1) / grid) * ch;
}
// The resident kernel's slices: ceil(V / grid) consecutive rows per CTA.
__host__ __device__ inline int resident_rows_per_cta(int V, int grid) { return (V + grid - 1) / grid; }

// Rows [lo, lo + n) of CTA c: the resident kernel's equal slices, or the streamed kernel's run
// of whole W2 chunks (the same split the kernels take for themselves).
__device__ __forceinline__ void cta_rows(const RolloutParams& p, int c, bool resident, int& lo, int& n) {
  const int V = p.V, grid = static_cast<int>(gridDim.x);
  if (resident) {
    const int rows = resident_rows_per_cta(V, grid);
    lo = min(V, c * rows);
    n = min(V, lo + rows) - lo;
  } else {
    const int ch = rollout_chunk_rows(p.R, p.head);
    const int nall = (V + ch - 1) / ch;
    const int cpc = (nall + grid - 1) / grid;
    const int c_lo = min(nall, c * cpc);
    const int nch = min(nall, c_lo + cpc) - c_lo;
    lo = c_lo * ch;
    n = max(0, min(V, (c_lo + nch) * ch) - lo);
  }
}

// Running (max, sum of exp relative to max, argmax) of a stream of logits.
struct Lse {
  float m, s;
  int i;
};

__device__ __forceinline__ Lse lse_empty() {
  Lse a;
  a.m = -INFINITY;
  a.s = 0.f;
  a.i = 0x7fffffff;
  return a;
}

__device__ __forceinline__ void lse_push(Lse& a, float x, int id) {
  if (x > a.m) {
    a.s = (a.m == -INFINITY ? 0.f : a.s * __expf(a.m - x)) + 1.f;
    a.m = x;
    a.i = id;
  } else {
    a.s += __expf(x - a.m);
  }
}

__device__ __forceinline__ void lse_merge(Lse& a, const Lse& b) {
  if (b.m == -INFINITY) return;
  if (a.m == -INFINITY) { a = b; return; }
  const float m = fmaxf(a.m, b.m);
  const float s = a.s * __expf(a.m - m) + b.s * __expf(b.m - m);
  const int i = (b.m > a.m || (b.m == a.m && b.i < a.i)) ? b.i : a.i;
  a.m = m;
  a.s = s;
  a.i = i;
}

// ---- the exponential race (Gumbel-max) of the seeded sampled loop: t_{j+1} = argmax_v L_j[v] +
//      g_j[v], a draw from softmax(L_j), with g_j[v] = -log(-log(u)) and u from a counter-based
//      generator, Philox-4x32-10 (Salmon, Moraes, Dror and Shaw, SC 2011): counter (v, j, b / 4, 0),
//      key = the 64-bit seed, word b % 4, u = (its top 23 bits + 1/2) / 2^23, in [2^-24, 1 - 2^-24].
__device__ __forceinline__ void philox4x32_10(uint32_t& c0, uint32_t& c1, uint32_t& c2, uint32_t& c3,
                                              uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
    c0 = hi1 ^ c1 ^ k0;
    c1 = lo1;
    c2 = hi0 ^ c3 ^ k1;
    c3 = lo0;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
}

// The four words of vocabulary entry v at step j for sequences 4 q .. 4 q + 3.
__device__ __forceinline__ uint4 race_words(unsigned long long seed, int q, int j, int v) {
  uint32_t c0 = static_cast<uint32_t>(v), c1 = static_cast<uint32_t>(j), c2 = static_cast<uint32_t>(q), c3 = 0u;
  philox4x32_10(c0, c1, c2, c3, static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32));
  return make_uint4(c0, c1, c2, c3);
}

// The perturbation of word w of race_words (sequence 4 q + w).  The inner logarithm keeps full
// precision: -log(u) for u near 1 is as small as 6e-8 and must keep its relative accuracy.  The
// outer one needs absolute accuracy only (its argument lies in [6e-8, 16.7], its value in
// [-2.9, 16.7]), which the fast intrinsic gives to about 1e-6.
__device__ __forceinline__ float race_gumbel(const uint4& x, int w) {
  const uint32_t bits = w == 0 ? x.x : (w == 1 ? x.y : (w == 2 ? x.z : x.w));
  const float u = __fmaf_rn(static_cast<float>(bits >> 9), 0x1p-23f, 0x1p-24f);  // exact
  return -__logf(-logf(u));
}

// The largest perturbed logit seen (equal values: the lowest id), its id and its logit.
struct Pick {
  float k;
  int i;
  float raw;
};

__device__ __forceinline__ Pick pick_empty() {
  Pick a;
  a.k = -INFINITY;
  a.i = 0x7fffffff;
  a.raw = 0.f;
  return a;
}

__device__ __forceinline__ void pick_push(Pick& a, float logit, float g, int id) {
  const float k = logit + g;
  if (k > a.k || (k == a.k && id < a.i)) {
    a.k = k;
    a.i = id;
    a.raw = logit;
  }
}

__device__ __forceinline__ void pick_merge(Pick& a, const Pick& b) {
  if (b.k > a.k || (b.k == a.k && b.i < a.i)) a = b;
}

// Barrier of the compute warps only (the streamed kernel's feeding warp runs on its own).
__device__ __forceinline__ void compute_sync() {
  asm volatile("bar.sync 1, %0;" ::"n"(kRollThreads) : "memory");
}

// Per-warp merge of each sequence's running state, lane 0 of warp w writing red[w][b]; on
// return (after a barrier of the compute warps) red holds every warp's result.
template <int NB>
__device__ __forceinline__ void block_reduce(Lse (&st)[NB], Lse (*red)[kRollMaxB], int B) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    if (b < B) {
#pragma unroll
      for (int o = 16; o; o >>= 1) {
        Lse t;
        t.m = __shfl_xor_sync(0xffffffffu, st[b].m, o);
        t.s = __shfl_xor_sync(0xffffffffu, st[b].s, o);
        t.i = __shfl_xor_sync(0xffffffffu, st[b].i, o);
        lse_merge(st[b], t);
      }
      if (lane == 0) red[warp][b] = st[b];
    }
  }
  compute_sync();
}

// Grid barrier number `n` (0, 1, ...) of the compute warps: every CTA arrives once per barrier.
// Returns false if the wait gave up or the CTA's abort flag is up (status set); the caller
// then stops.  Thread 0 alone reads the flag (which the feeding warp may raise at any time) and
// hands its decision to the compute threads through s_go, so that they all return the same
// value and leave together.
static __device__ bool grid_barrier(unsigned* ctr, unsigned n, int* status, volatile int* fail) {
  __shared__ int s_go;
  compute_sync();
  if (threadIdx.x == 0) {
    // release at GPU scope: every write the CTA made before the barrier above is visible to a
    // CTA that acquires the counter's new value
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(ctr) : "memory");
    const unsigned target = (n + 1) * gridDim.x;
    const long long t0 = clock64();
    while (true) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
      if (v >= target) break;
      if (clock64() - t0 > kWaitCycles) {
        set_status(status, kStatusTimeout);
        *fail = 1;
        break;
      }
      __nanosleep(32);
    }
    s_go = *fail == 0;
  }
  compute_sync();
  return s_go != 0;
}

// Waits until *ctr >= target (acquire at GPU scope): the rows of u phase C needs are written.  The
// same bounded wait and CTA-wide decision as grid_barrier, without an arrival.
static __device__ bool wait_count(const unsigned* ctr, unsigned target, int* status, volatile int* fail) {
  __shared__ int s_go;
  if (threadIdx.x == 0) {
    const long long t0 = clock64();
    while (true) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(ctr) : "memory");
      if (v >= target) break;
      if (clock64() - t0 > kWaitCycles) {
        set_status(status, kStatusTimeout);
        *fail = 1;
        break;
      }
      __nanosleep(32);
    }
    s_go = *fail == 0;
  }
  compute_sync();
  return s_go != 0;
}

// ---- phase A: h_j = GRU(emb[t_j], h_{j-1}) (torch.nn.GRU: gates r|z|n, r multiplies
//      W_hn h + b_hn), one warp per hidden unit q, every sequence.  With an input-projection
//      table the three input-gate sums W_i{r,z,n} emb[t_j] are entries of row t_j of it.
__device__ __forceinline__ void gru_phase(const RolloutParams& p, const int* s_tok, const float* hprev, float* hcur,
                                          int gw, int nwarps, int lane, uint64_t pol) {
  const int B = p.B, H = p.H, Ds = p.Ds;
  for (int q = gw; q < Ds; q += nwarps) {
    for (int b = 0; b < B; ++b) {
      const __nv_bfloat16* x = p.emb + static_cast<size_t>(s_tok[b]) * H;
      float ar = 0.f, az = 0.f, an = 0.f, hr = 0.f, hz = 0.f, hn = 0.f;
      if (p.x_table) {
        if (lane == 0) {  // summed over the warp below with the other lanes' zeros
          const float* xt = p.x_table + static_cast<size_t>(s_tok[b]) * 3 * Ds;
          ar = __ldg(xt + q);
          az = __ldg(xt + Ds + q);
          an = __ldg(xt + 2 * Ds + q);
        }
      } else {
#pragma unroll 4
        for (int c = lane * 8; c < H; c += 256) {
          float xv[8], wr[8], wz[8], wn[8];
          bf8(x + c, xv);
          bf8_hint(p.w_ih + static_cast<size_t>(q) * H + c, wr, pol);
          bf8_hint(p.w_ih + static_cast<size_t>(Ds + q) * H + c, wz, pol);
          bf8_hint(p.w_ih + static_cast<size_t>(2 * Ds + q) * H + c, wn, pol);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            ar += wr[e] * xv[e];
            az += wz[e] * xv[e];
            an += wn[e] * xv[e];
          }
        }
      }
      const float* hp = hprev + static_cast<size_t>(b) * Ds;
#pragma unroll 4
      for (int c = lane * 8; c < Ds; c += 256) {
        float wr[8], wz[8], wn[8];
        bf8_hint(p.w_hh + static_cast<size_t>(q) * Ds + c, wr, pol);
        bf8_hint(p.w_hh + static_cast<size_t>(Ds + q) * Ds + c, wz, pol);
        bf8_hint(p.w_hh + static_cast<size_t>(2 * Ds + q) * Ds + c, wn, pol);
        // written by other CTAs in this launch: read through L2, never a stale L1 line
        const float4 h0 = __ldcg(reinterpret_cast<const float4*>(hp + c));
        const float4 h1 = __ldcg(reinterpret_cast<const float4*>(hp + c + 4));
        const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          hr += wr[e] * hv[e];
          hz += wz[e] * hv[e];
          hn += wn[e] * hv[e];
        }
      }
      ar = warp_sum(ar); az = warp_sum(az); an = warp_sum(an);
      hr = warp_sum(hr); hz = warp_sum(hz); hn = warp_sum(hn);
      if (lane == 0) {
        const float bir = p.b_ih ? bf2f(p.b_ih[q]) : 0.f, biz = p.b_ih ? bf2f(p.b_ih[Ds + q]) : 0.f;
        const float bin = p.b_ih ? bf2f(p.b_ih[2 * Ds + q]) : 0.f;
        const float bhr = p.b_hh ? bf2f(p.b_hh[q]) : 0.f, bhz = p.b_hh ? bf2f(p.b_hh[Ds + q]) : 0.f;
        const float bhn = p.b_hh ? bf2f(p.b_hh[2 * Ds + q]) : 0.f;
        const float r = 1.f / (1.f + expf(-(ar + bir + hr + bhr)));
        const float z = 1.f / (1.f + expf(-(az + biz + hz + bhz)));
        const float n = tanhf(an + bin + r * (hn + bhn));
        hcur[static_cast<size_t>(b) * Ds + q] = (1.f - z) * n + z * __ldcg(hp + q);
      }
    }
  }
}

// Four consecutive bf16 values (8-byte aligned) as floats.
__device__ __forceinline__ void bf4(const __nv_bfloat16* p, float (&f)[4]) {
  const uint2 v = *reinterpret_cast<const uint2*>(p);
  const float2 a = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.x));
  const float2 b = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.y));
  f[0] = a.x; f[1] = a.y; f[2] = b.x; f[3] = b.y;
}

// ---- phase A with the input-projection table, two barriers per step (resident kernel): every
//      CTA computes h_j of every unit and sequence itself, so that no grid barrier follows.  The
//      input-gate sums are row t_j of the table, the recurrent sums W_hh h_{j-1} were computed in
//      the previous step's phase B (gh; none at j = 0), and h_{j-1} is the CTA's own copy in
//      shared memory, updated in place (unit q of h_j needs unit q of h_{j-1} only); four consecutive
//      units per thread, every load of them issued before any arithmetic.
__device__ __forceinline__ void gates_all(const RolloutParams& p, int j, const int* s_tok, float* s_h) {
  const int B = p.B, Ds = p.Ds, D4 = Ds / 4;
  const float* gh = p.gh + static_cast<size_t>((j + 1) & 1) * B * 3 * Ds;  // W_hh h_{j-1}
  for (int e = threadIdx.x; e < B * D4; e += kRollThreads) {
    const int b = e / D4, q = (e - b * D4) * 4;
    const float* xt = p.x_table + static_cast<size_t>(s_tok[b]) * 3 * Ds;
    float4 x[3], hh[3];
    float bi[3][4], bh[3][4];
#pragma unroll
    for (int g = 0; g < 3; ++g) {
      x[g] = __ldg(reinterpret_cast<const float4*>(xt + g * Ds + q));
      // written by other CTAs in this launch: read through L2
      hh[g] = j > 0 ? __ldcg(reinterpret_cast<const float4*>(gh + static_cast<size_t>(b) * 3 * Ds + g * Ds + q))
                    : make_float4(0.f, 0.f, 0.f, 0.f);
      if (p.b_ih) bf4(p.b_ih + g * Ds + q, bi[g]); else bi[g][0] = bi[g][1] = bi[g][2] = bi[g][3] = 0.f;
      if (p.b_hh) bf4(p.b_hh + g * Ds + q, bh[g]); else bh[g][0] = bh[g][1] = bh[g][2] = bh[g][3] = 0.f;
    }
    float* hrow = s_h + static_cast<size_t>(b) * Ds + q;
    const float4 hp = j > 0 ? *reinterpret_cast<const float4*>(hrow) : make_float4(0.f, 0.f, 0.f, 0.f);
    const float xa[3][4] = {{x[0].x, x[0].y, x[0].z, x[0].w}, {x[1].x, x[1].y, x[1].z, x[1].w},
                            {x[2].x, x[2].y, x[2].z, x[2].w}};
    const float ha[3][4] = {{hh[0].x, hh[0].y, hh[0].z, hh[0].w}, {hh[1].x, hh[1].y, hh[1].z, hh[1].w},
                            {hh[2].x, hh[2].y, hh[2].z, hh[2].w}};
    const float hpa[4] = {hp.x, hp.y, hp.z, hp.w};
    float out[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float r = 1.f / (1.f + expf(-(xa[0][i] + bi[0][i] + ha[0][i] + bh[0][i])));
      const float z = 1.f / (1.f + expf(-(xa[1][i] + bi[1][i] + ha[1][i] + bh[1][i])));
      const float n = tanhf(xa[2][i] + bi[2][i] + r * (ha[2][i] + bh[2][i]));
      out[i] = (1.f - z) * n + z * hpa[i];
    }
    *reinterpret_cast<float4*>(hrow) = make_float4(out[0], out[1], out[2], out[3]);
  }
}

// ---- phase B of the one-barrier step: one warp per row of [W1[:, H:]; W_hh] (R + 3 Ds rows;
//      the W_hh rows only when a next step follows), each multiplied with h_j of every sequence
//      from the CTA's shared memory: u_j = SiLU(uh + W1[q, H:] h_j + b1), and gh_j = W_hh h_j for
//      the next step's gates.  A finished row of u is counted in p.ucount (release), which phase C
//      waits for instead of a grid barrier; the gh rows are next needed after the step's partials
//      barrier.  When the grid has more warps than u has rows, warp q < R computes row q of u
//      alone (phase C waits for those) and the other warps take the W_hh rows four at a time;
//      otherwise every warp takes its rows three at a time.  Every weight load of a warp's rows is
//      issued before the arithmetic (Ds <= 1024: at most 4 chunks of 8 columns per lane and row).
// count_u: each finished row of u is counted in p.ucount here (otherwise the caller counts them).
template <int KB, int NR>
__device__ __forceinline__ void ub_rows(const RolloutParams& p, int j, const float* s_h, int row0, int stride,
                                        int rows, int lane, uint64_t pol, bool count_u = true) {
  const int B = p.B, K = p.K, H = p.H, Ds = p.Ds, R = p.R;
  float* gh = p.gh + static_cast<size_t>(j & 1) * B * 3 * Ds;
  constexpr int kCh = 4;
  // step 0: uh comes from every CTA's uh_prologue; lane 0 first waits for all of them (bounded;
  // a timeout leaves the status set), and the warp's loads of uh follow
  if (j == 0 && lane == 0 && row0 < R) {
    const unsigned target = gridDim.x;
    const long long t0 = clock64();
    while (true) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p.uhcount) : "memory");
      if (v >= target) break;
      if (clock64() - t0 > kWaitCycles) {
        set_status(p.status, kStatusTimeout);
        break;
      }
      __nanosleep(32);
    }
  }
  __syncwarp();  // lane 0's acquire orders the other lanes' loads of uh below
  // lane b < B: uh + b1 of sequence b for each u row, loaded with the weights
  float uhb[NR];
#pragma unroll
  for (int k = 0; k < NR; ++k) {
    const int row = row0 + k * stride;
    uhb[k] = (row < R && row < rows && lane < B)
                 ? __ldcg(p.uh + (static_cast<size_t>(lane) * K + j) * R + row) + (p.b1 ? bf2f(p.b1[row]) : 0.f)
                 : 0.f;
  }
  uint4 wraw[NR][kCh];
#pragma unroll
  for (int k = 0; k < NR; ++k) {
    const int row = row0 + k * stride;
    const __nv_bfloat16* w = row >= rows ? nullptr
                             : row < R   ? p.w1 + static_cast<size_t>(row) * (H + Ds) + H
                                         : p.w_hh + static_cast<size_t>(row - R) * Ds;
#pragma unroll
    for (int i = 0; i < kCh; ++i) {
      const int c = lane * 8 + 256 * i;
      wraw[k][i] = (w != nullptr && c < Ds) ? ld16_hint(w + c, pol) : make_uint4(0, 0, 0, 0);
    }
  }
  float acc[NR][KB];
#pragma unroll
  for (int k = 0; k < NR; ++k)
#pragma unroll
    for (int b = 0; b < KB; ++b) acc[k][b] = 0.f;
#pragma unroll
  for (int i = 0; i < kCh; ++i) {
    const int c = lane * 8 + 256 * i;
    if (c >= Ds) break;
    float wv[NR][8];
#pragma unroll
    for (int k = 0; k < NR; ++k) unpack8(wraw[k][i], wv[k]);
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      if (b < B) {
        const float4 h0 = *reinterpret_cast<const float4*>(s_h + static_cast<size_t>(b) * Ds + c);
        const float4 h1 = *reinterpret_cast<const float4*>(s_h + static_cast<size_t>(b) * Ds + c + 4);
#pragma unroll
        for (int k = 0; k < NR; ++k)
          acc[k][b] += wv[k][0] * h0.x + wv[k][1] * h0.y + wv[k][2] * h0.z + wv[k][3] * h0.w +
                       wv[k][4] * h1.x + wv[k][5] * h1.y + wv[k][6] * h1.z + wv[k][7] * h1.w;
      }
    }
  }
#pragma unroll
  for (int k = 0; k < NR; ++k) {
    const int row = row0 + k * stride;
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      if (b < B) {
        const float a = warp_sum(acc[k][b]);
        const float ub = __shfl_sync(0xffffffffu, uhb[k], b);
        if (lane == 0 && row < rows) {
          if (row < R) {
            const float x = a + ub;
            p.u[static_cast<size_t>(b) * R + row] = x / (1.f + expf(-x));
          } else {
            gh[static_cast<size_t>(b) * 3 * Ds + row - R] = a;
          }
        }
      }
    }
    if (count_u && lane == 0 && row < R)  // this row of u_j is written for every sequence
      asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(p.ucount) : "memory");
  }
}

template <int KB>
__device__ __forceinline__ void ub_phase(const RolloutParams& p, int j, const float* s_h, int gw, int nwarps,
                                         int lane, uint64_t pol) {
  const int R = p.R;
  const int rows = R + (j + 1 < p.K ? 3 * p.Ds : 0);
  if (nwarps > R) {
    if (gw < R) {
      // the CTA's warps with a row of u (warps 0 .. nu - 1) meet at a named barrier and one
      // thread counts their nu rows (one atomic per CTA rather than per row)
      const int warp = gw - static_cast<int>(blockIdx.x) * kRollWarps;
      const int nu = min(kRollWarps, R - static_cast<int>(blockIdx.x) * kRollWarps);
      ub_rows<KB, 1>(p, j, s_h, gw, 0, R, lane, pol, false);
      asm volatile("bar.sync 2, %0;" ::"r"(nu * 32) : "memory");
      if (warp == 0 && lane == 0)
        asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p.ucount), "r"(static_cast<unsigned>(nu)) : "memory");
    } else {
      const int n = nwarps - R;
      for (int row0 = gw; row0 < rows; row0 += 4 * n) ub_rows<KB, 4>(p, j, s_h, row0, n, rows, lane, pol);
    }
  } else {
    for (int row0 = gw; row0 < rows; row0 += 3 * nwarps) ub_rows<KB, 3>(p, j, s_h, row0, nwarps, rows, lane, pol);
  }
}

// ---- before the steps (resident kernel): uh[m][q] = W1[q, :H] . hidden_m for every position m
//      = b K + j and rank row q, the half of u's argument that does not depend on the
//      recurrence.  Warp w takes row q = w % R and the positions m = w / R, w / R + G, ...
//      (G = max(1, warps / R)), four at a time, so a W1 row is read once per four positions.
//      The caller then counts its CTA in p.uhcount (release): the two-barrier step reads uh
//      before any grid barrier, so its first phase B acquires that count instead.
static __device__ void uh_prologue(const RolloutParams& p, int gw, int nwarps, int lane, uint64_t pol) {
  const int H = p.H, Ds = p.Ds, R = p.R, M = p.B * p.K;
  const int groups = max(1, nwarps / R);
  for (int pi = gw; pi < R * groups; pi += nwarps) {
    const int q = pi % R, mg = pi / R;
    const __nv_bfloat16* w = p.w1 + static_cast<size_t>(q) * (H + Ds);
    for (int m0 = mg; m0 < M; m0 += 4 * groups) {
      float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 2
      for (int c = lane * 8; c < H; c += 256) {
        float wv[8];
        bf8_hint(w + c, wv, pol);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const int m = m0 + i * groups;
          if (m < M) {
            float xv[8];
            bf8(p.hidden + static_cast<size_t>(m) * H + c, xv);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[i] += wv[e] * xv[e];
          }
        }
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int m = m0 + i * groups;
        const float a = warp_sum(acc[i]);
        if (lane == 0 && m < M) p.uh[static_cast<size_t>(m) * R + q] = a;
      }
    }
  }
}

// ---- phase B: u_j = SiLU(W1 [hidden_j ; h_j] + b1), one warp per rank row q, every sequence.
//      With uh computed before the steps the warp adds uh[b K + j][q] instead of the 4096-long
//      hidden half of the dot.
__device__ __forceinline__ void u_phase(const RolloutParams& p, int j, const float* hcur, int gw, int nwarps,
                                        int lane, uint64_t pol) {
  const int B = p.B, K = p.K, H = p.H, Ds = p.Ds, R = p.R;
  for (int q = gw; q < R; q += nwarps) {
    const __nv_bfloat16* w = p.w1 + static_cast<size_t>(q) * (H + Ds);
    for (int b = 0; b < B; ++b) {
      const __nv_bfloat16* hid = p.hidden + (static_cast<size_t>(b) * K + j) * H;
      const float* hc = hcur + static_cast<size_t>(b) * Ds;
      float acc = 0.f;
      if (p.uh) {
        // written before the steps by other CTAs of this launch (ordered by the grid barriers)
        if (lane == 0) acc = __ldcg(p.uh + (static_cast<size_t>(b) * K + j) * R + q);
      } else {
#pragma unroll 4
        for (int c = lane * 8; c < H; c += 256) {
          float wv[8], xv[8];
          bf8_hint(w + c, wv, pol);
          bf8(hid + c, xv);
#pragma unroll
          for (int e = 0; e < 8; ++e) acc += wv[e] * xv[e];
        }
      }
#pragma unroll 4
      for (int c = lane * 8; c < Ds; c += 256) {
        float wv[8];
        bf8_hint(w + H + c, wv, pol);
        const float4 h0 = __ldcg(reinterpret_cast<const float4*>(hc + c));
        const float4 h1 = __ldcg(reinterpret_cast<const float4*>(hc + c + 4));
        const float hv[8] = {h0.x, h0.y, h0.z, h0.w, h1.x, h1.y, h1.z, h1.w};
#pragma unroll
        for (int e = 0; e < 8; ++e) acc += wv[e] * hv[e];
      }
      acc = warp_sum(acc);
      if (lane == 0) {
        const float a = acc + (p.b1 ? bf2f(p.b1[q]) : 0.f);
        p.u[static_cast<size_t>(b) * R + q] = a / (1.f + expf(-a));
      }
    }
  }
}

// ---- phase C, one pass of a warp: 4 rows x KB sequences.  A lane holds 8 consecutive columns
//      of each row (wv) and of u (ur); the 4 KB dot products are summed over the warp by a
//      reduce-scatter, after which lane `role.idx` holds row role.r of sequence role.b.
struct PassRole {
  int r, b;
  bool rep;  // the one lane of those holding the same value that pushes it
};

template <int KB>
__device__ __forceinline__ PassRole pass_role(int lane) {
  constexpr int kN = kRowsPerPass * KB;
  constexpr int kLogN = ilog2(kN);
  static_assert((1 << kLogN) == kN && kN <= 32, "rows x sequences per pass must be a power of two <= 32");
  const int idx = lane >> (5 - kLogN);
  PassRole role;
  role.r = idx / KB;
  role.b = idx % KB;
  role.rep = (lane & ((32 >> kLogN) - 1)) == 0;
  return role;
}

template <int KB>
__device__ __forceinline__ void pass_fma(const float (&wv)[kRowsPerPass][8], const float (&uv)[KB][8],
                                         float (&dot)[kRowsPerPass * KB]) {
#pragma unroll
  for (int r = 0; r < kRowsPerPass; ++r)
#pragma unroll
    for (int b = 0; b < KB; ++b)
#pragma unroll
      for (int e = 0; e < 8; ++e) dot[r * KB + b] += wv[r][e] * uv[b][e];
}

// Sums the pass over the warp and pushes row (row0 + role.r) of sequence role.b: CTA-local
// row index row0 (for the staged base logits), vocabulary id vid0 + role.r, nvalid rows valid.
// kRace (the exponential race): the perturbed logit of the row also goes into `pick` (step j, seed).
template <int KB, bool kRace>
__device__ __forceinline__ void pass_push(const float (&dot)[kRowsPerPass * KB], const PassRole& role, int nvalid,
                                          int row0, int vid0, float* s_base, int rows_cta, int B, Lse& mine,
                                          Pick& pick, int j, unsigned long long seed) {
  const float d = ReduceScatter<kRowsPerPass * KB, 16>::run(dot);
  if (role.rep && role.r < nvalid && role.b < B) {
    float* x = s_base + role.b * rows_cta + row0 + role.r;
    const float logit = *x + d;
    *x = logit;  // the final logit, for the sampled mode's scan of this CTA's rows
    lse_push(mine, logit, vid0 + role.r);
    if constexpr (kRace) {
      const float g = race_gumbel(race_words(seed, role.b >> 2, j, vid0 + role.r), role.b & 3);
      pick_push(pick, logit, g, vid0 + role.r);
    }
  }
}

// The end of a step, shared by both kernels: per-CTA partials, grid barrier, every CTA's
// combine (thread c loads CTA c's partials, then the same block reduction in every CTA, so all
// reach the same t_{j+1}), the outputs.  Returns false if the barrier gave up.
// Sampled mode, after the combine (s_max / s_lz: the merged max and log-sum of every sequence,
// the same in every CTA): t_{j+1} = the first id whose cumulative probability in id order
// exceeds u_{b,j}.  The CTAs' masses w_c = s_c exp(m_c - max) are scanned in CTA order (their
// slices are consecutive), which names the CTA whose rows hold the crossing; every CTA then
// reads that CTA's final logits (copied to global memory before the partials' barrier) and
// scans them in id order the same way, so every CTA reaches the same token with no further
// barrier.  (If rounding leaves the crossing past those rows, the last row of non-zero mass.)
template <int KB>
__device__ void sample_step(const RolloutParams& p, int j, const float4 (&mine)[KB], const float* lg_all,
                            float* s_stage, int rows_cta, int* s_tok, const float* s_max, const float* s_lz,
                            bool resident) {
  __shared__ float s_T[kRollMaxB], s_off[kRollMaxB];
  __shared__ int s_owner[kRollMaxB], s_pick[kRollMaxB], s_last[kRollMaxB];
  __shared__ float s_wsum[kRollWarps][kRollMaxB];
  const int B = p.B, K = p.K, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int grid = static_cast<int>(gridDim.x);  // <= kRollThreads (checked at launch)
  if (tid < kRollMaxB) { s_owner[tid] = -1; s_off[tid] = 0.f; s_T[tid] = 0.f; }
  // per-CTA masses (thread c: CTA c, whose partial the combine loaded into `mine`) and their
  // inclusive scan in CTA order
  float incl[KB], w[KB];
#pragma unroll
  for (int b = 0; b < KB; ++b) {
    w[b] = 0.f;
    if (b < B && tid < grid) {
      const float4 f = mine[b];
      w[b] = f.x == -INFINITY ? 0.f : f.y * __expf(f.x - s_max[b]);
    }
    incl[b] = w[b];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xffffffffu, incl[b], o);
      if (lane >= o) incl[b] += t;
    }
    if (lane == 31) s_wsum[warp][b] = incl[b];
  }
  compute_sync();
#pragma unroll
  for (int b = 0; b < KB; ++b) {
    if (b >= B) continue;
    float off = 0.f, total = 0.f;
    for (int ww = 0; ww < kRollWarps; ++ww) {
      if (ww < warp) off += s_wsum[ww][b];
    }
    for (int ww = 0; ww < kRollWarps; ++ww) total += s_wsum[ww][b];
    const float prev = __shfl_up_sync(0xffffffffu, incl[b], 1);
    const float excl = (lane == 0 ? 0.f : prev) + off;
    const float inc = incl[b] + off;
    float u = p.uniforms[static_cast<size_t>(b) * K + j];
    u = fminf(fmaxf(u, 0.f), 1.f - 1.2e-7f);  // [0, 1)
    const float T = u * total;
    if (tid < grid && w[b] > 0.f && excl <= T && T < inc) {
      s_owner[b] = tid;
      s_off[b] = excl;
      s_T[b] = T;
    }
  }
  compute_sync();
  for (int b = 0; b < B; ++b) {
    // no claim (no mass anywhere: non-finite logits) falls to CTA 0 and its first row
    const int owner = s_owner[b] >= 0 ? s_owner[b] : 0;
    int o_lo, o_n;
    cta_rows(p, owner, resident, o_lo, o_n);
    const float mx = s_max[b], T = s_T[b];
    float* lg = s_stage + b * rows_cta;  // o_n <= rows_cta: the slices differ only at the tail
    for (int r = tid; r < o_n; r += kRollThreads) lg[r] = __ldcg(lg_all + static_cast<size_t>(b) * p.V + o_lo + r);
    const int per = (o_n + kRollThreads - 1) / kRollThreads;
    const int q0 = min(o_n, tid * per), q1 = min(o_n, q0 + per);
    if (tid == 0) { s_pick[b] = 0x7fffffff; s_last[b] = -1; }
    compute_sync();
    float loc = 0.f;
    for (int r = q0; r < q1; ++r) loc += __expf(lg[r] - mx);
    // exclusive scan of the threads' sums (thread order = row order)
    float inc = loc;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const float t = __shfl_up_sync(0xffffffffu, inc, o);
      if (lane >= o) inc += t;
    }
    if (lane == 31) s_wsum[warp][b] = inc;
    compute_sync();
    float off = s_off[b];
    for (int ww = 0; ww < warp; ++ww) off += s_wsum[ww][b];
    float acc = off + inc - loc;
    int cand = 0x7fffffff, last = -1;
    for (int r = q0; r < q1; ++r) {
      const float e = __expf(lg[r] - mx);
      if (e > 0.f) last = r;
      acc += e;
      if (e > 0.f && acc > T) { cand = r; break; }
    }
    if (cand != 0x7fffffff) atomicMin(&s_pick[b], cand);
    if (last >= 0) atomicMax(&s_last[b], last);
    compute_sync();
    if (tid == 0) {
      const int r = s_pick[b] != 0x7fffffff ? s_pick[b] : max(0, s_last[b]);
      const int tok = o_lo + r;
      s_tok[b] = tok;
      if (blockIdx.x == 0) {
        p.tokens[static_cast<size_t>(b) * K + j] = tok;
        p.logp[static_cast<size_t>(b) * K + j] = lg[r] - mx - s_lz[b];
      }
    }
  }
  compute_sync();
}

// Greedy end of step j (p.best set): the CTA's best row of each sequence as one key -- the step
// (so that no earlier step's key competes), the logit in order-preserving form, then the id
// inverted, so that the largest key over the CTAs is the step's maximum with ties to the lowest
// id (ids below 2^22) -- from two integer warp reductions per warp; thread 0 folds the warps'
// keys into the sequence's slot with one red.max and arrives at the grid barrier.  While the
// other CTAs arrive (before the arrival at the last step, which no later barrier follows), each
// warp reduces its (max, sum of exp) of every sequence and writes it to the step's partials (the
// log-probabilities are merged from them once, after the last step: greedy_logp); then thread 0
// reads the slot.  The slots alternate by step parity: a CTA
// updates step j + 2's only after every CTA has passed step j + 1's barrier, so after every read
// of step j's.  Returns false if the barrier gave up.
// kRace (the exponential race, the seeded sampled loop): the keys are those of the perturbed logits
// (`pick`), and each warp's partial also carries its pick's id and logit, from which greedy_logp
// takes the drawn token's logit.
// s_base_next (the resident kernel): the next step's base logits are copied into it (cp.async)
// while the barrier completes.
template <int KB, bool kRace>
__device__ bool finish_greedy(const RolloutParams& p, int j, Lse (&st)[KB], const Pick (&pick)[KB], int* s_tok,
                              unsigned& nbar, volatile int* s_fail, float* s_base_next, int r_lo, int r_n,
                              int rows_cta) {
  __shared__ unsigned long long s_key[kRollWarps][kRollMaxB];
  __shared__ int s_go;
  const int B = p.B, K = p.K, tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int grid = static_cast<int>(gridDim.x);
  unsigned long long* slot = p.best + (j & 1) * kRollMaxB;
  // each warp's key: (order-preserving value, inverted id) of its best row of every sequence, and
  // (kRace) the logit of that row
  uint32_t whi[KB], wlo[KB];
  float wraw[KB];
#pragma unroll
  for (int b = 0; b < KB; ++b) {
    whi[b] = wlo[b] = 0u;
    wraw[b] = 0.f;
    if (b < B) {
      const float v = kRace ? pick[b].k : st[b].m;
      const int id = kRace ? pick[b].i : st[b].i;
      const bool has = id != 0x7fffffff;
      const uint32_t hi = has ? f32_ord(v) : 0u;
      const uint32_t lo = has ? kGreedyIdMask - static_cast<unsigned>(id) : 0u;
      whi[b] = __reduce_max_sync(0xffffffffu, hi);
      wlo[b] = __reduce_max_sync(0xffffffffu, hi == whi[b] ? lo : 0u);
      if constexpr (kRace) {
        const unsigned ball = __ballot_sync(0xffffffffu, has && hi == whi[b] && lo == wlo[b]);
        wraw[b] = __shfl_sync(0xffffffffu, pick[b].raw, ball ? __ffs(ball) - 1 : 0);
      }
    }
  }
  // each warp's (max, sum of exp) of every sequence, for the log-probabilities
  float4* part = reinterpret_cast<float4*>(p.partials) +
                 (static_cast<size_t>(j) * grid + blockIdx.x) * kRollWarps * kRollMaxB;
  auto write_partials = [&]() {
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      if (b < B) {
        Lse a = st[b];
#pragma unroll
        for (int o = 16; o; o >>= 1) {
          Lse t;
          t.m = __shfl_xor_sync(0xffffffffu, a.m, o);
          t.s = __shfl_xor_sync(0xffffffffu, a.s, o);
          t.i = __shfl_xor_sync(0xffffffffu, a.i, o);
          lse_merge(a, t);
        }
        if (lane == 0) {
          if constexpr (kRace) {
            const int pid = whi[b] != 0u ? static_cast<int>(kGreedyIdMask - wlo[b]) : -1;
            part[warp * kRollMaxB + b] = make_float4(a.m, a.s, __int_as_float(pid), wraw[b]);
          } else {
            part[warp * kRollMaxB + b] = make_float4(a.m, a.s, __int_as_float(a.i), 0.f);
          }
        }
      }
    }
  };
  // the last step's before the arrival (no barrier follows it), the others' while the barrier
  // completes
  const bool last = j + 1 == K;
  if (last) write_partials();
#pragma unroll
  for (int b = 0; b < KB; ++b) {
    // whi == 0: no lane has a row (an order-preserving value is never 0)
    if (b < B && lane == 0)
      s_key[warp][b] = whi[b] != 0u ? (static_cast<unsigned long long>(j + 1) << 54) |
                                          (static_cast<unsigned long long>(whi[b]) << 22) | wlo[b]
                                    : 0ull;
  }
  compute_sync();
  if (tid == 0) {
    for (int b = 0; b < B; ++b) {
      unsigned long long k = 0ull;
      for (int w = 0; w < kRollWarps; ++w) k = s_key[w][b] > k ? s_key[w][b] : k;
      if (k != 0ull) asm volatile("red.relaxed.gpu.global.max.u64 [%0], %1;" ::"l"(slot + b), "l"(k) : "memory");
    }
    // release at GPU scope: this CTA's keys (and its earlier writes) before its arrival
    asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(p.barrier) : "memory");
  }
  if (s_base_next != nullptr && j + 1 < K) {  // phase C has read this step's
    for (int e = tid; e < B * r_n; e += kRollThreads) {
      const int b = e / r_n, r = e - b * r_n;
      cp_async4(s_base_next + b * rows_cta + r, p.base + (static_cast<size_t>(b) * K + j + 1) * p.V + r_lo + r);
    }
  }
  if (!last) write_partials();
  if (tid == 0) {
    const unsigned target = (nbar + 1) * static_cast<unsigned>(grid);
    const long long t0 = clock64();
    while (true) {
      unsigned v;
      asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p.barrier) : "memory");
      if (v >= target) break;
      if (clock64() - t0 > kWaitCycles) {
        set_status(p.status, kStatusTimeout);
        *s_fail = 1;
        break;
      }
      __nanosleep(32);
    }
    s_go = *s_fail == 0;
    if (s_go) {  // every CTA's red.max came before its arrival
      for (int b = 0; b < B; ++b) {
        const unsigned long long key = __ldcg(slot + b);
        const int tok = static_cast<int>(key >> 54) == j + 1
                            ? static_cast<int>(kGreedyIdMask - static_cast<unsigned>(key & kGreedyIdMask))
                            : 0;  // no row with a finite logit anywhere
        s_tok[b] = tok;
        if (blockIdx.x == 0) p.tokens[static_cast<size_t>(b) * K + j] = tok;
      }
    }
  }
  ++nbar;
  compute_sync();
  return s_go != 0;
}

// End of step j: greedy (p.best set), finish_greedy.  Sampled: this CTA's (max, sum exp, argmax)
// per sequence go to the partials, and after a grid barrier every CTA combines all of them and
// draws t_{j+1}.  The partials and the final-logit copies alternate between two buffers by step
// parity: a CTA writes step j + 2's only after every CTA has passed step j + 1's barrier, so
// after every read of step j's (with the correction branch off no other barrier separates
// consecutive steps).
template <int KB, bool kRace>
__device__ __forceinline__ bool finish_step(const RolloutParams& p, int j, Lse (&st)[KB], const Pick (&pick)[KB],
                                            Lse (*s_red)[kRollMaxB], int* s_tok, unsigned& nbar, volatile int* s_fail,
                                            float* s_logit, int r_lo, int r_n, int rows_cta, bool resident) {
  const int B = p.B, V = p.V, tid = threadIdx.x;
  const int grid = static_cast<int>(gridDim.x);
  if (kRace || p.best != nullptr)
    return finish_greedy<KB, kRace>(p, j, st, pick, s_tok, nbar, s_fail, (resident && p.fast_gates) ? s_logit : nullptr,
                                r_lo, r_n, rows_cta);
  float4* part = reinterpret_cast<float4*>(p.partials) + static_cast<size_t>(j & 1) * grid * kRollMaxB;
  block_reduce(st, s_red, B);  // ends with a barrier: every row's final logit is in s_logit
  if (tid < B) {
    Lse a = s_red[0][tid];
    for (int w = 1; w < kRollWarps; ++w) lse_merge(a, s_red[w][tid]);
    part[static_cast<size_t>(blockIdx.x) * kRollMaxB + tid] = make_float4(a.m, a.s, __int_as_float(a.i), 0.f);
  }
  float* lg = p.lg ? p.lg + static_cast<size_t>(j & 1) * B * V : nullptr;
  if (p.uniforms && !resident) {  // this CTA's final logits (the resident kernel wrote them in phase C)
    for (int e = tid; e < B * r_n; e += kRollThreads) {
      const int b = e / r_n, r = e - b * r_n;
      lg[static_cast<size_t>(b) * V + r_lo + r] = s_logit[b * rows_cta + r];
    }
  }
  if (!grid_barrier(p.barrier, nbar++, p.status, s_fail)) return false;
  float4 mine[KB];  // sampled mode: CTA tid's partials (grid <= kRollThreads there)
#pragma unroll
  for (int b = 0; b < KB; ++b) {
    st[b] = lse_empty();
    mine[b] = make_float4(-INFINITY, 0.f, 0.f, 0.f);
  }
  for (int c = tid; c < grid; c += kRollThreads) {
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      if (b < B) {
        const float4 f = __ldcg(part + static_cast<size_t>(c) * kRollMaxB + b);
        if (c == tid) mine[b] = f;
        Lse t;
        t.m = f.x; t.s = f.y; t.i = __float_as_int(f.z);
        lse_merge(st[b], t);
      }
    }
  }
  block_reduce(st, s_red, B);
  __shared__ float s_gmax[kRollMaxB], s_glz[kRollMaxB];
  if (tid < B) {
    Lse a = s_red[0][tid];
    for (int w = 1; w < kRollWarps; ++w) lse_merge(a, s_red[w][tid]);
    s_gmax[tid] = a.m;
    s_glz[tid] = logf(a.s);
  }
  compute_sync();
  sample_step<KB>(p, j, mine, lg, s_logit, rows_cta, s_tok, s_gmax, s_glz, resident);
  return true;
}

// Greedy mode, after the last step: the log-probability of each step's token.  The token is the
// step's argmax, so its log-softmax is -log of the sum of exp(L - max) over the vocabulary, the
// merge of every warp's partials of that step (CTA c takes steps c, c + grid, ...).  Called by
// the compute threads of every CTA after the last step's barrier: every step's partials were
// written before some later arrival at a grid barrier (the last step's before its own).
// kRace: the token is the perturbed maximum, so its log-softmax is its logit - max - log(sum); the
// logit is the one the warp whose pick was the token wrote with its partial.  The token of a
// step before the last is read from the outputs (CTA 0 wrote it before its next arrival); the
// last step's is s_tok, which every CTA holds.
template <int KB, bool kRace>
__device__ void greedy_logp(const RolloutParams& p, Lse (*s_red)[kRollMaxB], const int* s_tok) {
  __shared__ float s_raw[kRollMaxB];
  const int B = p.B, K = p.K, tid = threadIdx.x;
  const int grid = static_cast<int>(gridDim.x);
  const int nw = grid * kRollWarps;
  for (int j = blockIdx.x; j < K; j += grid) {
    const float4* part = reinterpret_cast<const float4*>(p.partials) + static_cast<size_t>(j) * nw * kRollMaxB;
    int tok[KB];
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      tok[b] = -2;
      if (kRace && b < B) tok[b] = j + 1 == K ? s_tok[b] : __ldcg(p.tokens + static_cast<size_t>(b) * K + j);
    }
    if (kRace && tid < B) s_raw[tid] = 0.f;
    compute_sync();
    Lse st[KB];
#pragma unroll
    for (int b = 0; b < KB; ++b) st[b] = lse_empty();
    for (int c = tid; c < nw; c += kRollThreads) {
#pragma unroll
      for (int b = 0; b < KB; ++b) {
        if (b < B) {
          const float4 f = __ldcg(part + static_cast<size_t>(c) * kRollMaxB + b);
          Lse t;
          t.m = f.x; t.s = f.y; t.i = __float_as_int(f.z);
          lse_merge(st[b], t);
          if (kRace && __float_as_int(f.z) == tok[b]) s_raw[b] = f.w;  // the one warp that held the token
        }
      }
    }
    block_reduce(st, s_red, B);
    if (tid < B) {
      Lse a = s_red[0][tid];
      for (int w = 1; w < kRollWarps; ++w) lse_merge(a, s_red[w][tid]);
      p.logp[static_cast<size_t>(tid) * K + j] = kRace ? s_raw[tid] - a.m - logf(a.s) : -logf(a.s);
    }
    compute_sync();  // s_red is read before the next step's reduction overwrites it
  }
}

// Base logits + b2 of step j for this CTA's rows [r_lo, r_lo + r_n), staged in shared memory.
__device__ __forceinline__ void stage_base(const RolloutParams& p, int j, int r_lo, int r_n, int rows_cta,
                                           float* s_base) {
  const int B = p.B, K = p.K, V = p.V;
  for (int e = threadIdx.x; e < B * r_n; e += kRollThreads) {
    const int b = e / r_n, r = e - b * r_n;
    s_base[b * rows_cta + r] = __ldcg(p.base + (static_cast<size_t>(b) * K + j) * V + r_lo + r) +
                               (p.b2 ? bf2f(p.b2[r_lo + r]) : 0.f);
  }
}

// ---- phase C, resident kernel: a pass covers 32 / KB rows x KB sequences, so that after the
//      reduce-scatter every lane holds one finished dot product (row lane / KB, sequence
//      lane % KB); rows come in groups of up to 8, each a 16-byte load per lane.
template <int KB>
struct WidePass {
  static constexpr int kRows = 32 / KB;
  static constexpr int kGroup = kRows < 8 ? kRows : 8;
};

template <int KB, int G>
__device__ __forceinline__ void group_fma(const uint4 (&raw)[G], int r_in_pass, const float (&ur)[KB][8],
                                          float (&dot)[32]) {
#pragma unroll
  for (int r = 0; r < G; ++r) {
    float w[8];
    unpack8(raw[r], w);
#pragma unroll
    for (int b = 0; b < KB; ++b)
#pragma unroll
      for (int e = 0; e < 8; ++e) dot[(r_in_pass + r) * KB + b] += w[e] * ur[b][e];
  }
}

// After the reduce-scatter each lane holds one finished dot product: the logit of its row and
// sequence is pushed into the lane's running (max, sum, argmax).  glg (sampled mode): the
// step's [B, V] buffer of final logits, which every CTA reads the draw's CTA's rows from;
// nullptr in greedy mode.
// kRace: g is the lane's perturbation (lane_gumbel), computed before the dot products it waits for.
template <int KB, bool kRace>
__device__ __forceinline__ void wide_push(const float (&dot)[32], int lane, int nvalid, int row0, int vid0,
                                          const float* s_base, const float* s_b2, int rows_cta, int B, Lse& mine,
                                          float* glg, int V, Pick& pick, float g) {
  const float d = ReduceScatter<32, 16>::run(dot);
  const int r = lane / KB, b = lane % KB;
  if (r < nvalid && b < B) {
    const float logit = s_base[b * rows_cta + row0 + r] + s_b2[row0 + r] + d;
    if (glg) glg[static_cast<size_t>(b) * V + vid0 + r] = logit;
    lse_push(mine, logit, vid0 + r);
    if constexpr (kRace) pick_push(pick, logit, g, vid0 + r);
  }
}

// The perturbation wide_push gives `lane` (row vid0 + lane / KB, sequence lane % KB) at step j;
// it depends on no data, so it is computed while the row's loads are in flight.
template <int KB, bool kRace>
__device__ __forceinline__ float lane_gumbel(unsigned long long seed, int lane, int j, int vid0) {
  if constexpr (!kRace) {
    return 0.f;
  } else {
    const int b = lane % KB;
    return race_gumbel(race_words(seed, b >> 2, j, vid0 + lane / KB), b & 3);
  }
}

// ================================================================ resident kernel (r <= 256)

// Phase C on the tensor cores (kMma).  A CTA's W2 rows form 128-row blocks: the first mma_tb in
// tensor memory as the MMA's A operand (row in lane, K along the columns), the next mma_sb in
// shared memory as 128-byte swizzled K-major tiles (loaded once by TMA); rows past those blocks
// are read through L2 on the CUDA cores as in the other layout.  u_j is the B operand with
// N = 16 rows: row 2b holds bf16(u_j[b]) and row 2b + 1 the bf16 of what that rounding left out,
// so that D[:, 2b] + D[:, 2b + 1] is W2 u_j to about 2^-16 relative (fp32 accumulation, the
// precision the CUDA-core layout keeps u in).  Each block's MMAs go into its own 16 columns of D,
// issued by one thread of its own warp; the epilogue adds the staged base logit and b2 of each row.
// Tensor memory (512 columns): A block i at columns [i r/2, (i+1) r/2), D of block i at
// mma_tb r/2 + 16 i.  Shared memory from a 1024-byte boundary: the A blocks (r/64 tiles of
// 128 rows x 64 columns each), the B operand (r/64 tiles of 16 rows x 64 columns), then u, the
// base logits, b2 and h as in the other layout.
constexpr int kMmaBopTileBytes = 16 * 128;   // B operand: 16 rows x 64 bf16 columns
constexpr int kMmaTileBytes = 128 * 128;     // A block: 128 rows x 64 bf16 columns
constexpr int kMmaMaxL2Rows = 384;           // at most this many rows a CTA reads through L2

// Byte offset of element (n, k) of the B operand in its 128-byte swizzled K-major tiles: tile
// k / 64, 8-row groups 1024 bytes apart, 16-byte chunk c of row r stored at chunk c ^ (r % 8).
__device__ __forceinline__ uint32_t bop_offset(int n, int k) {
  const int kin = k & 63, r = n & 7;
  return static_cast<uint32_t>((k >> 6) * kMmaBopTileBytes + (n >> 3) * 1024 + r * 128 + (((kin >> 3) ^ r) << 4) +
                               (kin & 7) * 2);
}

template <int KB, bool kMma, bool kRace>
__global__ void __launch_bounds__(kRollThreads, 1)
    rollout_resident_kernel(const RolloutParams p, const __grid_constant__ CUtensorMap tm_w2) {
  static_assert(!kMma || KB <= 2, "the B operand holds two rows per sequence in its 16");
  const int B = p.B, K = p.K, V = p.V, R = p.R;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = gridDim.x * kRollWarps;
  const int gw = blockIdx.x * kRollWarps + warp;
  // this CTA's rows: [r_lo, r_lo + r_n); the first n_t in tensor memory, the next n_s in
  // shared memory, the last n_g read from global memory (L2) every step
  const int rows_cta = resident_rows_per_cta(V, gridDim.x);
  const int r_lo = min(V, static_cast<int>(blockIdx.x) * rows_cta);
  const int r_n = min(V, r_lo + rows_cta) - r_lo;
  const int n_blk = kMma ? p.mma_tb + p.mma_sb : 0;
  const int n_t = kMma ? min(r_n, 128 * p.mma_tb) : min(r_n, kTmemRows);
  const int n_s = kMma ? max(0, min(r_n, 128 * n_blk) - n_t) : min(r_n - n_t, p.smem_rows);
  const int n_g = r_n - n_t - n_s;
  extern __shared__ __align__(128) uint8_t s_dyn[];
  uint8_t* s_al = kMma ? reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(s_dyn) + 1023) &
                                                    ~static_cast<uintptr_t>(1023))
                       : s_dyn;
  uint8_t* s_bop = s_al + static_cast<size_t>(kMma ? p.mma_sb : 0) * (R / 64) * kMmaTileBytes;  // kMma
  __nv_bfloat16* s_w2 = reinterpret_cast<__nv_bfloat16*>(s_dyn);  // [smem_rows][R] (!kMma)
  float* s_u = kMma ? reinterpret_cast<float*>(s_bop + (R / 64) * kMmaBopTileBytes)
                    : reinterpret_cast<float*>(s_dyn + static_cast<size_t>(p.smem_rows) * R * 2);  // [B][R]
  float* s_base = s_u + B * R;                                                          // [B][rows_cta]
  float* s_b2 = s_base + B * rows_cta;                                                  // [rows_cta]
  // [B][Ds] h_j of every sequence (two-barrier steps only), 16-byte aligned for vector reads
  float* s_h = reinterpret_cast<float*>((reinterpret_cast<uintptr_t>(s_b2 + rows_cta) + 15) & ~static_cast<uintptr_t>(15));
  __shared__ __align__(8) uint64_t s_fill;  // the shared-memory rows landed
  __shared__ __align__(8) uint64_t s_mma;   // kMma: this step's MMAs completed
  __shared__ uint32_t s_tmem;
  __shared__ int s_tok[kRollMaxB];
  __shared__ Lse s_red[kRollWarps][kRollMaxB];
  __shared__ int s_fail;
  if (tid == 0) {
    s_fail = 0;
    mbar_init(&s_fill, 1);
    mbar_init(&s_mma, kMma ? max(1, min(n_blk, kRollWarps)) : 1);  // one commit per issuing thread
    fence_mbar_init();
  }
  if (warp == 0) {
    tmem_alloc(&s_tmem, kTmemCols);
    tmem_relinquish();
  }
  if (tid < B) s_tok[tid] = p.anchors[tid];
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tbase = s_tmem;
  const int dcol0 = kMma ? p.mma_tb * (R / 2) : 0;  // first D column
  // shared-memory rows were requested (the TMA tiles of the last CTAs may lie past V: zero fill)
  const bool fill_any = kMma ? p.mma_sb > 0 : n_s > 0;
  int mma_steps = 0;  // thread 0: steps whose MMAs were issued (their completion is awaited)
  bool tokens_ok = true;
  for (int b = 0; b < B; ++b)
    if (s_tok[b] < 0 || s_tok[b] >= V) tokens_ok = false;  // the same ids in every CTA
  bool fill_issued = false;
  if (!tokens_ok) {
    if (tid == 0) set_status(p.status, kStatusBadToken);
  } else {
    // ---- fill: shared-memory rows by bulk copies (one barrier, pieces of at most 64 KB), or
    //      with the MMA layout the A blocks' swizzled tiles by TMA
    if (tid == 0) {
      if constexpr (kMma) {
        const int tiles = R / 64;
        mbar_arrive_expect_tx(&s_fill, static_cast<uint32_t>(p.mma_sb * tiles * kMmaTileBytes));
        const uint64_t pol = l2_policy_evict_first();
        for (int sb = 0; sb < p.mma_sb; ++sb)
          for (int a = 0; a < tiles; ++a)
            tma_load_2d(s_al + static_cast<size_t>(sb * tiles + a) * kMmaTileBytes, &tm_w2, &s_fill, 64 * a,
                        r_lo + 128 * (p.mma_tb + sb), pol);
      } else {
        const uint32_t bytes = static_cast<uint32_t>(n_s) * R * 2;
        mbar_arrive_expect_tx(&s_fill, bytes);
        const uint8_t* src = reinterpret_cast<const uint8_t*>(p.w2 + static_cast<size_t>(r_lo + n_t) * R);
        for (uint32_t off = 0; off < bytes; off += 64 * 1024) {
          const uint32_t n = min(bytes - off, 64u * 1024u);
          bulk_load(reinterpret_cast<uint8_t*>(s_w2) + off, src + off, n, &s_fill, l2_policy_evict_first());
        }
      }
    }
    fill_issued = true;
    // ---- u's hidden halves while the bulk copies land (read by phase B after a grid barrier)
    if (p.uh) {
      uh_prologue(p, gw, nwarps, lane, l2_policy_evict_normal());
      compute_sync();  // one count per CTA: every warp's share of uh is written
      if (tid == 0 && p.uhcount) asm volatile("red.release.gpu.global.add.u32 [%0], 1;" ::"l"(p.uhcount) : "memory");
    }
    const int q = warp & 3, half = warp >> 2;
    const uint32_t tq = tbase + (static_cast<uint32_t>(32 * q) << 16);
    const uint64_t pol_once = l2_policy_evict_first();
    if constexpr (kMma) {
      // ---- fill: the tensor-memory A blocks.  Thread l of warp w writes lane 32 (w % 4) + l, the
      //      row 128 i + 32 (w % 4) + l of block i in its natural order (two elements a column);
      //      warps w and w + 4 take the two halves of the block's r / 2 columns.  Rows past the
      //      CTA's slice are zero.
      const int cols = R / 2, hc = R / 4;  // hc, the columns of a half: a multiple of 16
      for (int i = 0; i < p.mma_tb; ++i) {
        const int row = 128 * i + 32 * q + lane;
        const bool valid = row < r_n;
        const __nv_bfloat16* src = p.w2 + static_cast<size_t>(r_lo + (valid ? row : 0)) * R + 2 * half * hc;
        for (int c0 = 0; c0 < hc; c0 += 16) {
          uint32_t r[16];
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            const uint4 x = valid ? ld16_hint(src + 2 * c0 + 8 * v, pol_once) : make_uint4(0, 0, 0, 0);
            r[4 * v] = x.x;
            r[4 * v + 1] = x.y;
            r[4 * v + 2] = x.z;
            r[4 * v + 3] = x.w;
          }
          tc_st_x16(tq + static_cast<uint32_t>(i * cols + half * hc + c0), r);
        }
      }
      // the B operand's rows 2B .. 15 stay zero
      for (int e = tid; e < (R / 64) * kMmaBopTileBytes / 16; e += kRollThreads)
        reinterpret_cast<uint4*>(s_bop)[e] = make_uint4(0, 0, 0, 0);
    } else {
      // ---- fill: tensor-memory rows.  Warp w writes lane quarter q = w % 4, rows 64 (w / 4) ..
      //      64 (w / 4) + 63 of the quarter's 128, 4 rows (16 columns) per store.
#pragma unroll 1
      for (int g0 = 0; g0 < 64; g0 += 32) {
        uint4 v[32];  // 8 groups of 4 rows in flight
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const int row = 128 * q + 64 * half + g0 + i;  // CTA-local
          v[i] = (row < n_t && lane * 8 < R)
                     ? ld16_hint(p.w2 + static_cast<size_t>(r_lo + row) * R + lane * 8, pol_once)
                     : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int gi = 0; gi < 8; ++gi) {
          const uint32_t r[16] = {v[4 * gi].x,     v[4 * gi].y,     v[4 * gi].z,     v[4 * gi].w,
                                  v[4 * gi + 1].x, v[4 * gi + 1].y, v[4 * gi + 1].z, v[4 * gi + 1].w,
                                  v[4 * gi + 2].x, v[4 * gi + 2].y, v[4 * gi + 2].z, v[4 * gi + 2].w,
                                  v[4 * gi + 3].x, v[4 * gi + 3].y, v[4 * gi + 3].z, v[4 * gi + 3].w};
          tc_st_x16(tq + static_cast<uint32_t>(4 * (64 * half + g0 + 4 * gi)), r);
        }
      }
    }
    tc_wait_st();  // (!kMma) a warp reads back only what it wrote itself; (kMma) the MMA reads
                   // the A blocks after the step's first barrier
    for (int r = tid; r < r_n; r += kRollThreads) s_b2[r] = p.b2 ? bf2f(p.b2[r_lo + r]) : 0.f;

    constexpr int kRows = WidePass<KB>::kRows, kGroup = WidePass<KB>::kGroup;
    const uint64_t pol_ab = l2_policy_evict_normal();
    const uint64_t pol_rest = l2_policy_evict_last();
    unsigned nbar = 0;
    for (int j = 0; j < K; ++j) {
      const float* hprev = p.h + static_cast<size_t>((j + 1) & 1) * B * p.Ds;  // h_{j-1} (zeros at j = 0)
      float* hcur = p.h + static_cast<size_t>(j & 1) * B * p.Ds;
      // this step's base logits for the CTA's rows: asynchronous copies that land during A and B
      // (greedy two-barrier step: issued by the previous step's finish, from step 1 on)
      if (j == 0 || p.best == nullptr || !p.fast_gates) {
        for (int e = tid; e < B * r_n; e += kRollThreads) {
          const int b = e / r_n, r = e - b * r_n;
          cp_async4(s_base + b * rows_cta + r, p.base + (static_cast<size_t>(b) * K + j) * V + r_lo + r);
        }
      }
      if (p.fast_gates) {
        gates_all(p, j, s_tok, s_h);
        compute_sync();  // h_j of every sequence in this CTA's shared memory
        ub_phase<KB>(p, j, s_h, gw, nwarps, lane, pol_ab);
        // phase C needs u_j only: every one of its R rows counted, not a grid barrier
        if (!wait_count(p.ucount, static_cast<unsigned>(R) * (j + 1), p.status, &s_fail)) break;
      } else {
        gru_phase(p, s_tok, hprev, hcur, gw, nwarps, lane, pol_ab);
        if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) break;
        u_phase(p, j, hcur, gw, nwarps, lane, pol_ab);
        if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) break;
      }
      for (int e = tid; e < B * R; e += kRollThreads) {
        const float v = __ldcg(p.u + e);
        s_u[e] = v;
        if constexpr (kMma) {  // u_j as the B operand: rows 2b (bf16 of u) and 2b + 1 (the rest)
          const int b = e / R, k = e - b * R;
          const __nv_bfloat16 hi = __float2bfloat16_rn(v);
          const __nv_bfloat16 lo = __float2bfloat16_rn(v - __bfloat162float(hi));
          *reinterpret_cast<__nv_bfloat16*>(s_bop + bop_offset(2 * b, k)) = hi;
          *reinterpret_cast<__nv_bfloat16*>(s_bop + bop_offset(2 * b + 1, k)) = lo;
        }
      }
      if constexpr (kMma) {
        fence_proxy_async_smem();  // the B operand, for the tensor core
        tc_fence_before();
      }
      cp_async_wait_all();
      compute_sync();
      if constexpr (kMma) {
        // ---- lane 0 of warp 7 - (i % 8) issues block i's MMAs, and each issuing thread commits
        //      once (a thread issues a K step in about 150 cycles, so the blocks go out in
        //      parallel); the epilogue below waits for every commit
        if (lane == 0 && kRollWarps - 1 - warp < n_blk) {
          bool ok = true;
          if (j == 0 && fill_any) ok = mbar_wait(&s_fill, 0, &s_fail, p.status);
          if (ok) {
            tc_fence_after();
            constexpr uint32_t kIdesc = idesc_bf16_f32(128, 16);
            const uint64_t bd0 = smem_desc_sw128(smem_u32(s_bop));
            const uint32_t ab_a = smem_u32(s_al);
            const int ksteps = R / 16;
            for (int i = kRollWarps - 1 - warp; i < n_blk; i += kRollWarps) {
              const uint32_t d = tbase + static_cast<uint32_t>(dcol0 + 16 * i);
              if (i < p.mma_tb) {
                const uint32_t a0 = tbase + static_cast<uint32_t>(i * (R / 2));
#pragma unroll 4
                for (int kk = 0; kk < ksteps; ++kk)
                  tc_mma_bf16_ta(d, a0 + static_cast<uint32_t>(8 * kk),
                                 bd0 + static_cast<uint64_t>((kk >> 2) * (kMmaBopTileBytes >> 4) + 2 * (kk & 3)), kIdesc,
                                 kk > 0 ? 1u : 0u);
              } else {
                const uint64_t ad0 =
                    smem_desc_sw128(ab_a + static_cast<uint32_t>((i - p.mma_tb) * (R / 64) * kMmaTileBytes));
#pragma unroll 4
                for (int kk = 0; kk < ksteps; ++kk)
                  tc_mma_bf16(d, ad0 + static_cast<uint64_t>((kk >> 2) * (kMmaTileBytes >> 4) + 2 * (kk & 3)),
                              bd0 + static_cast<uint64_t>((kk >> 2) * (kMmaBopTileBytes >> 4) + 2 * (kk & 3)), kIdesc,
                              kk > 0 ? 1u : 0u);
              }
            }
            tc_commit(&s_mma);
          } else {
            mbar_arrive(&s_mma);  // nothing issued: the epilogue's wait ends (the step fails)
          }
        }
        if (tid == 0) ++mma_steps;
      }
      float ur[KB][8];  // u at this lane's 8 columns (zero past r)
#pragma unroll
      for (int b = 0; b < KB; ++b)
#pragma unroll
        for (int e = 0; e < 8; ++e) ur[b][e] = (b < B && lane * 8 < R) ? s_u[(b < B && lane * 8 < R) ? b * R + lane * 8 + e : 0] : 0.f;
      Lse mine = lse_empty();
      Pick pmine = pick_empty();  // kRace: the perturbed maximum of the same rows
      float* glg = p.uniforms ? p.lg + static_cast<size_t>(j & 1) * B * V : nullptr;  // sampled: final logits
      // rows read through L2 first (the longest latency): one group of rows per warp at a time.
      // kRace: a pass has kGroup x KB (row, sequence) lanes, so one perturbation per lane serves
      // kBatch passes (lane l computes lane l % kPerPass's of pass l / kPerPass and hands it over)
      constexpr int kPerPass = kGroup * KB;
      constexpr int kBatch = 32 / kPerPass;
      float gbatch = 0.f;
      int pass = 0;
      for (int r0 = warp * kGroup; r0 < n_g; r0 += kRollWarps * kGroup, ++pass) {
        uint4 raw[kGroup];
#pragma unroll
        for (int r = 0; r < kGroup; ++r)
          raw[r] = (r0 + r < n_g && lane * 8 < R)
                       ? ld16_hint(p.w2 + static_cast<size_t>(r_lo + n_t + n_s + r0 + r) * R + lane * 8, pol_rest)
                       : make_uint4(0, 0, 0, 0);
        float pg = 0.f;
        if constexpr (kRace) {
          if (pass % kBatch == 0) {
            const int li = lane % kPerPass;
            gbatch = lane_gumbel<KB, kRace>(p.seed, li, j,
                                            r_lo + n_t + n_s + r0 + (lane / kPerPass) * kRollWarps * kGroup);
          }
          pg = __shfl_sync(0xffffffffu, gbatch, (pass % kBatch) * kPerPass + lane % kPerPass);
        }
        float dot[32] = {};
        group_fma<KB, kGroup>(raw, 0, ur, dot);
        wide_push<KB, kRace>(dot, lane, min(kGroup, n_g - r0), n_t + n_s + r0, r_lo + n_t + n_s + r0, s_base, s_b2,
                             rows_cta, B, mine, glg, V, pmine, pg);
      }
      Lse st[KB];
      Pick pst[KB];
#pragma unroll
      for (int b = 0; b < KB; ++b) {
        st[b] = lse_empty();
        pst[b] = pick_empty();
      }
      if constexpr (kMma) {
        // ---- epilogue: warp w reads lane quarter w % 4 of every other D block (warps w and
        //      w + 4 alternate), one row per thread, in increasing row order
        // one row of block i: its logits from the accumulator (g0, g1: kRace, the row's
        // perturbations for sequences 0 and 1)
        auto epi_row = [&](int i, float g0, float g1) {
          float d[4];
          tc_ld_x4(tq + static_cast<uint32_t>(dcol0 + 16 * i), d);
          tc_wait_ld();
          const int row = 128 * i + 32 * q + lane;
          if (row < r_n) {
#pragma unroll
            for (int b = 0; b < KB; ++b) {
              if (b < B) {
                const float logit = s_base[b * rows_cta + row] + s_b2[row] + (d[2 * b] + d[2 * b + 1]);
                if (glg) glg[static_cast<size_t>(b) * V + r_lo + row] = logit;
                lse_push(st[b], logit, r_lo + row);
                if constexpr (kRace) pick_push(pst[b], logit, b == 0 ? g0 : g1, r_lo + row);
              }
            }
          }
        };
        // kRace: the perturbations of this thread's first kEpiRows rows, computed while the MMAs
        // run (they depend on no data) as independent chains, without branches (a row past the
        // CTA's blocks costs one unused chain); KB <= 2, so one counter serves the row
        constexpr int kEpiRows = 4;
        float gq[kEpiRows][2];
#pragma unroll
        for (int t = 0; t < kEpiRows; ++t) {
          gq[t][0] = gq[t][1] = 0.f;
          if constexpr (kRace) {
            const uint4 x = race_words(p.seed, 0, j, r_lo + 128 * (half + 2 * t) + 32 * q + lane);
            gq[t][0] = race_gumbel(x, 0);
            gq[t][1] = KB > 1 ? race_gumbel(x, 1) : 0.f;
          }
        }
        const bool done = mbar_wait(&s_mma, static_cast<uint32_t>(j & 1), &s_fail, p.status);
        if (__all_sync(0xffffffffu, done)) {  // warp-uniform: the loads are .sync.aligned
          tc_fence_after();
#pragma unroll
          for (int t = 0; t < kEpiRows; ++t)
            if (half + 2 * t < n_blk) epi_row(half + 2 * t, gq[t][0], gq[t][1]);
          for (int i = half + 2 * kEpiRows; i < n_blk; i += 2) {  // more than 8 blocks: perturbed here
            float g0 = 0.f, g1 = 0.f;
            if constexpr (kRace) {
              const uint4 x = race_words(p.seed, 0, j, r_lo + 128 * i + 32 * q + lane);
              g0 = race_gumbel(x, 0);
              g1 = KB > 1 ? race_gumbel(x, 1) : 0.f;
            }
            epi_row(i, g0, g1);
          }
        }
        tc_fence_before();  // every read of D before the next step's MMAs overwrite it
      } else {
        // rows in tensor memory: this warp's 64 rows of its lane quarter, 8 rows (32 columns) a load
        for (int rho0 = 64 * half; rho0 < 64 * half + 64; rho0 += kRows) {
          const int row0 = 128 * q + rho0;
          if (row0 >= n_t) break;
          const float pg = lane_gumbel<KB, kRace>(p.seed, lane, j, r_lo + row0);
          float dot[32] = {};
#pragma unroll
          for (int g = 0; g < kRows; g += kGroup) {
            uint4 raw[kGroup];
            if (kGroup == 8) {
              float t[32];
              tc_ld_x32(tq + static_cast<uint32_t>(4 * (rho0 + g)), t);
              tc_wait_ld();
#pragma unroll
              for (int r = 0; r < kGroup; ++r)
                raw[r] = make_uint4(__float_as_uint(t[4 * r]), __float_as_uint(t[4 * r + 1]),
                                    __float_as_uint(t[4 * r + 2]), __float_as_uint(t[4 * r + 3]));
            } else {
              float t[16];
              tc_ld_x16(tq + static_cast<uint32_t>(4 * (rho0 + g)), t);
              tc_wait_ld();
#pragma unroll
              for (int r = 0; r < kGroup; ++r)
                raw[r] = make_uint4(__float_as_uint(t[4 * r]), __float_as_uint(t[4 * r + 1]),
                                    __float_as_uint(t[4 * r + 2]), __float_as_uint(t[4 * r + 3]));
            }
            group_fma<KB, kGroup>(raw, g, ur, dot);
          }
          wide_push<KB, kRace>(dot, lane, n_t - row0, row0, r_lo + row0, s_base, s_b2, rows_cta, B, mine, glg, V, pmine,
                               pg);
        }
        // rows in shared memory (landed before the first step's phase C)
        bool filled = true;
        if (j == 0 && n_s > 0) filled = mbar_wait(&s_fill, 0, &s_fail, p.status);
        if (__all_sync(0xffffffffu, filled && !s_fail)) {  // warp-uniform: the passes shuffle
          for (int r0 = warp * kRows; r0 < n_s; r0 += kRollWarps * kRows) {
            const float pg = lane_gumbel<KB, kRace>(p.seed, lane, j, r_lo + n_t + r0);
            float dot[32] = {};
#pragma unroll
            for (int g = 0; g < kRows; g += kGroup) {
              uint4 raw[kGroup];
#pragma unroll
              for (int r = 0; r < kGroup; ++r)
                raw[r] = (r0 + g + r < n_s && lane * 8 < R)
                             ? *reinterpret_cast<const uint4*>(
                                   s_w2 + ((r0 + g + r < n_s && lane * 8 < R) ? static_cast<size_t>(r0 + g + r) * R +
                                                                                     lane * 8
                                                                               : 0))
                             : make_uint4(0, 0, 0, 0);
              group_fma<KB, kGroup>(raw, g, ur, dot);
            }
            wide_push<KB, kRace>(dot, lane, n_s - r0, n_t + r0, r_lo + n_t + r0, s_base, s_b2, rows_cta, B, mine, glg,
                                 V, pmine, pg);
          }
        }
      }
      // the L2 rows (and, in the CUDA-core layout, every row) of this lane's sequence
      // lane % KB; ties go to the lower id
#pragma unroll
      for (int b = 0; b < KB; ++b) {
        if (b == lane % KB) {
          lse_merge(st[b], mine);
          if constexpr (kRace) pick_merge(pst[b], pmine);
        }
      }
      if (!finish_step<KB, kRace>(p, j, st, pst, s_red, s_tok, nbar, &s_fail, s_base, r_lo, r_n, rows_cta, true)) break;
      if (j + 1 == K && (kRace || p.best)) greedy_logp<KB, kRace>(p, s_red, s_tok);
    }
  }
  // ---- teardown: the asynchronous copies have landed (the fill: bounded), the MMAs are done
  //      (bounded), tensor memory is released
  cp_async_wait_all();
  if (tid == 0 && fill_issued && fill_any) {
    const long long t0 = clock64();
    while (!mbar_try_wait(&s_fill, 0))
      if (clock64() - t0 > kWaitCycles) break;
  }
  if (kMma && tid == 0 && mma_steps > 0) {
    const long long t0 = clock64();
    while (!mbar_try_wait(&s_mma, static_cast<uint32_t>((mma_steps - 1) & 1)))
      if (clock64() - t0 > kWaitCycles) break;
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tbase, kTmemCols);
  }
}

// ================================================================ streamed kernel (any r)
template <int KB, bool kRace>
__global__ void __launch_bounds__(kRollThreadsAll, 1) rollout_kernel(const RolloutParams p) {
  const int B = p.B, K = p.K, V = p.V, R = p.R;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nwarps = gridDim.x * kRollWarps;
  const int gw = blockIdx.x * kRollWarps + warp;
  extern __shared__ __align__(128) uint8_t s_dyn[];
  uint8_t* s_ring = s_dyn;                                                 // [kW2Stages][kW2StageBytes]
  float* s_u = reinterpret_cast<float*>(s_dyn + (p.head ? kW2Stages * kW2StageBytes : 0));  // [B][R]
  __shared__ __align__(8) uint64_t s_full[kW2Stages];   // chunk landed
  __shared__ __align__(8) uint64_t s_empty[kW2Stages];  // every compute warp is done with it
  __shared__ int s_tok[kRollMaxB];                      // t_j of each sequence
  __shared__ Lse s_red[kRollWarps][kRollMaxB];
  __shared__ int s_fail;
  // W2 stream: this CTA's contiguous run of chunks of `ch` rows, re-read every step (W2 is
  // constant, so the next step's first chunks load while its phases A and B run)
  const int ch = rollout_chunk_rows(R, p.head);
  const int nchunk_all = (V + ch - 1) / ch;
  const int cpc = (nchunk_all + gridDim.x - 1) / gridDim.x;
  const int c_lo = min(nchunk_all, static_cast<int>(blockIdx.x) * cpc);
  const int nch = min(nchunk_all, c_lo + cpc) - c_lo;
  // this CTA's rows and their base logits + b2 of the current step, staged in shared memory
  const int r_lo = c_lo * ch;
  const int r_n = max(0, min(V, (c_lo + nch) * ch) - r_lo);
  const int rows_cta = rollout_rows_per_cta(V, R, p.head, gridDim.x);
  float* s_base = s_u + (p.head ? B * R : 0);  // [B][rows_cta]
  if (tid == 0) {
    s_fail = 0;
    for (int sidx = 0; sidx < kW2Stages; ++sidx) {
      mbar_init(&s_full[sidx], 1);
      mbar_init(&s_empty[sidx], kRollWarps);
    }
    fence_mbar_init();
  }
  if (tid < B) s_tok[tid] = p.anchors[tid];
  __syncthreads();
  for (int b = 0; b < B; ++b)
    if (s_tok[b] < 0 || s_tok[b] >= V) {
      if (tid == 0) set_status(p.status, kStatusBadToken);
      return;  // every CTA sees the same ids and returns before the first barrier
    }

  if (warp == kRollWarps) {
    // ---- feeding warp: chunk g of the stream (step g / nch) into stage g % kW2Stages once
    //      every compute warp has released the chunk g - kW2Stages held there
    const long long n_loads = p.head ? static_cast<long long>(K) * nch : 0;
    if (lane == 0 && n_loads > 0) {
      // W2 streams through L2 at first-eviction priority so that the GRU and W1 weights of
      // phases A and B, re-read every step, stay in L2
      const uint64_t pol_w2 = l2_policy_evict_first();
      long long g = 0;
      for (; g < n_loads; ++g) {
        const int sidx = static_cast<int>(g % kW2Stages);
        if (g >= kW2Stages &&
            !mbar_wait(&s_empty[sidx], static_cast<uint32_t>((g / kW2Stages - 1) & 1), &s_fail, p.status))
          break;
        const int c = c_lo + static_cast<int>(g % nch);
        const int rows = min(ch, V - c * ch);
        const uint32_t bytes = static_cast<uint32_t>(rows) * R * 2;
        mbar_arrive_expect_tx(&s_full[sidx], bytes);
        bulk_load(s_ring + sidx * kW2StageBytes, p.w2 + static_cast<size_t>(c) * ch * R, bytes, &s_full[sidx],
                  pol_w2);
      }
      // the CTA leaves only once its copies in flight have landed (bounded)
      for (long long q = g > kW2Stages ? g - kW2Stages : 0; q < g; ++q) {
        const long long t0 = clock64();
        while (!mbar_try_wait(&s_full[q % kW2Stages], static_cast<uint32_t>((q / kW2Stages) & 1)))
          if (clock64() - t0 > kWaitCycles) break;
      }
    }
    return;
  }

  const PassRole role = pass_role<KB>(lane);
  const uint64_t pol_ab = l2_policy_evict_normal();
  unsigned nbar = 0;
  for (int j = 0; j < K; ++j) {
    const float* hprev = p.h + static_cast<size_t>((j + 1) & 1) * B * p.Ds;  // h_{j-1} (zeros at j = 0)
    float* hcur = p.h + static_cast<size_t>(j & 1) * B * p.Ds;
    if (p.head) {
      gru_phase(p, s_tok, hprev, hcur, gw, nwarps, lane, pol_ab);
      if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) return;
      u_phase(p, j, hcur, gw, nwarps, lane, pol_ab);
      if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) return;
      for (int e = tid; e < B * R; e += kRollThreads) s_u[e] = __ldcg(p.u + e);
    }
    // ---- C: L_j = base_j + W2 u_j + b2 over this CTA's rows; running max / sum exp / argmax
    stage_base(p, j, r_lo, r_n, rows_cta, s_base);
    compute_sync();
    Lse st[KB];
    Pick pst[KB];  // kRace: the perturbed maximum of every sequence
#pragma unroll
    for (int b = 0; b < KB; ++b) {
      st[b] = lse_empty();
      pst[b] = pick_empty();
    }
    if (p.head) {
      // W2 rows arrive chunk by chunk in the ring; warp w takes rows 4w .. 4w + 3, 4w + 32, ...
      // of a chunk
      float ur[KB][8];  // u at this lane's first 8 columns
#pragma unroll
      for (int b = 0; b < KB; ++b)
#pragma unroll
        for (int e = 0; e < 8; ++e) ur[b][e] = (b < B && lane * 8 < R) ? s_u[(b < B && lane * 8 < R) ? b * R + lane * 8 + e : 0] : 0.f;
      Lse mine = lse_empty();
      Pick pmine = pick_empty();
      for (int i = 0; i < nch; ++i) {
        const long long g = static_cast<long long>(j) * nch + i;
        const int sidx = static_cast<int>(g % kW2Stages);
        const bool landed = mbar_wait(&s_full[sidx], static_cast<uint32_t>((g / kW2Stages) & 1), &s_fail, p.status);
        if (!__all_sync(0xffffffffu, landed)) break;  // warp-uniform: the passes shuffle
        const int c = c_lo + i;
        const int rows = min(ch, V - c * ch);
        const __nv_bfloat16* sw = reinterpret_cast<const __nv_bfloat16*>(s_ring + sidx * kW2StageBytes);
        for (int r0 = warp * kRowsPerPass; r0 < rows; r0 += kRollWarps * kRowsPerPass) {
          float dot[kRowsPerPass * KB] = {};
          // columns lane*8 .. +8 against u held in registers, then (r > 256) the rest from shared memory
          if (lane * 8 < R) {
            float wv[kRowsPerPass][8];
            load_rows(sw, r0, rows, R, lane * 8, wv);
            pass_fma<KB>(wv, ur, dot);
          }
          for (int cc = lane * 8 + 256; cc < R; cc += 256) {
            float wv[kRowsPerPass][8];
            load_rows(sw, r0, rows, R, cc, wv);
            float uv[KB][8];
#pragma unroll
            for (int b = 0; b < KB; ++b) {
              if (b < B) {
                const float4 u0 = *reinterpret_cast<const float4*>(s_u + b * R + cc);
                const float4 u1 = *reinterpret_cast<const float4*>(s_u + b * R + cc + 4);
                uv[b][0] = u0.x; uv[b][1] = u0.y; uv[b][2] = u0.z; uv[b][3] = u0.w;
                uv[b][4] = u1.x; uv[b][5] = u1.y; uv[b][6] = u1.z; uv[b][7] = u1.w;
              } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) uv[b][e] = 0.f;
              }
            }
            pass_fma<KB>(wv, uv, dot);
          }
          pass_push<KB, kRace>(dot, role, rows - r0, i * ch + r0, c * ch + r0, s_base, rows_cta, B, mine, pmine, j,
                           p.seed);
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_empty[sidx]);  // this warp is done with the stage
      }
#pragma unroll
      for (int b = 0; b < KB; ++b)
        if (b == role.b) {
          st[b] = mine;
          pst[b] = pmine;
        }
    } else {
      for (int r = tid; r < r_n; r += kRollThreads) {
        uint4 x[(KB + 3) / 4];
        if constexpr (kRace) {
#pragma unroll
          for (int w = 0; w < (KB + 3) / 4; ++w) x[w] = race_words(p.seed, w, j, r_lo + r);
        }
#pragma unroll
        for (int b = 0; b < KB; ++b) {
          if (b < B) {
            lse_push(st[b], s_base[b * rows_cta + r], r_lo + r);
            if constexpr (kRace) pick_push(pst[b], s_base[b * rows_cta + r], race_gumbel(x[b >> 2], b & 3), r_lo + r);
          }
        }
      }
    }
    if (!finish_step<KB, kRace>(p, j, st, pst, s_red, s_tok, nbar, &s_fail, s_base, r_lo, r_n, rows_cta, false)) return;
  }
  if (kRace || p.best) greedy_logp<KB, kRace>(p, s_red, s_tok);
}

// ================================================================ launch helpers
static inline bool use_resident(const RolloutParams& p) { return p.head && p.R <= kResidentMaxR; }

template <typename Kern, typename... Extra>
static cudaError_t launch_coop(Kern kern, const RolloutParams& p, int grid, int threads, size_t smem,
                               cudaStream_t stream, Extra... extra) {
  if (smem > 48 * 1024) {
    const cudaError_t e = ensure_smem_attr(reinterpret_cast<const void*>(kern), smem, false);
    if (e != cudaSuccess) return e;
  }
  RolloutParams pp = p;
  void* args[] = {&pp, &extra...};
  cudaError_t e = cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(kern), dim3(grid), dim3(threads), args,
                                              smem, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

template <int KB, bool kRace>
static cudaError_t launch_rollout_kb(const RolloutParams& p, int grid, size_t smem, cudaStream_t stream,
                                     const CUtensorMap& tm) {
  if (use_resident(p)) {
    if constexpr (KB <= 2) {
      if (p.mma_tb + p.mma_sb > 0)
        return launch_coop(rollout_resident_kernel<KB, true, kRace>, p, grid, kRollThreads, smem, stream, tm);
    }
    return launch_coop(rollout_resident_kernel<KB, false, kRace>, p, grid, kRollThreads, smem, stream, tm);
  }
  return launch_coop(rollout_kernel<KB, kRace>, p, grid, kRollThreadsAll, smem, stream);
}

template <bool kRace>
static cudaError_t launch_rollout_b(const RolloutParams& p, int grid, size_t smem, cudaStream_t stream,
                                    const CUtensorMap& tm) {
  if (p.B <= 1) return launch_rollout_kb<1, kRace>(p, grid, smem, stream, tm);
  if (p.B <= 2) return launch_rollout_kb<2, kRace>(p, grid, smem, stream, tm);
  if (p.B <= 4) return launch_rollout_kb<4, kRace>(p, grid, smem, stream, tm);
  return launch_rollout_kb<8, kRace>(p, grid, smem, stream, tm);
}

// The seeded exponential-race instantiations (rollout_race.cu).
cudaError_t launch_rollout_race(const RolloutParams& p, int grid, size_t smem, cudaStream_t stream,
                                const CUtensorMap& tm);

}  // namespace dm
