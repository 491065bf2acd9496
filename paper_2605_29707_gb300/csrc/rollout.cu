// rollout.cu -- the greedy sequential draft loop (section 4.1.2 and Fig. 3: at inference each
// draft token is chosen from the final logits L_j = L_base_j + W2 u_j + b2 and becomes the
// causal encoder's next input).  The base logits W_lm hidden_j of every position come first from
// the tensor-core GEMM (store mode, fp32); this persistent cooperative kernel then runs the K
// dependent steps, each in three phases separated by grid barriers:
//   A  GRU step: h_j = GRU(emb[t_j], h_{j-1}), one warp per hidden unit (torch.nn.GRU gates);
//   B  u_j = SiLU(W1 [hidden_j ; h_j] + b1), one warp per rank row;
//   C  L_j = base_j + W2 u_j + b2, each lane owning vocabulary rows, with a running max, sum of
//      exp and argmax (equal values: the lowest id) per sequence, reduced per CTA;
// after the third barrier every CTA combines the per-CTA partials itself (the same result
// everywhere), so t_{j+1} needs no fourth barrier.  Every wait is bounded.
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

namespace dm {

constexpr int kRollThreads = 256;                 // the compute warps
constexpr int kRollWarps = kRollThreads / 32;
constexpr int kRollThreadsAll = kRollThreads + 32;  // + one warp streaming W2 into shared memory
constexpr int kW2Stages = 6;                        // shared-memory ring of W2 chunks
constexpr int kW2StageBytes = 16 * 1024;            // one chunk: kW2StageBytes / (2 r) rows of W2
constexpr int kRowsPerPass = 4;                     // W2 rows one warp takes at a time

__device__ __forceinline__ float bf2f(__nv_bfloat16 x) { return __bfloat162float(x); }

__device__ __forceinline__ void bf8(const __nv_bfloat16* p, float (&f)[8]) {
  const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

// 8 bf16 of global memory with an L2 eviction-priority hint
__device__ __forceinline__ void bf8_hint(const __nv_bfloat16* p, float (&f)[8], uint64_t pol) {
  uint4 v;
  asm("ld.global.nc.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
      : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
      : "l"(p), "l"(pol));
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

// 8 bf16 of shared memory (16-byte aligned) to fp32
__device__ __forceinline__ void bf8_smem(const __nv_bfloat16* p, float (&f)[8]) {
  const uint4 v = *reinterpret_cast<const uint4*>(p);
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = __bfloat1622float2(h[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}

// Columns cc .. cc + 7 of the pass's rows r0 .. r0 + 3 of a W2 chunk in shared memory (rows
// past the chunk's end read as zero).
__device__ __forceinline__ void load_rows(const __nv_bfloat16* sw, int r0, int rows, int R, int cc,
                                          float (&wv)[kRowsPerPass][8]) {
#pragma unroll
  for (int r = 0; r < kRowsPerPass; ++r) {
    if (r0 + r < rows) {
      bf8_smem(sw + static_cast<size_t>(r0 + r) * R + cc, wv[r]);
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) wv[r][e] = 0.f;
    }
  }
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

// Rows of the vocabulary one CTA covers: a contiguous run of chunks of `ch` rows (ch = the rows
// of W2 in one ring stage with the head on, 1024 without it).
__host__ __device__ inline int rollout_chunk_rows(int R, int head) {
  return head ? max(1, kW2StageBytes / (2 * R)) : 1024;
}
__host__ __device__ inline int rollout_rows_per_cta(int V, int R, int head, int grid) {
  const int ch = rollout_chunk_rows(R, head);
  const int nchunk_all = (V + ch - 1) / ch;
  return ((nchunk_all + grid - 1) / grid) * ch;
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

// Barrier of the compute warps only (the streaming warp runs on its own).
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
// then stops.
__device__ bool grid_barrier(unsigned* ctr, unsigned n, int* status, volatile int* fail) {
  compute_sync();
  if (threadIdx.x == 0) {
    __threadfence();
    atomicAdd(ctr, 1u);
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
  }
  compute_sync();
  return *fail == 0;
}

// KB: sequences the phase-C arithmetic is laid out for (B <= KB; the extra ones compute on
// zeros and are never read).
template <int KB>
__global__ void __launch_bounds__(kRollThreadsAll, 1) rollout_kernel(const RolloutParams p) {
  const int B = p.B, K = p.K, H = p.H, V = p.V, Ds = p.Ds, R = p.R;
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
    // ---- streaming warp: chunk g of the stream (step g / nch) into stage g % kW2Stages once
    //      every compute warp has released the chunk g - kW2Stages held there
    const long long n_loads = p.head ? static_cast<long long>(K) * nch : 0;
    if (lane == 0 && n_loads > 0) {
      // W2 (r x V, the largest operand) streams through L2 at first-eviction priority so that
      // the GRU and W1 weights of phases A and B, re-read every step, stay in L2
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

  // phase-C lane roles: value (r, b) of a pass lands on lanes with idx = r * KB + b
  constexpr int kN = kRowsPerPass * KB;
  constexpr int kLogN = ilog2(kN);
  static_assert((1 << kLogN) == kN && kN <= 32, "rows x sequences per pass must be a power of two <= 32");
  const int my_idx = lane >> (5 - kLogN);
  const int my_r = my_idx / KB, my_b = my_idx % KB;
  const bool my_rep = (lane & ((32 >> kLogN) - 1)) == 0;  // one lane per value pushes it

  const uint64_t pol_ab = l2_policy_evict_normal();
  unsigned nbar = 0;
  for (int j = 0; j < K; ++j) {
    const float* hprev = p.h + static_cast<size_t>((j + 1) & 1) * B * Ds;  // h_{j-1} (zeros at j = 0)
    float* hcur = p.h + static_cast<size_t>(j & 1) * B * Ds;
    if (p.head) {
      // ---- A: GRU step (torch.nn.GRU: gates r|z|n, r multiplies W_hn h + b_hn)
      for (int q = gw; q < Ds; q += nwarps) {
        for (int b = 0; b < B; ++b) {
          const __nv_bfloat16* x = p.emb + static_cast<size_t>(s_tok[b]) * H;
          float ar = 0.f, az = 0.f, an = 0.f, hr = 0.f, hz = 0.f, hn = 0.f;
#pragma unroll 4
          for (int c = lane * 8; c < H; c += 256) {
            float xv[8], wr[8], wz[8], wn[8];
            bf8(x + c, xv);
            bf8_hint(p.w_ih + static_cast<size_t>(q) * H + c, wr, pol_ab);
            bf8_hint(p.w_ih + static_cast<size_t>(Ds + q) * H + c, wz, pol_ab);
            bf8_hint(p.w_ih + static_cast<size_t>(2 * Ds + q) * H + c, wn, pol_ab);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              ar += wr[e] * xv[e];
              az += wz[e] * xv[e];
              an += wn[e] * xv[e];
            }
          }
          const float* hp = hprev + static_cast<size_t>(b) * Ds;
#pragma unroll 4
          for (int c = lane * 8; c < Ds; c += 256) {
            float wr[8], wz[8], wn[8];
            bf8_hint(p.w_hh + static_cast<size_t>(q) * Ds + c, wr, pol_ab);
            bf8_hint(p.w_hh + static_cast<size_t>(Ds + q) * Ds + c, wz, pol_ab);
            bf8_hint(p.w_hh + static_cast<size_t>(2 * Ds + q) * Ds + c, wn, pol_ab);
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
      if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) return;
      // ---- B: u_j = SiLU(W1 [hidden_j ; h_j] + b1)
      for (int q = gw; q < R; q += nwarps) {
        const __nv_bfloat16* w = p.w1 + static_cast<size_t>(q) * (H + Ds);
        for (int b = 0; b < B; ++b) {
          const __nv_bfloat16* hid = p.hidden + (static_cast<size_t>(b) * K + j) * H;
          const float* hc = hcur + static_cast<size_t>(b) * Ds;
          float acc = 0.f;
#pragma unroll 4
          for (int c = lane * 8; c < H; c += 256) {
            float wv[8], xv[8];
            bf8_hint(w + c, wv, pol_ab);
            bf8(hid + c, xv);
#pragma unroll
            for (int e = 0; e < 8; ++e) acc += wv[e] * xv[e];
          }
#pragma unroll 4
          for (int c = lane * 8; c < Ds; c += 256) {
            float wv[8];
            bf8_hint(w + H + c, wv, pol_ab);
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
      if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) return;
      for (int e = tid; e < B * R; e += kRollThreads) s_u[e] = __ldcg(p.u + e);
    }
    // ---- C: L_j = base_j + W2 u_j + b2 over this CTA's rows; running max / sum exp / argmax
    for (int e = tid; e < B * r_n; e += kRollThreads) {
      const int b = e / r_n, r = e - b * r_n;
      s_base[b * rows_cta + r] = __ldcg(p.base + (static_cast<size_t>(b) * K + j) * V + r_lo + r) +
                                 (p.b2 ? bf2f(p.b2[r_lo + r]) : 0.f);
    }
    compute_sync();
    Lse st[KB];
#pragma unroll
    for (int b = 0; b < KB; ++b) st[b] = lse_empty();
    if (p.head) {
      // W2 rows arrive chunk by chunk in the ring; warp w takes rows 4w .. 4w + 3, 4w + 32, ...
      // of a chunk, a lane holding 8 consecutive columns of each (one 16-byte load per row); the
      // 4 x KB dot products of a pass are summed over the warp by a reduce-scatter, after which
      // lane my_idx holds row my_r of sequence my_b.
      float ur[KB][8];  // u at this lane's first 8 columns
#pragma unroll
      for (int b = 0; b < KB; ++b)
#pragma unroll
        for (int e = 0; e < 8; ++e) ur[b][e] = (b < B && lane * 8 < R) ? s_u[b * R + lane * 8 + e] : 0.f;
      Lse mine = lse_empty();
      for (int i = 0; i < nch; ++i) {
        const long long g = static_cast<long long>(j) * nch + i;
        const int sidx = static_cast<int>(g % kW2Stages);
        if (!mbar_wait(&s_full[sidx], static_cast<uint32_t>((g / kW2Stages) & 1), &s_fail, p.status)) break;
        const int c = c_lo + i;
        const int rows = min(ch, V - c * ch);
        const __nv_bfloat16* sw = reinterpret_cast<const __nv_bfloat16*>(s_ring + sidx * kW2StageBytes);
        for (int r0 = warp * kRowsPerPass; r0 < rows; r0 += kRollWarps * kRowsPerPass) {
          float dot[kN];
#pragma unroll
          for (int v = 0; v < kN; ++v) dot[v] = 0.f;
          // columns lane*8 .. +8 against u held in registers, then (r > 256) the rest from shared memory
          if (lane * 8 < R) {
            float wv[kRowsPerPass][8];
            load_rows(sw, r0, rows, R, lane * 8, wv);
#pragma unroll
            for (int r = 0; r < kRowsPerPass; ++r)
#pragma unroll
              for (int b = 0; b < KB; ++b)
#pragma unroll
                for (int e = 0; e < 8; ++e) dot[r * KB + b] += wv[r][e] * ur[b][e];
          }
          for (int cc = lane * 8 + 256; cc < R; cc += 256) {
            float wv[kRowsPerPass][8];
            load_rows(sw, r0, rows, R, cc, wv);
#pragma unroll
            for (int b = 0; b < KB; ++b) {
              float uv[8];
              if (b < B) {
                const float4 u0 = *reinterpret_cast<const float4*>(s_u + b * R + cc);
                const float4 u1 = *reinterpret_cast<const float4*>(s_u + b * R + cc + 4);
                uv[0] = u0.x; uv[1] = u0.y; uv[2] = u0.z; uv[3] = u0.w;
                uv[4] = u1.x; uv[5] = u1.y; uv[6] = u1.z; uv[7] = u1.w;
              } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) uv[e] = 0.f;
              }
#pragma unroll
              for (int r = 0; r < kRowsPerPass; ++r)
#pragma unroll
                for (int e = 0; e < 8; ++e) dot[r * KB + b] += wv[r][e] * uv[e];
            }
          }
          const float d = ReduceScatter<kN, 16>::run(dot);
          if (my_rep && r0 + my_r < rows && my_b < B) {
            const int v = c * ch + r0 + my_r;
            lse_push(mine, s_base[my_b * rows_cta + (v - r_lo)] + d, v);
          }
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(&s_empty[sidx]);  // this warp is done with the stage
      }
#pragma unroll
      for (int b = 0; b < KB; ++b)
        if (b == my_b) st[b] = mine;
    } else {
      for (int r = tid; r < r_n; r += kRollThreads) {
#pragma unroll
        for (int b = 0; b < KB; ++b)
          if (b < B) lse_push(st[b], s_base[b * rows_cta + r], r_lo + r);
      }
    }
    block_reduce(st, s_red, B);
    if (tid < B) {
      Lse a = s_red[0][tid];
      for (int w = 1; w < kRollWarps; ++w) lse_merge(a, s_red[w][tid]);
      float4* out = reinterpret_cast<float4*>(p.partials) + static_cast<size_t>(blockIdx.x) * kRollMaxB + tid;
      *out = make_float4(a.m, a.s, __int_as_float(a.i), 0.f);
    }
    if (!grid_barrier(p.barrier, nbar++, p.status, &s_fail)) return;
    // ---- every CTA: combine the partials (thread c loads CTA c's, then the same block reduction;
    //      every CTA reduces in the same order, so all reach the same t_{j+1}), choose t_{j+1}
#pragma unroll
    for (int b = 0; b < KB; ++b) st[b] = lse_empty();
    for (int c = tid; c < static_cast<int>(gridDim.x); c += kRollThreads) {
#pragma unroll
      for (int b = 0; b < KB; ++b) {
        if (b < B) {
          const float4 f = __ldcg(reinterpret_cast<const float4*>(p.partials) + static_cast<size_t>(c) * kRollMaxB + b);
          Lse t;
          t.m = f.x; t.s = f.y; t.i = __float_as_int(f.z);
          lse_merge(st[b], t);
        }
      }
    }
    block_reduce(st, s_red, B);
    if (tid < B) {
      Lse a = s_red[0][tid];
      for (int w = 1; w < kRollWarps; ++w) lse_merge(a, s_red[w][tid]);
      const int tok = a.i == 0x7fffffff ? 0 : a.i;
      s_tok[tid] = tok;
      if (blockIdx.x == 0) {
        p.tokens[static_cast<size_t>(tid) * K + j] = tok;
        p.logp[static_cast<size_t>(tid) * K + j] = -logf(a.s);  // the argmax's logit is the max
      }
    }
    compute_sync();
  }
}

size_t rollout_smem_bytes(int B, int V, int R, bool head, int grid) {
  return (head ? static_cast<size_t>(kW2Stages) * kW2StageBytes : 0) +
         static_cast<size_t>(B) * (head ? R : 0) * sizeof(float) +
         static_cast<size_t>(B) * rollout_rows_per_cta(V, R, head, grid) * sizeof(float);
}

template <int KB>
static cudaError_t launch_rollout_kb(const RolloutParams& p, int grid, size_t smem, cudaStream_t stream) {
  static size_t attr_smem = 0;
  if (smem > 48 * 1024 && smem > attr_smem) {
    cudaError_t e = cudaFuncSetAttribute(rollout_kernel<KB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    attr_smem = smem;
  }
  RolloutParams pp = p;
  void* args[] = {&pp};
  cudaError_t e = cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(rollout_kernel<KB>), dim3(grid),
                                              dim3(kRollThreadsAll), args, smem, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

cudaError_t launch_rollout(const RolloutParams& p, int grid, cudaStream_t stream) {
  if (p.B < 1 || p.B > kRollMaxB || grid < 1) return cudaErrorInvalidValue;
  const size_t smem = rollout_smem_bytes(p.B, p.V, p.R, p.head, grid);
  if (smem > kRollMaxSmem) return cudaErrorInvalidValue;
  if (p.B <= 1) return launch_rollout_kb<1>(p, grid, smem, stream);
  if (p.B <= 2) return launch_rollout_kb<2>(p, grid, smem, stream);
  if (p.B <= 4) return launch_rollout_kb<4>(p, grid, smem, stream);
  return launch_rollout_kb<8>(p, grid, smem, stream);
}

}  // namespace dm
