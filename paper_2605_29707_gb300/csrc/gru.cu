// gru.cu -- embedding gather (E_j, section 4.1.2) and the GRU causal encoder
// S_{i-1} = GRU(E_{<=i-1}) followed by the low-rank code u = SiLU(W1 [H_i; S_{i-1}] + b1).
//
// The recurrence is the only sequential part of the step: K dependent steps.  One cooperative
// launch keeps a slice of W_hh resident in each CTA's shared memory for all K steps (CTA c owns
// hidden units [c*U, c*U+U) and the three gate rows r|z|n of each), exchanges the new state
// through global memory (L2) and separates the steps with a bounded grid barrier.  After the
// last step the same CTAs finish u: the hidden half of W1 was computed earlier by the
// tensor-core projection (split-K partial sums); the state half is added here.
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

namespace dm {

constexpr int kGruThreads = 256;

__global__ void __launch_bounds__(128) gather_kernel(const GatherParams p) {
  const int m = blockIdx.x;
  const int id = p.ids[m];
  const bool ok = id >= 0 && id < p.V;
  if (!ok && threadIdx.x == 0) set_status(p.status, kStatusBadToken);
  if (p.E == nullptr) return;
  uint4* dst = reinterpret_cast<uint4*>(p.E + static_cast<size_t>(m) * p.H);
  const uint4* src = reinterpret_cast<const uint4*>(p.emb + static_cast<size_t>(ok ? id : 0) * p.H);
  for (int c = threadIdx.x; c < p.H / 8; c += blockDim.x) dst[c] = ok ? __ldg(src + c) : make_uint4(0, 0, 0, 0);
}

cudaError_t launch_gather(const GatherParams& p, cudaStream_t stream) {
  gather_kernel<<<p.M, 128, 0, stream>>>(p);
  return cudaGetLastError();
}

__device__ __forceinline__ unsigned ld_acquire_u32(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void red_release_add(unsigned* p, unsigned v) {
  asm volatile("red.release.gpu.global.add.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Bounded grid barrier on a monotonically increasing counter (release on arrival, acquire
// while polling).  The outcome is uniform over the CTA: false means this CTA gave up and
// recorded DOMINO_ERR_TIMEOUT.
__device__ bool grid_barrier(unsigned* counter, unsigned target, int* status, volatile int* flag) {
  __syncthreads();
  if (threadIdx.x == 0) {
    red_release_add(counter, 1u);
    int ok = 1;
    const long long t0 = clock64();
    while (ld_acquire_u32(counter) < target) {
      if (clock64() - t0 > kWaitCycles) {
        set_status(status, kStatusTimeout);
        ok = 0;
        break;
      }
    }
    *flag = ok;
  }
  __syncthreads();
  return *flag != 0;
}

__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gmem_src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gmem_src) : "memory");
}

__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n\tcp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ float dot8_bf16(const uint4 w, const float4 h0, const float4 h1) {
  const __nv_bfloat162* w2 = reinterpret_cast<const __nv_bfloat162*>(&w);
  const float2 a = __bfloat1622float2(w2[0]);
  const float2 b = __bfloat1622float2(w2[1]);
  const float2 c = __bfloat1622float2(w2[2]);
  const float2 d = __bfloat1622float2(w2[3]);
  float s = a.x * h0.x;
  s = fmaf(a.y, h0.y, s);
  s = fmaf(b.x, h0.z, s);
  s = fmaf(b.y, h0.w, s);
  s = fmaf(c.x, h1.x, s);
  s = fmaf(c.y, h1.y, s);
  s = fmaf(d.x, h1.z, s);
  s = fmaf(d.y, h1.w, s);
  return s;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ float bf_or0(const __nv_bfloat16* p, int i) {
  return p ? __bfloat162float(p[i]) : 0.f;
}

// Shared-memory layout of one GRU CTA (U hidden units, M = B*K rows, BG staged sequences):
//   whh [3][U][Ds] bf16 | xs [M][3][U] f32 (input-gate sums + b_ih) | bh [3][U] f32 (b_hh)
//   | hs [BG][Ds] f32 (h_{t-1}) | gs [BG][3][U] f32 (W_hh . h_{t-1}) | flag
struct GruSmem {
  size_t whh, xs, bh, hs, gs, flag, total;
};

__host__ __device__ inline GruSmem gru_layout(int Ds, int U, int M, int BG) {
  GruSmem L;
  size_t o = 0;
  L.whh = o; o += static_cast<size_t>(3) * U * Ds * 2;
  L.xs = o;  o += static_cast<size_t>(M) * 3 * U * 4;
  L.bh = o;  o += static_cast<size_t>(3) * U * 4;
  o = (o + 15) & ~static_cast<size_t>(15);
  L.hs = o;  o += static_cast<size_t>(BG) * Ds * 4;
  L.gs = o;  o += static_cast<size_t>(BG) * 3 * U * 4;
  L.flag = o; o += 16;
  L.total = o;
  return L;
}

__global__ void __launch_bounds__(kGruThreads) gru_kernel(const GruParams p, const int BG) {
  extern __shared__ __align__(16) uint8_t gsm[];
  const int U = p.units, Ds = p.Ds, K = p.K, B = p.B, R = p.R, H = p.H;
  const int M = B * K;
  const int j0 = blockIdx.x * U;
  const int Uc = min(U, Ds - j0);
  const GruSmem L = gru_layout(Ds, U, M, BG);
  __nv_bfloat16* whh = reinterpret_cast<__nv_bfloat16*>(gsm + L.whh);
  float* xs = reinterpret_cast<float*>(gsm + L.xs);
  float* bh = reinterpret_cast<float*>(gsm + L.bh);
  float* hs = reinterpret_cast<float*>(gsm + L.hs);
  float* gs = reinterpret_cast<float*>(gsm + L.gs);
  volatile int* flag = reinterpret_cast<volatile int*>(gsm + L.flag);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  constexpr int kWarps = kGruThreads / 32;

  // this CTA's rows of W_hh (gate g, unit j0 + jl), copied asynchronously
  const int rowlen8 = Ds / 8;
  for (int e = tid; e < 3 * Uc * rowlen8; e += kGruThreads) {
    const int c8 = e % rowlen8;
    const int r = e / rowlen8;
    const int g = r / Uc, jl = r % Uc;
    cp_async16(whh + (static_cast<size_t>(g) * U + jl) * Ds + c8 * 8,
               p.w_hh + (static_cast<size_t>(g) * Ds + j0 + jl) * Ds + c8 * 8);
  }
  // input-gate sums for every row and this CTA's units: b_ih + sum over split-K partials
  for (int e = tid; e < M * 3 * Uc; e += kGruThreads) {
    const int jl = e % Uc;
    const int g = (e / Uc) % 3;
    const int m = e / (3 * Uc);
    const int col = g * Ds + j0 + jl;
    float a = bf_or0(p.b_ih, col);
    for (int s = 0; s < p.xsplits; ++s) a += __ldg(p.xpart + (static_cast<size_t>(s) * M + m) * 3 * Ds + col);
    xs[(static_cast<size_t>(m) * 3 + g) * U + jl] = a;
  }
  for (int e = tid; e < 3 * Uc; e += kGruThreads) bh[(e / Uc) * U + e % Uc] = bf_or0(p.b_hh, (e / Uc) * Ds + j0 + e % Uc);
  cp_async_wait_all();
  __syncthreads();

  for (int t = 0; t < K; ++t) {
    for (int b0 = 0; b0 < B; b0 += BG) {
      const int nb = min(BG, B - b0);
      if (t > 0) {
        // h_{t-1} of sequences b0 .. b0+nb-1 (written by every CTA in step t-1)
        for (int e = tid; e < nb * (Ds / 4); e += kGruThreads) {
          const int bb = e / (Ds / 4), c4 = e % (Ds / 4);
          reinterpret_cast<float4*>(hs + static_cast<size_t>(bb) * Ds)[c4] = __ldcg(
              reinterpret_cast<const float4*>(p.S + (static_cast<size_t>(b0 + bb) * K + (t - 1)) * Ds) + c4);
        }
        __syncthreads();
        // W_hh[rows of this CTA] . h_{t-1}
        for (int d = warp; d < 3 * Uc * nb; d += kWarps) {
          const int r = d % (3 * Uc), bb = d / (3 * Uc);
          const int g = r / Uc, jl = r % Uc;
          const __nv_bfloat16* wrow = whh + (static_cast<size_t>(g) * U + jl) * Ds;
          const float* hrow = hs + static_cast<size_t>(bb) * Ds;
          float acc = 0.f;
          for (int c = lane * 8; c < Ds; c += 256) {
            const uint4 wv = *reinterpret_cast<const uint4*>(wrow + c);
            const float4 h0 = *reinterpret_cast<const float4*>(hrow + c);
            const float4 h1 = *reinterpret_cast<const float4*>(hrow + c + 4);
            acc += dot8_bf16(wv, h0, h1);
          }
          acc = warp_sum(acc);
          if (lane == 0) gs[(bb * 3 + g) * U + jl] = acc;
        }
        __syncthreads();
      }
      // gates and the new state (torch.nn.GRU convention)
      for (int e = tid; e < nb * Uc; e += kGruThreads) {
        const int bb = e / Uc, jl = e % Uc;
        const int j = j0 + jl;
        const int m = (b0 + bb) * K + t;
        const float* x = xs + static_cast<size_t>(m) * 3 * U;
        float hr = bh[jl], hz = bh[U + jl], hn = bh[2 * U + jl];
        float hprev = 0.f;
        if (t > 0) {
          hr += gs[(bb * 3 + 0) * U + jl];
          hz += gs[(bb * 3 + 1) * U + jl];
          hn += gs[(bb * 3 + 2) * U + jl];
          hprev = hs[static_cast<size_t>(bb) * Ds + j];
        }
        const float r = 1.f / (1.f + expf(-(x[jl] + hr)));
        const float z = 1.f / (1.f + expf(-(x[U + jl] + hz)));
        const float n = tanhf(x[2 * U + jl] + r * hn);
        p.S[static_cast<size_t>(m) * Ds + j] = (1.f - z) * n + z * hprev;
      }
      __syncthreads();
    }
    if (!grid_barrier(p.barrier, static_cast<unsigned>(gridDim.x) * (t + 1), p.status, flag)) return;
  }

  // u[m, q] = SiLU(b1[q] + hidden_m . W1[q, :H] + S_m . W1[q, H:])
  const int total_warps = gridDim.x * kWarps;
  const int gw = blockIdx.x * kWarps + warp;
  const int groups = max(1, total_warps / R);
  for (int pi = gw; pi < R * groups; pi += total_warps) {
    const int q = pi % R, mg = pi / R;
    const __nv_bfloat16* w1row = p.w1 + static_cast<size_t>(q) * (H + Ds) + H;
    const float bq = bf_or0(p.b1, q);
    for (int m = mg; m < M; m += groups) {
      const float* srow = p.S + static_cast<size_t>(m) * Ds;
      float acc = 0.f;
      for (int c = lane * 8; c < Ds; c += 256) {
        const uint4 wv = __ldg(reinterpret_cast<const uint4*>(w1row + c));
        const float4 h0 = __ldcg(reinterpret_cast<const float4*>(srow + c));
        const float4 h1 = __ldcg(reinterpret_cast<const float4*>(srow + c + 4));
        acc += dot8_bf16(wv, h0, h1);
      }
      // the hidden half arrives as split-K partial sums; the lanes add them in parallel
      for (int s = lane; s < p.usplits; s += 32) acc += __ldg(p.upart + (static_cast<size_t>(s) * M + m) * R + q);
      acc = warp_sum(acc);
      if (lane == 0) {
        const float a = acc + bq;
        p.u[static_cast<size_t>(m) * R + q] = __float2bfloat16_rn(a / (1.f + expf(-a)));
      }
    }
  }
}

int gru_grid(int Ds, int num_sms, int* units) {
  int G = Ds < 128 ? Ds : 128;
  if (G > num_sms) G = num_sms;
  int U = (Ds + G - 1) / G;
  if (static_cast<size_t>(3) * U * Ds * 2 > 160 * 1024) {
    G = Ds < num_sms ? Ds : num_sms;
    U = (Ds + G - 1) / G;
  }
  G = (Ds + U - 1) / U;
  *units = U;
  return G;
}

static constexpr size_t kGruSmemBudget = 220 * 1024;

static int gru_bg(int Ds, int U, int M, int B) {
  int bg = B < 8 ? B : 8;
  while (bg > 1 && gru_layout(Ds, U, M, bg).total > kGruSmemBudget) --bg;
  return gru_layout(Ds, U, M, bg).total > kGruSmemBudget ? 0 : bg;
}

size_t gru_smem_bytes(int Ds, int units, int M, int B) {
  const int bg = gru_bg(Ds, units, M, B);
  return bg == 0 ? 0 : gru_layout(Ds, units, M, bg).total;
}

cudaError_t launch_gru(const GruParams& p, int grid, cudaStream_t stream) {
  const int M = p.B * p.K;
  const int bg = gru_bg(p.Ds, p.units, M, p.B);
  if (bg == 0) return cudaErrorInvalidValue;
  const size_t smem = gru_layout(p.Ds, p.units, M, bg).total;
  static size_t attr_smem = 0;
  if (smem > attr_smem) {
    cudaError_t e = cudaFuncSetAttribute(gru_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    attr_smem = smem;
  }
  GruParams pp = p;
  int bgv = bg;
  void* args[] = {&pp, &bgv};
  cudaError_t e = cudaLaunchCooperativeKernel(reinterpret_cast<const void*>(gru_kernel), dim3(grid),
                                              dim3(kGruThreads), args, smem, stream);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

}  // namespace dm
