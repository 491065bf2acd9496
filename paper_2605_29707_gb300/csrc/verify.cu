// verify.cu -- greedy verification of a draft tree against the target's logits (the step after
// the draft, section 3.1: one target pass checks the whole draft, draft tokens are kept up to the
// first one the target rejects, and tau counts them plus the target's own extra token).
//
// Row argmax: a cluster of kSplit CTAs per row of target logits (the target's next-token logits
// after the anchor, row 0, and after each tree node i, row i + 1); each CTA finds the greatest
// value of its slice of the row and, among equal values, the lowest id, and the cluster's first
// CTA combines the slices through distributed shared memory.  Walk: one warp per sequence
// starts at the anchor, takes the argmax of the current node's row and moves to the child
// carrying that token (the lowest node index if several do), until no child does; that argmax
// is the bonus token.
#include <math.h>

#include "kernels.h"
#include "ptx.cuh"

namespace dm {

constexpr int kArgmaxThreads = 256;
constexpr int kSplit = 8;  // CTAs (one cluster) per row

__device__ __forceinline__ uint32_t dsmem_addr(const void* local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(local)), "r"(rank));
  return r;
}

__device__ __forceinline__ void better_of(float& v, int& id, float v2, int id2) {
  if (v2 > v || (v2 == v && id2 < id)) { v = v2; id = id2; }
}

__global__ void __launch_bounds__(kArgmaxThreads) row_argmax_kernel(const float* __restrict__ logits, int V,
                                                                    int32_t* __restrict__ row_argmax) {
  const size_t row = blockIdx.x / kSplit;
  const uint32_t part = cluster_ctarank();  // == blockIdx.x % kSplit: clusters are consecutive CTAs
  const float* x = logits + row * static_cast<size_t>(V);
  // this CTA's slice [lo, hi): kSplit slices of a multiple of 4 entries (the last is short)
  const int slice = ((V + kSplit - 1) / kSplit + 3) & ~3;
  const int lo = static_cast<int>(part) * slice;
  const int hi = min(V, lo + slice);
  float bv = -INFINITY;
  int bi = 0x7fffffff;
  if ((V & 3) == 0 && (reinterpret_cast<uintptr_t>(x) & 15) == 0) {
    const float4* x4 = reinterpret_cast<const float4*>(x);
    for (int q = lo / 4 + threadIdx.x; q < hi / 4; q += kArgmaxThreads) {
      const float4 f = __ldg(x4 + q);
      better_of(bv, bi, f.x, 4 * q);
      better_of(bv, bi, f.y, 4 * q + 1);
      better_of(bv, bi, f.z, 4 * q + 2);
      better_of(bv, bi, f.w, 4 * q + 3);
    }
  } else {
    for (int v = lo + threadIdx.x; v < hi; v += kArgmaxThreads) better_of(bv, bi, __ldg(x + v), v);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
    const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
    better_of(bv, bi, v2, i2);
  }
  __shared__ float s_v[kArgmaxThreads / 32];
  __shared__ int s_i[kArgmaxThreads / 32];
  __shared__ float s_cv;  // this CTA's result, read by the cluster's first CTA
  __shared__ int s_ci;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) { s_v[warp] = bv; s_i[warp] = bi; }
  __syncthreads();
  if (warp == 0) {
    bv = lane < kArgmaxThreads / 32 ? s_v[lane] : -INFINITY;
    bi = lane < kArgmaxThreads / 32 ? s_i[lane] : 0x7fffffff;
#pragma unroll
    for (int o = 16; o; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
      better_of(bv, bi, v2, i2);
    }
    if (lane == 0) { s_cv = bv; s_ci = bi; }
  }
  cluster_sync();  // every slice's result is in its CTA's shared memory
  if (part == 0 && warp == 0) {
    bv = -INFINITY;
    bi = 0x7fffffff;
    if (lane < kSplit) {
      float v2;
      int i2;
      asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v2) : "r"(dsmem_addr(&s_cv, lane)) : "memory");
      asm volatile("ld.shared::cluster.s32 %0, [%1];" : "=r"(i2) : "r"(dsmem_addr(&s_ci, lane)) : "memory");
      bv = v2;
      bi = i2;
    }
#pragma unroll
    for (int o = 4; o; o >>= 1) {
      const float v2 = __shfl_xor_sync(0xffffffffu, bv, o);
      const int i2 = __shfl_xor_sync(0xffffffffu, bi, o);
      better_of(bv, bi, v2, i2);
    }
    // a row of -inf only (or of NaN only) keeps id 0, as a plain scan would
    if (lane == 0) row_argmax[row] = bi == 0x7fffffff ? 0 : bi;
  }
  cluster_sync();  // no CTA leaves while the first one may still read its result
}

__global__ void __launch_bounds__(32) tree_walk_kernel(const int32_t* __restrict__ parent,
                                                       const int32_t* __restrict__ token,
                                                       const int32_t* __restrict__ row_argmax, int N,
                                                       int32_t* __restrict__ nodes, int32_t* __restrict__ count,
                                                       int32_t* __restrict__ bonus) {
  const int b = blockIdx.x;
  const int lane = threadIdx.x;
  const int32_t* par = parent + static_cast<size_t>(b) * N;
  const int32_t* tok = token + static_cast<size_t>(b) * N;
  const int32_t* ra = row_argmax + static_cast<size_t>(b) * (N + 1);
  int32_t* out = nodes + static_cast<size_t>(b) * N;
  for (int i = lane; i < N; i += 32) out[i] = -1;
  __syncwarp();
  int cur = -1, n = 0, a = ra[0];
  // every accepted node is a child of the previous one, so at most N steps (also bounds the walk
  // on a malformed tree whose parents are not earlier nodes)
  for (int step = 0; step <= N; ++step) {
    a = ra[cur + 1];
    int next = -1;
    for (int c0 = 0; c0 < N && next < 0; c0 += 32) {
      const int c = c0 + lane;
      const bool hit = c < N && par[c] == cur && tok[c] == a;
      const unsigned m = __ballot_sync(0xffffffffu, hit);
      if (m) next = c0 + __ffs(m) - 1;
    }
    if (next < 0 || n >= N) break;
    if (lane == 0) out[n] = next;
    ++n;
    cur = next;
  }
  if (lane == 0) {
    count[b] = n;
    bonus[b] = a;
  }
}

cudaError_t launch_verify_greedy(const float* logits, const int32_t* parent, const int32_t* token, int B, int N,
                                 int V, int32_t* row_argmax, int32_t* nodes, int32_t* count, int32_t* bonus,
                                 cudaStream_t stream) {
  const long long rows = static_cast<long long>(B) * (N + 1);
  if (rows <= 0 || rows > 0x7fffffffLL) return cudaErrorInvalidValue;
  if (rows * kSplit > 0x7fffffffLL) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(rows * kSplit));
  cfg.blockDim = dim3(kArgmaxThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kSplit;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, row_argmax_kernel, logits, V, row_argmax);
  if (e != cudaSuccess) return e;
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  tree_walk_kernel<<<B, 32, 0, stream>>>(parent, token, row_argmax, N, nodes, count, bonus);
  return cudaGetLastError();
}

}  // namespace dm
