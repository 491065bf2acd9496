// verify.cu -- verification of a draft tree against the target's logits (the step after the
// draft, section 3.1: one target pass checks the whole draft, draft tokens are kept up to the
// first one the target rejects, and tau counts them plus the target's own extra token), greedy
// (temperature 0: the target's choice after a node is its argmax) and sampled (temperature T > 0:
// its choice is a draw from softmax(logits / T) with the caller's uniform).
//
// Row argmax: a cluster of kSplit CTAs per row of target logits (the target's next-token logits
// after the anchor, row 0, and after each tree node i, row i + 1); each CTA finds the greatest
// value of its slice of the row and, among equal values, the lowest id, and the cluster's first
// CTA combines the slices through distributed shared memory.  Walk: one warp per sequence
// starts at the anchor, takes the argmax of the current node's row and moves to the child
// carrying that token (the lowest node index if several do), until no child does; that argmax
// is the bonus token.
//
// Row draw (sampled): the same clusters; each CTA stages its slice of the row in shared memory
// (one DRAM read), the cluster agrees on the row maximum, each CTA sums exp((x - max) / T) over
// its slice, and every CTA combines the eight slice sums in the same order, so all agree on the
// total Z and on the slice whose interval holds u Z; that CTA alone finds the first id whose
// cumulative sum (in id order) passes it.  The walk is the greedy one on the draws.
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
    constexpr int kBatch = 8;  // loads in flight per thread
    for (int q0 = lo / 4 + threadIdx.x; q0 < hi / 4; q0 += kArgmaxThreads * kBatch) {
      float4 f[kBatch];
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int q = q0 + j * kArgmaxThreads;
        if (q < hi / 4) f[j] = __ldg(x4 + q);
      }
#pragma unroll
      for (int j = 0; j < kBatch; ++j) {
        const int q = q0 + j * kArgmaxThreads;
        if (q < hi / 4) {  // ids rise with j: the first of equal values stays first
          better_of(bv, bi, f[j].x, 4 * q);
          better_of(bv, bi, f[j].y, 4 * q + 1);
          better_of(bv, bi, f[j].z, 4 * q + 2);
          better_of(bv, bi, f[j].w, 4 * q + 3);
        }
      }
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
  // launched as a programmatic dependent of the row kernel: its choices are complete after this
  asm volatile("griddepcontrol.wait;" ::: "memory");
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

// The walk, launched as a programmatic dependent of the row kernel before it: its launch and the
// clearing of the accepted-node list overlap the row kernel's tail.
static cudaError_t launch_walk(const int32_t* parent, const int32_t* token, const int32_t* row_choice, int B,
                               int N, int32_t* nodes, int32_t* count, int32_t* bonus, cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(B));
  cfg.blockDim = dim3(32);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, tree_walk_kernel, parent, token, row_choice, N, nodes, count, bonus);
  if (e != cudaSuccess) return e;
  return cudaGetLastError();
}

// ------------------------------------------------------------------------------ row draw
constexpr int kSampleThreads = 256;
constexpr int kLoadBatch = 8;  // float4 loads a thread has in flight while staging

__device__ __forceinline__ float ld_cluster_f32(const void* local, uint32_t rank) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(dsmem_addr(local, rank)) : "memory");
  return v;
}

// One draw per row from softmax(row * inv_t) with uniform u = uniforms[row] (clamped to [0, 1)):
// the first id whose cumulative weight, in id order, exceeds u Z.  Where rounding leaves no such
// id (u Z at or past the computed total), the last id of non-zero weight; a row with no finite
// value gives id 0.  The cumulative sums are fp32 and their order is fixed (per thread a
// contiguous run, then thread order, then slice order), so the draw is deterministic.
__global__ void __launch_bounds__(kSampleThreads) row_sample_kernel(const float* __restrict__ logits, int V,
                                                                    float inv_t, const float* __restrict__ uniforms,
                                                                    int32_t* __restrict__ row_sample) {
  extern __shared__ __align__(16) float s_x[];  // this CTA's slice of the row
  __shared__ float s_red[kSampleThreads / 32];
  __shared__ float s_incl[kSampleThreads];  // inclusive scan of the threads' run sums
  __shared__ float s_sum[kSampleThreads];   // the threads' run sums
  __shared__ float s_pmax, s_psum;          // this CTA's slice maximum and slice sum (read by the cluster)
  __shared__ float s_m;
  __shared__ float s_theta;  // u Z minus the sums of the slices before the owner
  __shared__ int s_owner, s_last, s_pick;

  const size_t row = blockIdx.x / kSplit;
  const uint32_t part = cluster_ctarank();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const float* x = logits + row * static_cast<size_t>(V);
  const int slice = ((V + kSplit - 1) / kSplit + 3) & ~3;
  const int lo = static_cast<int>(part) * slice;
  const int len = max(0, min(V, lo + slice) - lo);
  const float u_row = tid == 0 ? __ldg(uniforms + row) : 0.f;  // issued early, used after the sums

  // ---- stage the slice, slice maximum
  float mx = -INFINITY;
  if ((V & 3) == 0 && (reinterpret_cast<uintptr_t>(x) & 15) == 0) {
    const float4* x4 = reinterpret_cast<const float4*>(x + lo);
    float4* s4 = reinterpret_cast<float4*>(s_x);
    const int n4 = len / 4;
    for (int q0 = tid; q0 < n4; q0 += kSampleThreads * kLoadBatch) {
      float4 f[kLoadBatch];  // the batch's loads are all in flight before the first store
#pragma unroll
      for (int j = 0; j < kLoadBatch; ++j) {
        const int q = q0 + j * kSampleThreads;
        if (q < n4) f[j] = __ldg(x4 + q);
      }
#pragma unroll
      for (int j = 0; j < kLoadBatch; ++j) {
        const int q = q0 + j * kSampleThreads;
        if (q < n4) {
          s4[q] = f[j];
          mx = fmaxf(mx, fmaxf(fmaxf(f[j].x, f[j].y), fmaxf(f[j].z, f[j].w)));
        }
      }
    }
  } else {
    for (int i = tid; i < len; i += kSampleThreads) {
      const float f = __ldg(x + lo + i);
      s_x[i] = f;
      mx = fmaxf(mx, f);
    }
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  if (lane == 0) s_red[warp] = mx;
  __syncthreads();
  if (tid == 0) {
    float m = s_red[0];
#pragma unroll
    for (int w = 1; w < kSampleThreads / 32; ++w) m = fmaxf(m, s_red[w]);
    s_pmax = m;
  }
  cluster_sync();  // every slice maximum is published
  if (warp == 0) {  // the eight remote loads in parallel, one per lane
    float m = lane < kSplit ? ld_cluster_f32(&s_pmax, lane) : -INFINITY;
#pragma unroll
    for (int o = kSplit / 2; o; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    if (lane == 0) s_m = m;
  }
  __syncthreads();
  const float m = s_m;

  // ---- per-thread run sums of exp((x - m) / T) = 2^((x - m) log2(e) / T), contiguous runs (odd
  //      length: no bank conflicts)
  const float k2 = inv_t * 1.44269504f;  // log2(e) / T
  const int run = ((len + kSampleThreads - 1) / kSampleThreads) | 1;
  const int r0 = min(len, tid * run), r1 = min(len, r0 + run);
  float sum = 0.f;
  if (m > -INFINITY) {
    // the exps of a group are independent; only their sum is a chain (in id order)
    int i = r0;
    for (; i + 8 <= r1; i += 8) {
      float w[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) w[q] = exp2f((s_x[i + q] - m) * k2);
#pragma unroll
      for (int q = 0; q < 8; ++q) sum += w[q];
    }
    for (; i < r1; ++i) sum += exp2f((s_x[i] - m) * k2);
  }
  // inclusive scan in thread order
  float incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const float y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  __syncthreads();  // s_red is reused
  if (lane == 31) s_red[warp] = incl;
  __syncthreads();
  float base = 0.f;
  for (int w = 0; w < warp; ++w) base += s_red[w];
  incl += base;
  s_incl[tid] = incl;
  s_sum[tid] = sum;
  if (tid == kSampleThreads - 1) s_psum = incl;
  cluster_sync();  // every slice sum is published

  // ---- the owner slice: the same sequential combination in every CTA
  float my_sc = 0.f;
  if (warp == 0 && lane < kSplit) my_sc = ld_cluster_f32(&s_psum, lane);  // in parallel, one per lane
  float e[kSplit + 1];
  e[0] = 0.f;
  int last = -1;
  if (warp == 0) {
#pragma unroll
    for (int c = 0; c < kSplit; ++c) {
      const float sc = __shfl_sync(0xffffffffu, my_sc, c);
      if (sc > 0.f) last = c;
      e[c + 1] = e[c] + sc;
    }
  }
  if (tid == 0) {
    float u = u_row;
    if (!(u >= 0.f)) u = 0.f;
    if (u >= 1.f) u = __uint_as_float(0x3F7FFFFFu);  // the largest float below 1
    const float theta = u * e[kSplit];
    int owner = -1;
    float before = 0.f;  // the sum of the slices before the owner
#pragma unroll
    for (int c = 0; c < kSplit; ++c)
      if (owner < 0 && e[c + 1] > theta) { owner = c; before = e[c]; }
    s_last = owner < 0;
    if (owner < 0) {
#pragma unroll
      for (int c = 0; c < kSplit; ++c)
        if (c == last) before = e[c];
      owner = last;
    }
    s_owner = owner;
    s_theta = owner >= 0 ? theta - before : 0.f;
    s_pick = kSampleThreads;
    if (m == -INFINITY && part == 0) row_sample[row] = 0;  // no finite value
  }
  __syncthreads();
  if (m > -INFINITY && s_owner == static_cast<int>(part)) {
    const float th = s_theta;
    // the first thread of non-zero weight whose inclusive sum passes th (the scan need not be
    // monotone in fp32: the first one is unique); none: the last thread of non-zero weight
    if (!s_last && sum > 0.f && incl > th) atomicMin(&s_pick, tid);
    __syncthreads();
    if (tid == 0 && s_pick == kSampleThreads) {
      s_last = 1;
      int t = 0;
      for (int j = kSampleThreads - 1; j >= 0; --j)
        if (s_sum[j] > 0.f) { t = j; break; }
      s_pick = t;
    }
    __syncthreads();
    if (warp == 0) {  // the picked thread's run, 32 ids at a time: weights, a warp scan, a ballot
      const int t = s_pick;
      const int q0 = min(len, t * run), q1 = min(len, q0 + run);
      const float th2 = s_last ? INFINITY : th - (t ? s_incl[t - 1] : 0.f);
      float carry = 0.f;
      int y = -1, lastnz = -1;
      for (int i0 = q0; i0 < q1 && y < 0; i0 += 32) {
        const int i = i0 + lane;
        const float w = i < q1 ? exp2f((s_x[i] - m) * k2) : 0.f;
        float c = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const float z = __shfl_up_sync(0xffffffffu, c, o);
          if (lane >= o) c += z;
        }
        c += carry;
        const unsigned nz = __ballot_sync(0xffffffffu, w > 0.f);  // ids of zero weight are never drawn
        const unsigned hit = __ballot_sync(0xffffffffu, w > 0.f && c > th2);
        if (hit) y = i0 + __ffs(hit) - 1;
        if (nz) lastnz = i0 + 31 - __clz(nz);
        carry = __shfl_sync(0xffffffffu, c, 31);
      }
      // the picked run has non-zero weight, so lastnz is set (q0 < len otherwise)
      if (lane == 0) row_sample[row] = lo + (y >= 0 ? y : (lastnz >= 0 ? lastnz : min(q0, len - 1)));
    }
  }
  cluster_sync();  // no CTA leaves while another may still read its slice sum
}

cudaError_t launch_verify_sample(const float* logits, const int32_t* parent, const int32_t* token,
                                 const float* uniforms, int B, int N, int V, float inv_t, int32_t* row_sample,
                                 int32_t* nodes, int32_t* count, int32_t* bonus, cudaStream_t stream) {
  const long long rows = static_cast<long long>(B) * (N + 1);
  if (rows <= 0 || rows * kSplit > 0x7fffffffLL) return cudaErrorInvalidValue;
  const int slice = ((V + kSplit - 1) / kSplit + 3) & ~3;
  if (slice > kMaxSampleSlice) return cudaErrorInvalidValue;
  const size_t smem = static_cast<size_t>(slice) * sizeof(float);
  static bool attr_set = false;  // the largest staging size is set once per process
  if (!attr_set) {
    const cudaError_t e = cudaFuncSetAttribute(row_sample_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               kMaxSampleSlice * static_cast<int>(sizeof(float)));
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(rows * kSplit));
  cfg.blockDim = dim3(kSampleThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kSplit;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaError_t e = cudaLaunchKernelEx(&cfg, row_sample_kernel, logits, V, inv_t, uniforms, row_sample);
  if (e != cudaSuccess) return e;
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_walk(parent, token, row_sample, B, N, nodes, count, bonus, stream);
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
  return launch_walk(parent, token, row_argmax, B, N, nodes, count, bonus, stream);
}

}  // namespace dm
