// Log-sum-exp merge kernels.
//
// Partial attentions over disjoint key sets combine exactly: with
// m = max_i LSE_i and w_i = exp(LSE_i - m),
//     O = sum_i w_i O_i / sum_i w_i,   LSE = m + ln sum_i w_i,
// where each O_i is normalised by its own softmax sum.  Parts with LSE = -inf
// are empty and get weight 0.  One warp handles one (fork, head) row; lanes
// own 4-column float4 slices so the partial rows are read fully coalesced.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "lse_merge.h"

namespace specgen {

namespace {

constexpr int kMergeWarps = 4;

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One warp per (fork, head) row.  Lane i holds the LSE (and then the weight) of
// part i, so the max and the normaliser are two warp reductions; the weighted
// sum then streams the parts' rows with four independent loads in flight.
__global__ void __launch_bounds__(kMergeWarps * 32) merge_parts_kernel(const MergeParams p) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * kMergeWarps + warp;
  if (row >= p.n_rows) return;
  const int f = row / p.hq, h = row % p.hq;
  const int base = p.part_base[f], n = p.n_parts[f];
  __nv_bfloat16* out = p.out + (size_t)row * p.dv;

  float m = -INFINITY;
  for (int i = lane; i < n; i += 32) m = fmaxf(m, p.part_lse[(size_t)(base + i) * p.hq + h]);
  m = warp_max(m);
  if (m == -INFINITY) {  // no keys at all: O = 0, LSE = -inf
    for (int c = lane; c < p.dv; c += 32) out[c] = __float2bfloat16_rn(0.f);
    if (lane == 0) p.lse[row] = -INFINITY;
    return;
  }
  float wsum = 0.f;
  for (int i0 = 0; i0 < n; i0 += 32) {
    const int i = i0 + lane;
    const float li = i < n ? p.part_lse[(size_t)(base + i) * p.hq + h] : -INFINITY;
    wsum += li == -INFINITY ? 0.f : fast_exp2((li - m) * kLog2e);
  }
  wsum = warp_sum(wsum);
  const float inv = 1.f / wsum;
  // every lane runs every iteration (the shuffles need the full warp); lanes
  // past the row's last column load nothing and store nothing
  for (int c0 = 0; c0 < p.dv / 4; c0 += 32) {
    const int c4 = c0 + lane;
    const bool active = c4 < p.dv / 4;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int i0 = 0; i0 < n; i0 += 32) {
      const int i = i0 + lane;
      const float li = i < n ? p.part_lse[(size_t)(base + i) * p.hq + h] : -INFINITY;
      const float wl = li == -INFINITY ? 0.f : fast_exp2((li - m) * kLog2e);
      const int cnt = n - i0 < 32 ? n - i0 : 32;
      int k = 0;
      for (; k + 4 <= cnt; k += 4) {
        float w[4];
        float4 v[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          w[e] = __shfl_sync(0xffffffffu, wl, k + e);
          v[e] = active ? reinterpret_cast<const float4*>(
                              p.part_o + ((size_t)(base + i0 + k + e) * p.hq + h) * p.dv)[c4]
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          if (w[e] == 0.f) continue;  // empty part: its row may hold anything
          acc.x += w[e] * v[e].x;
          acc.y += w[e] * v[e].y;
          acc.z += w[e] * v[e].z;
          acc.w += w[e] * v[e].w;
        }
      }
      for (; k < cnt; ++k) {
        const float we = __shfl_sync(0xffffffffu, wl, k);
        if (we == 0.f || !active) continue;
        const float4 v = reinterpret_cast<const float4*>(
            p.part_o + ((size_t)(base + i0 + k) * p.hq + h) * p.dv)[c4];
        acc.x += we * v.x;
        acc.y += we * v.y;
        acc.z += we * v.z;
        acc.w += we * v.w;
      }
    }
    __nv_bfloat162 lo = __floats2bfloat162_rn(acc.x * inv, acc.y * inv);
    __nv_bfloat162 hi = __floats2bfloat162_rn(acc.z * inv, acc.w * inv);
    uint2 packed;
    packed.x = *reinterpret_cast<uint32_t*>(&lo);
    packed.y = *reinterpret_cast<uint32_t*>(&hi);
    if (active) reinterpret_cast<uint2*>(out)[c4] = packed;
  }
  if (lane == 0) p.lse[row] = m + log2f(wsum) * kLn2;
}

template <typename T>
__device__ __forceinline__ float ld_as_float(const T* p, size_t i);
template <>
__device__ __forceinline__ float ld_as_float<float>(const float* p, size_t i) {
  return p[i];
}
template <>
__device__ __forceinline__ float ld_as_float<__nv_bfloat16>(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void st_from_float(float* p, size_t i, float v) { p[i] = v; }
__device__ __forceinline__ void st_from_float(__nv_bfloat16* p, size_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

// Two-way merge; out/lse may alias the a-side inputs (each element is read
// before it is written by the same thread).
template <typename T>
__global__ void __launch_bounds__(256) lse_merge2_kernel(const T* oa, const float* la,
                                                         const T* ob, const float* lb, T* o,
                                                         float* l, int rows, int dv) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * 8 + warp;
  if (row >= rows) return;
  const float a = la[row], b = lb[row];
  const float m = fmaxf(a, b);
  float wa = 0.f, wb = 0.f;
  if (m != -INFINITY) {
    wa = a == -INFINITY ? 0.f : fast_exp2((a - m) * kLog2e);
    wb = b == -INFINITY ? 0.f : fast_exp2((b - m) * kLog2e);
  }
  const float inv = m == -INFINITY ? 0.f : 1.f / (wa + wb);
  for (int c = lane; c < dv; c += 32) {
    const size_t i = (size_t)row * dv + c;
    float va = wa == 0.f ? 0.f : ld_as_float(oa, i);
    float vb = wb == 0.f ? 0.f : ld_as_float(ob, i);
    st_from_float(o, i, (wa * va + wb * vb) * inv);
  }
  __syncwarp();
  if (lane == 0) l[row] = m == -INFINITY ? -INFINITY : m + log2f(wa + wb) * kLn2;
}

}  // namespace

cudaError_t launch_merge_parts(const MergeParams& p, cudaStream_t stream) {
  if (p.n_rows == 0) return cudaSuccess;
  const int blocks = (p.n_rows + kMergeWarps - 1) / kMergeWarps;
  merge_parts_kernel<<<blocks, kMergeWarps * 32, 0, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t launch_lse_merge2(const void* oa, const float* la, const void* ob, const float* lb,
                              void* o, float* l, int rows, int dv, int dtype,
                              cudaStream_t stream) {
  if (rows == 0) return cudaSuccess;
  const int blocks = (rows + 7) / 8;
  if (dtype == 0) {
    lse_merge2_kernel<__nv_bfloat16><<<blocks, 256, 0, stream>>>(
        static_cast<const __nv_bfloat16*>(oa), la, static_cast<const __nv_bfloat16*>(ob), lb,
        static_cast<__nv_bfloat16*>(o), l, rows, dv);
  } else {
    lse_merge2_kernel<float><<<blocks, 256, 0, stream>>>(
        static_cast<const float*>(oa), la, static_cast<const float*>(ob), lb,
        static_cast<float*>(o), l, rows, dv);
  }
  return cudaGetLastError();
}

}  // namespace specgen
