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
#include "merge_row.cuh"
#include "plan.h"

namespace specgen {

namespace {


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

// One thread per (fork, 4-column slice, head), heads fastest: a warp reads
// consecutive heads' LSE words and float4 slices of each part (contiguous in
// the head-interleaved partial layout), all loads independent, so a row costs
// about two memory round trips.  With programmatic dependent launch the grid starts while the kernel
// producing the partials is still running and waits for it here.
constexpr int kMergeThreads = 128;  // small blocks can sit beside a running tensor-core CTA

// BATCH parts are loaded together; MIN_BLOCKS bounds the registers so that
// grids of several waves keep enough rows in flight per SM.
template <int BATCH, int MIN_BLOCKS>
__global__ void __launch_bounds__(kMergeThreads, MIN_BLOCKS) merge_parts_kernel(const MergeParams p) {
  // the next kernel of the stream may get launched now (it waits for this grid
  // before it uses anything this grid writes or reads)
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  const int c4n = p.dv / 4;
  const int gid = blockIdx.x * kMergeThreads + threadIdx.x;
  const bool live = gid < p.n_rows * c4n;
  const int h = gid % p.hq, rest = gid / p.hq;
  const int c4 = rest % c4n, f = rest / c4n;
  const int row = f * p.hq + h;
  // the plan is written by a host copy, never by a kernel: read it before the
  // wait, so that only the partials' loads follow the producing grid
  const int base = live ? p.part_base[f] : 0;
  const int n = live ? p.n_parts[f * p.n_groups + h / (p.hq / p.n_groups)] : 0;
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  if (!live) return;
  const RowMerge mr = merge_row<BATCH>(
      p.part_lse + (size_t)base * p.hq + h, (size_t)p.hq,
      reinterpret_cast<const float4*>(p.part_o) + part_o_f4(base, h, c4, p.hq, p.dv),
      (size_t)c4n * p.hq, n);
  store_merged(mr, p.out + (size_t)row * p.dv, c4, p.lse + row, c4 == 0);
}

// merge_parts_kernel with two 4-column slices per thread (c4 = 2 k and 2 k + 1
// of the same head): the form for grids of many waves.
template <int BATCH, int MIN_BLOCKS>
__global__ void __launch_bounds__(kMergeThreads, MIN_BLOCKS) merge_parts2_kernel(const MergeParams p) {
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  const int c4n = p.dv / 4, c2n = c4n / 2;
  const int gid = blockIdx.x * kMergeThreads + threadIdx.x;
  const bool live = gid < p.n_rows * c2n;
  const int h = gid % p.hq, rest = gid / p.hq;
  const int c4 = 2 * (rest % c2n), f = rest / c2n;
  const int row = f * p.hq + h;
  const int base = live ? p.part_base[f] : 0;
  const int n = live ? p.n_parts[f * p.n_groups + h / (p.hq / p.n_groups)] : 0;
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  if (!live) return;
  RowMerge r0, r1;
  merge_row2<BATCH>(p.part_lse + (size_t)base * p.hq + h, (size_t)p.hq,
                    reinterpret_cast<const float4*>(p.part_o) + part_o_f4(base, h, c4, p.hq, p.dv),
                    (size_t)c4n * p.hq, (size_t)p.hq, n, &r0, &r1);
  store_merged(r0, p.out + (size_t)row * p.dv, c4, p.lse + row, c4 == 0);
  store_merged(r1, p.out + (size_t)row * p.dv, c4 + 1, p.lse + row, false);
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

cudaError_t launch_merge_parts(const MergeParams& p, cudaStream_t stream, bool after_dependent) {
  if (p.n_rows == 0) return cudaSuccess;
  // Wide batches (one memory round trip for up to 16 parts) need many
  // registers, so few blocks fit on an SM.  A grid of several such waves takes
  // 4-part batches at 8 blocks per SM (one wave, more round trips); a one-wave
  // grid whose rows have at most 8 parts takes 8-part batches.
  static thread_local int configured = -1, sms = 0;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured != dev) {
    const void* kernels[4] = {reinterpret_cast<const void*>(merge_parts_kernel<16, 1>),
                              reinterpret_cast<const void*>(merge_parts_kernel<8, 4>),
                              reinterpret_cast<const void*>(merge_parts_kernel<4, 8>),
                              reinterpret_cast<const void*>(merge_parts2_kernel<4, 4>)};
    // keep the SMs in the shared-memory-heavy configuration of the kernels
    // around this one, so that no L1/shared-memory reconfiguration is needed
    for (const void* k : kernels) {
      e = cudaFuncSetAttribute(k, cudaFuncAttributePreferredSharedMemoryCarveout,
                               (int)cudaSharedmemCarveoutMaxShared);
      if (e != cudaSuccess) return e;
    }
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  const long long threads = (long long)p.n_rows * (p.dv / 4);
  long long blocks = (threads + kMergeThreads - 1) / kMergeThreads;
  int form = blocks > 3LL * sms ? 2 : (p.max_parts <= 8 ? 1 : 0);
  // grids of many waves over rows of few parts: two slices per thread (half
  // the threads, twice the bytes in flight each; with many parts per row the
  // one-slice form keeps more rows in flight)
  if (form == 2 && p.max_parts <= 8 && (p.dv / 4) % 2 == 0) {
    form = 3;
    blocks = (threads / 2 + kMergeThreads - 1) / kMergeThreads;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)blocks);
  cfg.blockDim = dim3(kMergeThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = after_dependent ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  if (form == 3) return cudaLaunchKernelEx(&cfg, merge_parts2_kernel<4, 4>, p);
  if (form == 2) return cudaLaunchKernelEx(&cfg, merge_parts_kernel<4, 8>, p);
  if (form == 1) return cudaLaunchKernelEx(&cfg, merge_parts_kernel<8, 4>, p);
  return cudaLaunchKernelEx(&cfg, merge_parts_kernel<16, 1>, p);
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
