// Combining a row's partial attentions, latency-tolerant form (device helper).
//
// A row owns n partials (O_i normalised by its own sum, LSE_i).  They are
// combined online in batches of BATCH: the batch's LSE words and float4
// output slices are loaded together (independent loads, one memory round trip
// per batch), the running maximum moves to the batch maximum and the accumulated
// sum is rescaled, exactly as in an online softmax:
//     m' = max(m, max_b LSE_i),  acc' = acc e^{m-m'} + sum_b e^{LSE_i-m'} O_i,
//     w' = w e^{m-m'} + sum_b e^{LSE_i-m'};   O = acc / w,  LSE = m + ln w.
// Parts with LSE = -inf are empty (their slices may hold anything).
#pragma once
#include "common.cuh"

namespace specgen {

struct RowMerge {
  float4 acc;
  float w, m;
};

// lse_p[i * lse_stride], o_p[i * o_stride] (float4 units) for i < n; L2 loads
// (the partials may have been written by other SMs during this kernel).
template <int BATCH>
__device__ __forceinline__ RowMerge merge_row(const float* lse_p, size_t lse_stride,
                                              const float4* o_p, size_t o_stride, int n) {
  RowMerge r;
  r.acc = make_float4(0.f, 0.f, 0.f, 0.f);
  r.w = 0.f;
  r.m = -INFINITY;
  for (int i0 = 0; i0 < n; i0 += BATCH) {
    float li[BATCH];
    float4 v[BATCH];
#pragma unroll
    for (int e = 0; e < BATCH; ++e) {
      const bool in = i0 + e < n;
      li[e] = in ? __ldcg(lse_p + (size_t)(i0 + e) * lse_stride) : -INFINITY;
      v[e] = in ? __ldcg(o_p + (size_t)(i0 + e) * o_stride) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float mb = r.m;
#pragma unroll
    for (int e = 0; e < BATCH; ++e) mb = fmaxf(mb, li[e]);
    if (mb == -INFINITY) continue;  // nothing yet
    const float sc = r.m == -INFINITY ? 0.f : fast_exp2((r.m - mb) * kLog2e);
    r.acc.x *= sc;
    r.acc.y *= sc;
    r.acc.z *= sc;
    r.acc.w *= sc;
    r.w *= sc;
    r.m = mb;
#pragma unroll
    for (int e = 0; e < BATCH; ++e) {
      if (li[e] == -INFINITY) continue;
      const float we = fast_exp2((li[e] - mb) * kLog2e);
      r.w += we;
      r.acc.x += we * v[e].x;
      r.acc.y += we * v[e].y;
      r.acc.z += we * v[e].z;
      r.acc.w += we * v[e].w;
    }
  }
  return r;
}

// merge_row for two 4-column slices of the same row (o_p and o_p + o_off2):
// one LSE load per part serves both, and twice the bytes are in flight per
// thread (for grids of many waves).
template <int BATCH>
__device__ __forceinline__ void merge_row2(const float* lse_p, size_t lse_stride,
                                           const float4* o_p, size_t o_stride, size_t o_off2,
                                           int n, RowMerge* r0, RowMerge* r1) {
  r0->acc = r1->acc = make_float4(0.f, 0.f, 0.f, 0.f);
  r0->w = r1->w = 0.f;
  r0->m = r1->m = -INFINITY;
  float m = -INFINITY, w = 0.f;
  float4 a0 = make_float4(0.f, 0.f, 0.f, 0.f), a1 = a0;
  for (int i0 = 0; i0 < n; i0 += BATCH) {
    float li[BATCH];
    float4 v0[BATCH], v1[BATCH];
#pragma unroll
    for (int e = 0; e < BATCH; ++e) {
      const bool in = i0 + e < n;
      const size_t o = (size_t)(i0 + e) * o_stride;
      li[e] = in ? __ldcg(lse_p + (size_t)(i0 + e) * lse_stride) : -INFINITY;
      v0[e] = in ? __ldcg(o_p + o) : make_float4(0.f, 0.f, 0.f, 0.f);
      v1[e] = in ? __ldcg(o_p + o + o_off2) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float mb = m;
#pragma unroll
    for (int e = 0; e < BATCH; ++e) mb = fmaxf(mb, li[e]);
    if (mb == -INFINITY) continue;  // nothing yet
    const float sc = m == -INFINITY ? 0.f : fast_exp2((m - mb) * kLog2e);
    a0.x *= sc; a0.y *= sc; a0.z *= sc; a0.w *= sc;
    a1.x *= sc; a1.y *= sc; a1.z *= sc; a1.w *= sc;
    w *= sc;
    m = mb;
#pragma unroll
    for (int e = 0; e < BATCH; ++e) {
      if (li[e] == -INFINITY) continue;
      const float we = fast_exp2((li[e] - mb) * kLog2e);
      w += we;
      a0.x += we * v0[e].x; a0.y += we * v0[e].y; a0.z += we * v0[e].z; a0.w += we * v0[e].w;
      a1.x += we * v1[e].x; a1.y += we * v1[e].y; a1.z += we * v1[e].z; a1.w += we * v1[e].w;
    }
  }
  r0->acc = a0;
  r1->acc = a1;
  r0->w = r1->w = w;
  r0->m = r1->m = m;
}

// Final bf16 slice and natural-log LSE of a merged row.
__device__ __forceinline__ void store_merged(const RowMerge& r, __nv_bfloat16* out_row, int c4,
                                             float* lse_out, bool write_lse) {
  const float inv = r.w > 0.f ? 1.f / r.w : 0.f;
  __nv_bfloat162 lo = __floats2bfloat162_rn(r.acc.x * inv, r.acc.y * inv);
  __nv_bfloat162 hi = __floats2bfloat162_rn(r.acc.z * inv, r.acc.w * inv);
  uint2 packed;
  packed.x = *reinterpret_cast<uint32_t*>(&lo);
  packed.y = *reinterpret_cast<uint32_t*>(&hi);
  reinterpret_cast<uint2*>(out_row)[c4] = packed;
  if (write_lse) *lse_out = r.m == -INFINITY ? -INFINITY : r.m + log2f(r.w) * kLn2;
}

}  // namespace specgen
