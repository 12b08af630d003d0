// Pack / unpack of a paged sequence for the remote prefix cache.
//
// A suspended trace's prefix KV leaves the GPU and comes back later
// (Section 6.2.3); on the device that is a gather of the sequence's pages into
// one contiguous buffer and a scatter back under a new block table.  A page of
// a pool ([num_pages][Hkv][B][D]) is one contiguous block, so both directions
// are block copies: buffer word w belongs to section s (K, then V), page i and
// offset o, and pairs with word o of block table[i] of that section's pool.
// Grid-stride over the buffer's 16-byte words, four independent words per
// thread in flight; a page id outside the pool is skipped and reported.  The
// kernel is a programmatic dependent: it waits for the stream's previous
// kernel before it reads anything and lets the next one launch at once.
#include <cuda_runtime.h>

#include "pack_pages.h"
#include "plan.h"

namespace specgen {

namespace {

constexpr int kThreads = 256;
constexpr int kUnroll = 4;

__global__ void __launch_bounds__(kThreads) pack_pages_kernel(const PackParams p) {
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  const size_t nk = (size_t)p.n_pages * p.k_block16;
  const size_t total = nk + (p.v_pages ? (size_t)p.n_pages * p.v_block16 : 0);
  const size_t stride = (size_t)gridDim.x * kThreads * kUnroll;
  for (size_t w0 = ((size_t)blockIdx.x * kThreads) * kUnroll + threadIdx.x; w0 < total;
       w0 += stride) {
    uint4 v[kUnroll];
    uint4* pool_at[kUnroll];
    bool ok[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const size_t w = w0 + (size_t)u * kThreads;
      ok[u] = false;
      pool_at[u] = nullptr;
      if (w >= total) continue;
      const bool is_v = w >= nk;
      const size_t blk = is_v ? p.v_block16 : p.k_block16;
      const size_t r = is_v ? w - nk : w;
      const size_t i = r / blk, o = r % blk;
      const int page = p.table[i];
      if (page < 0 || page >= p.num_pages) {
        if (o == 0 && p.status) atomicOr(p.status, kStatusIndex);
        continue;
      }
      ok[u] = true;
      pool_at[u] = (is_v ? p.v_pages : p.k_pages) + (size_t)page * blk + o;
      v[u] = p.unpack ? p.packed[w] : *pool_at[u];
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      if (!ok[u]) continue;
      if (p.unpack)
        *pool_at[u] = v[u];
      else
        p.packed[w0 + (size_t)u * kThreads] = v[u];
    }
  }
}

}  // namespace

cudaError_t launch_pack_pages(const PackParams& p, int n_sm, cudaStream_t stream) {
  const size_t total = (size_t)p.n_pages * (p.k_block16 + (p.v_pages ? p.v_block16 : 0));
  if (total == 0) return cudaSuccess;
  const size_t per_cta = (size_t)kThreads * kUnroll;
  size_t grid = (total + per_cta - 1) / per_cta;
  const size_t cap = (size_t)n_sm * 8;  // enough CTAs in flight to cover HBM latency
  if (grid > cap) grid = cap;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, pack_pages_kernel, p);
}

}  // namespace specgen
