// Decode-step append: one new key/value row per fork into its paged suffix.
//
// Every fork decodes its own continuation after a fork event while the prefix
// stays shared (Algorithm 1; Section 4.2), so each step adds one K/V row per
// fork.  Fork f with n = lens[f] tokens already in its suffix writes slot
// n % B of page table[offs[f] + n / B]; when n % B == 0 that page is new: the
// fork takes free_pages[j], j = the number of forks before f that also start
// a page this step (fork order), and records it in its block table.  One warp
// per fork: the lanes count those earlier forks, then copy the fork's rows
// (all kv heads) 16 bytes a lane.  A fork whose table is full, whose free-list
// entry does not exist or whose page id is outside the pool writes nothing and
// raises the index bit of the status word.  With lens_next, lane 0 of a fork's
// warp also writes the fork's length after the call there (a separate array:
// the counts of other forks still read lens).  The kernel waits for the
// stream's previous kernel before it reads anything and lets the next kernel
// launch at once (that kernel waits for this one's completion before it reads
// the pools, tables or lengths).
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "append_kv.h"
#include "plan.h"

namespace specgen {

namespace {

constexpr int kWarps = 4;

__device__ __forceinline__ void copy_rows(__nv_bfloat16* pool, const __nv_bfloat16* rows, int f,
                                          int page, int slot, int hkv, int width, int B,
                                          bool tiled, int lane) {
  const int chunks = width / 8;  // 16-byte pieces of one row
  for (int x = lane; x < hkv * chunks; x += 32) {
    const int g = x / chunks, c = x % chunks;
    const uint4 v = reinterpret_cast<const uint4*>(rows + ((size_t)f * hkv + g) * width)[c];
    const size_t block = ((size_t)page * hkv + g) * (size_t)B * width;
    const size_t at = tiled ? ((size_t)(slot / 8) * chunks + c) * 64 + (slot % 8) * 8
                            : (size_t)slot * width + (size_t)c * 8;
    *reinterpret_cast<uint4*>(pool + block + at) = v;
  }
}

__global__ void __launch_bounds__(32 * kWarps) append_kv_kernel(const AppendParams p) {
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int f = blockIdx.x * kWarps + warp;
  if (f >= p.F) return;
  int j = 0;
  for (int i = lane; i < f; i += 32) j += (p.lens[i] % p.B == 0) ? 1 : 0;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) j += __shfl_xor_sync(0xffffffffu, j, o);
  const int n = p.lens[f];
  const int pidx = n / p.B, slot = n % p.B;
  const int off = p.offs[f], cap = p.offs[f + 1] - off;
  bool bad = n < 0 || pidx >= cap;
  int page = -1;
  if (!bad) {
    page = slot == 0 ? (j < p.num_free ? p.free_pages[j] : -1) : p.table[off + pidx];
    bad = page < 0 || page >= p.num_pages;
  }
  if (lane == 0 && p.lens_next) p.lens_next[f] = bad ? n : n + 1;
  if (bad) {
    if (lane == 0 && p.status) atomicOr(p.status, kStatusIndex);
    return;
  }
  if (slot == 0 && lane == 0) p.table[off + pidx] = page;
  copy_rows(p.k_pages, p.k_new, f, page, slot, p.hkv, p.dqk, p.B, p.tiled, lane);
  if (p.v_pages) copy_rows(p.v_pages, p.v_new, f, page, slot, p.hkv, p.dv, p.B, p.tiled, lane);
}

}  // namespace

cudaError_t launch_append_kv(const AppendParams& p, cudaStream_t stream) {
  if (p.F == 0) return cudaSuccess;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((p.F + kWarps - 1) / kWarps));
  cfg.blockDim = dim3(32 * kWarps);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, append_kv_kernel, p);
}

}  // namespace specgen
