// Host-visible interface of the page pack / unpack kernel (internal).
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace specgen {

struct PackParams {
  uint4* k_pages;           // pool blocks as 16-byte words
  uint4* v_pages;           // or nullptr (latent pool)
  uint4* packed;
  const int32_t* table;     // [n_pages]
  uint32_t* status;         // or nullptr
  size_t k_block16, v_block16;  // 16-byte words per page of each pool
  int n_pages, num_pages;
  bool unpack;              // false: pool -> packed; true: packed -> pool
};

cudaError_t launch_pack_pages(const PackParams& p, int n_sm, cudaStream_t stream);

}  // namespace specgen
