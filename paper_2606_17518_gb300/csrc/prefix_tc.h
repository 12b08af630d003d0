// Host-visible interface of the tensor-core shared-prefix kernel (internal).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "plan.h"

namespace specgen {

struct PrefixParams {
  const __nv_bfloat16* q;
  const int32_t* prefix_bt;
  const int32_t* prefix_bt_off;
  const PrefixItem* items;
  const int32_t* part_base;  // [forks] first partial slot of each fork
  float* part_o;             // [slots][hq][dv]
  float* part_lse;           // [slots][hq]
  uint32_t* status;
  int hq, hkv, G, dv, page_size, num_pages;
  float scale_log2;          // softmax scale * log2(e)
};

bool prefix_tc_supported(int dqk, int dv, bool latent, int page_size, int G);
int prefix_tc_tile_tokens();
int prefix_tc_page_size();
cudaError_t launch_prefix_tc(const PrefixParams& p, const void* k_pages, const void* v_pages,
                             int n_items, int dqk, cudaStream_t stream);

}  // namespace specgen
