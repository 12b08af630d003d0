// Host-visible interface of the split-K paged decode kernel (internal).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "plan.h"

namespace specgen {

struct SplitParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_pages;
  const __nv_bfloat16* v_pages;  // unused for latent KV
  const int32_t* prefix_bt;
  const int32_t* prefix_bt_off;
  const int32_t* suffix_bt;
  const int32_t* suffix_bt_off;
  const SplitItem* items;
  float* part_o;    // head-interleaved partials (part_o_f4)
  float* part_lse;  // [slots][hq]
  uint32_t* status;
  const int32_t* suffix_lens;  // device lengths that clamp suffix items, or nullptr
  int hq, hkv, dqk, dv, page_size, num_pages;
  float scale_log2;  // softmax scale * log2(e)
};

bool split_variant_supported(int dqk, int dv, bool latent);
int split_dv_tile(int dqk, int dv, bool latent);
cudaError_t launch_split_decode(const SplitParams& p, int n_items, bool latent,
                                cudaStream_t stream);

}  // namespace specgen
