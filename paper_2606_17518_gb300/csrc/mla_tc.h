// Host-visible interface of the latent-KV (MLA-style) tensor-core kernel (internal).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "plan.h"

namespace specgen {

struct MlaParams {
  const __nv_bfloat16* q;      // [forks][128][576]
  const int32_t* prefix_bt;
  const int32_t* prefix_bt_off;
  const int32_t* suffix_bt;
  const int32_t* suffix_bt_off;
  const TcItem* items;         // dv0 selects the value half (0 or 256)
  const int32_t* cta_offsets;  // [grid + 1]: CTA c takes items [cta_offsets[c], cta_offsets[c+1])
  const int32_t* part_base;
  float* part_o;               // head-interleaved partials (part_o_f4), hq = 128, dv = 512
  float* part_lse;             // [slots][128]
  uint32_t* status;
  const int32_t* suffix_lens;  // device lengths that clamp suffix items, or nullptr
  int hq, num_pages;
  float scale_log2;
};

bool mla_tc_supported(int dqk, int dv, bool latent, int page_size, int hq, int hkv);
int mla_tc_tile_tokens();
cudaError_t launch_mla_tc(const MlaParams& p, const void* k_pages, int grid, cudaStream_t stream);

}  // namespace specgen
