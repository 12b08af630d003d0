// Host-visible interface of the tensor-core fork-decode kernel (internal).
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "plan.h"

namespace specgen {

struct TcParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_pages;  // used directly with the tiled layout (bulk copies)
  const __nv_bfloat16* v_pages;
  const int32_t* prefix_bt;
  const int32_t* prefix_bt_off;
  const int32_t* suffix_bt;
  const int32_t* suffix_bt_off;
  const TcItem* items;
  const int32_t* cta_offsets;  // [grid + 1]: CTA c takes items [cta_offsets[c], cta_offsets[c+1])
  const int32_t* part_base;    // [forks] first partial slot of each fork
  float* part_o;               // head-interleaved partials (part_o_f4)
  float* part_lse;             // [slots][hq]
  uint32_t* status;
  const int32_t* suffix_lens;  // device lengths that clamp suffix items, or nullptr
  int hq, hkv, G, dv, num_pages;
  float scale_log2;            // softmax scale * log2(e), > 0
  // 1: this grid follows the suffix-stage kernel in the stream and runs beside
  // it.  It is launched only once every suffix-stage CTA has passed its wait for
  // the kernel before both, so it starts without a wait of its own; it waits for
  // the suffix-stage grid at its end instead, so that the merge, which waits for
  // this grid, sees the suffix partials too.
  int wait_at_end;
};

bool fork_tc_supported(int dqk, int dv, bool latent, int page_size, int G);
// Tensor map of a paged pool [num_pages][hkv][16][D] bf16 whose box is one whole
// (page, head) block, landing as [D/64 panels][16 rows][128 B], 128-byte swizzled.
bool fork_tc_block_map(CUtensorMap* map, const void* pool, int D, int hkv, int num_pages);
int fork_tc_tile_tokens(int dqk);
int fork_tc_page_size();
// causal: the plan holds causal suffix items (TcItem::row_limit0 > 0)
cudaError_t launch_fork_tc(const TcParams& p, const void* k_pages, const void* v_pages, int grid,
                           int dqk, bool tiled, bool causal, cudaStream_t stream);

}  // namespace specgen
