// Host-visible interface of the suffix-stage kernel (internal).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "plan.h"

namespace specgen {

// Worker warps of a suffix-stage CTA (each walks its own list of items), page
// slots in each worker's ring, and suffix-stage CTAs resident on one SM.
constexpr int kSuffixWarps = 8;
constexpr int kSuffixSlots = 3;
constexpr int kSuffixCtasPerSm = 1;
// Group sizes served (one or two n-tiles of 8 query heads).
constexpr int kSuffixMaxG = 16;

struct SfxParams {
  const __nv_bfloat16* q;
  const __nv_bfloat16* k_pages;  // read directly with the tiled layout (bulk copies)
  const __nv_bfloat16* v_pages;
  const int32_t* suffix_bt;
  const int32_t* suffix_bt_off;
  const TcItem* items;           // suffix items (table_kind 1, one query row each)
  const int32_t* worker_offsets; // [grid * kSuffixWarps + 1]: worker w takes items
                                 // [worker_offsets[w], worker_offsets[w + 1])
  const int32_t* part_base;      // [rows] first partial slot of each query row
  float* part_o;                 // head-interleaved partials (part_o_f4)
  float* part_lse;               // [slots][hq]
  uint32_t* status;
  const int32_t* suffix_lens;    // device lengths that clamp the items, or nullptr
  int hq, hkv, G, dv, num_pages;
  float scale_log2;              // softmax scale * log2(e), > 0
  // This grid is the first partial-attention kernel of a call: it waits for the
  // stream's previous kernel before it touches anything.  late_trigger 1: the
  // prefix kernel follows it in the stream and runs beside it, so this grid's
  // dependents are released only once every CTA has passed that wait (the
  // prefix kernel then starts without a wait of its own); 0: they (the merge)
  // are released at the start.
  int late_trigger;
};

bool suffix_stage_supported(int dqk, int dv, bool latent, int page_size, int G);
cudaError_t launch_suffix_stage(const SfxParams& p, const void* k_pages, const void* v_pages,
                                int grid, int dqk, bool tiled, cudaStream_t stream);

}  // namespace specgen
