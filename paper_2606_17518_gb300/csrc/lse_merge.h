// Host-visible interface of the log-sum-exp merge kernels (internal).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace specgen {

struct MergeParams {
  const float* part_o;       // head-interleaved partials (part_o_f4)
  const float* part_lse;     // [slots][hq]
  const int32_t* part_base;  // [forks]
  const int32_t* n_parts;    // [forks][n_groups]: slots used by each group of hq/n_groups heads
  __nv_bfloat16* out;        // [forks][hq][dv]
  float* lse;                // [forks][hq]
  int n_rows, hq, dv, n_groups;
  int max_parts;             // the most parts any row has (picks the batch width)
};

// after_dependent: launch as a programmatic dependent of the previous kernel on
// the stream (which must trigger griddepcontrol.launch_dependents); the merge
// waits for that kernel's completion before reading the partials.
cudaError_t launch_merge_parts(const MergeParams& p, cudaStream_t stream, bool after_dependent);
cudaError_t launch_lse_merge2(const void* oa, const float* la, const void* ob, const float* lb,
                              void* o, float* l, int rows, int dv, int dtype,
                              cudaStream_t stream);

}  // namespace specgen
