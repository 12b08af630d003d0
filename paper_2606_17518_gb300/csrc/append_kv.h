// Host-visible interface of the decode-step append kernel (internal).
#pragma once
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace specgen {

struct AppendParams {
  const __nv_bfloat16* k_new;  // [F][hkv][dqk]
  const __nv_bfloat16* v_new;  // [F][hkv][dv] or nullptr (latent pool)
  __nv_bfloat16* k_pages;
  __nv_bfloat16* v_pages;
  int32_t* table;              // suffix block table (CSR, capacity per fork)
  const int32_t* offs;         // [F + 1]
  const int32_t* lens;         // [F] tokens already in each suffix
  int32_t* lens_next;          // [F] lengths after the call, or nullptr (never lens itself)
  const int32_t* free_pages;
  uint32_t* status;            // or nullptr
  int F, hkv, dqk, dv, B, num_pages, num_free;
  bool tiled;                  // 8x8 core-matrix blocks instead of token rows
};

cudaError_t launch_append_kv(const AppendParams& p, cudaStream_t stream);

}  // namespace specgen
