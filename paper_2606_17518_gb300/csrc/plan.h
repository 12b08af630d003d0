// Work-list records shared by the host planner and the kernels (internal).
//
// A fork-decode call is cut into work items, each producing one partial
// attention (O normalised by its own softmax sum, plus its LSE) over a
// contiguous range of logical tokens of one paged sequence.  Every (fork, head)
// row owns `n_parts` consecutive partial slots starting at `part_base`; the
// merge kernel combines them by log-sum-exp.
#pragma once
#include <stddef.h>
#include <stdint.h>

namespace specgen {

// Partial outputs in the workspace, "head-interleaved": element (slot, head h,
// value column c) of part_o sits at ((slot * dv/4 + c/4) * hq + h) * 4 + c%4, so
// threads that hold consecutive heads store (and the merge loads) consecutive
// 16-byte pieces.  part_lse is [slot][hq].  Index of the float4 (slot, h, c4):
#ifdef __CUDACC__
__host__ __device__
#endif
inline size_t part_o_f4(size_t slot, int h, int c4, int hq, int dv) {
  return (slot * (size_t)(dv / 4) + (size_t)c4) * (size_t)hq + (size_t)h;
}

constexpr uint32_t kStatusIndex = 1u;    // a page id outside [0, num_pages) was seen
constexpr uint32_t kStatusTimeout = 2u;  // a device wait hit its iteration limit

// Split-K paged decode item: query rows [h0, h0+nrows) of one fork against
// tokens [tok_begin, tok_end) of one sequence (the fork's trace prefix or the
// fork's own suffix), value columns [dv0, dv0 + tile width).
struct SplitItem {
  int32_t fork;
  int32_t table_kind;  // 0: prefix table of trace `seq`; 1: suffix table of fork `seq`
  int32_t seq;
  int32_t kv_head;
  int32_t h0;
  int32_t nrows;
  int32_t dv0;
  int32_t tok_begin;
  int32_t tok_end;
  int32_t slot;        // partial slot of rows h0.. (part_o_f4 layout), part_lse[slot][h]
};

// Tensor-core item (shared prefix or one fork's suffix): the query rows of
// forks [fork0, fork0 + nforks) for kv head `kv_head` (nforks * G <= 128 rows)
// against tokens [tok_begin, tok_end) of one paged sequence.  Row (fork, head)
// writes partial slot part_base[fork] + part.
struct TcItem {
  int32_t table_kind;  // 0: prefix table of trace `seq`; 1: suffix table of fork `seq`
  int32_t seq;
  int32_t kv_head;
  int32_t fork0;
  int32_t nforks;
  int32_t tok_begin;
  int32_t tok_end;
  int32_t part;
  int32_t dv0;         // first value column this item produces (latent KV: 0 or 256)
  int32_t table_off;   // index of the sequence's first page in its block table, or -1
                       // (then the kernel reads it from the device offset array)
  int32_t row_limit0;  // causal suffix items (prefill chunks): query row r of the item
                       // sees only tokens < row_limit0 + r / G; 0 = every token
};

// Plan header at the start of the plan region.
struct PlanHeader {
  int32_t n_split, n_tc, n_tc_ctas, n_forks;
  int32_t split_off, tc_off, cta_items_off, cta_offsets_off, part_base_off, n_parts_off;
  // suffix-stage items (TcItem records, worker order) and the worker ranges
  // ([n_sfx_ctas * suffix warps + 1] offsets)
  int32_t n_sfx, n_sfx_ctas, sfx_off, sfx_offsets_off;
};

}  // namespace specgen
