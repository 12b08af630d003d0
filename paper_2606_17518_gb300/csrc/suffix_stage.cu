// Suffix stage of fork decode: a split-K, bandwidth-bound paged decode kernel
// that runs beside the tensor-core prefix kernel, each on its own share of the
// SMs (launched first, this grid takes its share; the prefix kernel, launched
// once every CTA here has passed the wait for the previous kernel, the rest).
//
// The suffix of one fork is private to that fork, so its keys serve only the
// G = hq / hkv query heads of one kv head: a 128-row tensor-core tile would
// carry G live rows.  Here every warp of a suffix-stage CTA is an independent
// worker with its own list of (fork, kv head, page range) items and its own
// ring of page slots:
//
//   - one lane per copy issues the page's K block and V block (4 KB each at
//     head dim 128) into the ring slot with one bulk copy each (tiled pools:
//     cp.async.bulk of the contiguous block; token-major pools: one TMA box of
//     the whole block, 128-byte swizzled so that the 8x8 matrix loads below hit
//     eight different bank groups), completing on the slot's mbarrier; the
//     item's query rows come the same way into a per-warp buffer;
//   - S^T = K Q^T on mma.sync m16n8k16 with the page's 16 tokens on M and the
//     query heads on N (8 per n-tile, so G = 8 fills the instruction), K read
//     with ldmatrix from the slot;
//   - softmax in fp32 over the tokens: each thread holds two tokens of two
//     heads, the row max and (at the item's end) the row sum are reduced with
//     three xor shuffles over the eight lanes of a head; running max in log2
//     units with lazy rescaling (only when it grows by more than 2^8);
//   - P^T goes back into registers as the B operand of O^T += V^T P^T with one
//     movmatrix transpose per 8x8 block, V^T read with ldmatrix.trans;
//   - at the item's end the partial (O / l, LSE) of its G rows is stored in the
//     head-interleaved partial layout that the merge reads.
//
// Items are cut at page boundaries by the planner and clamped by the optional
// device suffix lengths; a token past an item's end, or on a page id outside
// the pool, gets score -inf, and its value row is zeroed in shared memory before
// the PV product (stale or NaN data must not reach the output).  Every wait is
// bounded; before the warp leaves, every copy it issued has landed.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "common.cuh"
#include "fork_tc.h"
#include "plan.h"
#include "suffix_stage.h"
#include "tc_common.cuh"

namespace specgen {
namespace {

using namespace tc;

constexpr int kPage = 16;                    // tokens per page (the tensor-core path's page size)
constexpr int kSlots = kSuffixSlots;         // ring slots (pages) per warp
constexpr float kRescale = 8.0f;             // lazy-rescale threshold, log2 units

__device__ __forceinline__ uint32_t movmatrix_trans(uint32_t a) {
  uint32_t d;
  asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;\n" : "=r"(d) : "r"(a));
  return d;
}

// Shared memory of a suffix-stage CTA: per worker warp, kSlots page slots (K
// block, then V block) and one query buffer of 8 * NT rows; then per warp
// kSlots + 1 mbarriers and the slots' valid-page flags; per warp its first
// kCache items; then the abort flag.
template <int D, int NT>
struct Layout {
  static constexpr uint32_t kBlk = kPage * D * 2u;
  static constexpr uint32_t kSlot = 2u * kBlk;
  static constexpr uint32_t kQ = 8u * NT * D * 2u;
  static constexpr uint32_t kWarp = kSlots * kSlot + kQ;
  static constexpr uint32_t kBar = kSuffixWarps * kWarp;
  // kSlots + 1 mbarriers and kSlots flags, in 64-byte units
  static constexpr uint32_t kWarpBar = (8u * (kSlots + 1) + 4u * kSlots + 63u) / 64u * 64u;
  static constexpr int kCache = NT == 1 ? 16 : 4;
  static constexpr uint32_t kItems = kBar + kSuffixWarps * kWarpBar;
  static constexpr uint32_t kAbort = kItems + kSuffixWarps * kCache * (uint32_t)sizeof(TcItem);
  static constexpr uint32_t kBytes = kAbort + 16u;
  static_assert(kBlk % 1024 == 0 && kQ % 1024 == 0, "slots stay 1024-byte aligned");
  static_assert(8 * (kSlots + 1) + 4 * kSlots <= (int)kWarpBar, "per-warp barrier block");
};

// Byte offset of the 16-byte piece (token t, 8-column chunk c) of one
// (page, head) block in shared memory.  Tiled pools land as the pool stores
// them (8x8 core matrices of 128 contiguous bytes); token-major pools land as
// [64-column panel][16 rows][128 B] with the 128-byte swizzle (chunk index
// XOR row mod 8).
template <int D, bool TL>
__device__ __forceinline__ uint32_t piece(int t, int c) {
  if constexpr (TL)
    return (uint32_t)((((t >> 3) * (D / 8) + c) << 7) + ((t & 7) << 4));
  else
    return (uint32_t)(((c >> 3) << 11) + (t << 7) + (((c & 7) ^ (t & 7)) << 4));
}

// One worker warp: worker blockIdx.x * kSuffixWarps + warp of the grid.
template <int D, bool TL, int NT>
__device__ __forceinline__ void suffix_warp(const SfxParams& p, const CUtensorMap* tmk,
                                            const CUtensorMap* tmv, uint32_t sbase,
                                            unsigned char* gbase, int warp,
                                            volatile int* abort_flag) {
  using L = Layout<D, NT>;
  constexpr int KS = D / 16;  // k-steps of Q K^T, m-tiles of V^T P^T
  const int lane = threadIdx.x & 31;
  const int g8 = lane >> 2, tig = lane & 3;
  const int G = p.G;
  const int worker = blockIdx.x * kSuffixWarps + warp;
  const int ib = p.worker_offsets[worker];
  const int n_items = p.worker_offsets[worker + 1] - ib;
  const uint32_t wslot = sbase + (uint32_t)warp * L::kWarp;
  const uint32_t sQ = wslot + kSlots * L::kSlot;
  const uint32_t bar = sbase + L::kBar + (uint32_t)warp * L::kWarpBar;
  auto full = [&](int s) { return bar + 8u * (uint32_t)s; };
  const uint32_t qbar = bar + 8u * kSlots;
  volatile int* sflag =
      reinterpret_cast<volatile int*>(gbase + L::kBar + warp * L::kWarpBar + 8 * (kSlots + 1));

  if (lane == 0) {
    for (int s = 0; s <= kSlots; ++s) mbar_init(bar + 8u * s, 1);
    mbar_init_fence();
  }
  // this warp's first items, one coalesced read: the plan is written by a host
  // copy, never by a kernel, so it may be read before waiting for one
  TcItem* cache = reinterpret_cast<TcItem*>(gbase + L::kItems) + warp * L::kCache;
  const int n_cached = n_items < L::kCache ? n_items : L::kCache;
  {
    constexpr int kWords = sizeof(TcItem) / 4;
    const int32_t* src = reinterpret_cast<const int32_t*>(p.items + ib);
    int32_t* dst = reinterpret_cast<int32_t*>(cache);
    for (int x = lane; x < n_cached * kWords; x += 32) dst[x] = src[x];
  }
  __syncwarp();
  // Before waiting for the previous kernel (below), the warp asks L2 for
  // its first item's first pages and query rows, read with the item as
  // planned: only plans with host-resolved table offsets take part, so every
  // read here is of the plan or of table entries at positions the plan was made
  // for.  A prefetch moves nothing into this CTA: a table or length the previous
  // kernel still rewrites can at worst warm the wrong pages.  Not with the
  // prefix kernel behind this grid: there the requests would compete with the
  // previous call's last prefix CTAs, which are on the critical path.
  if (!p.late_trigger && n_cached > 0 && cache[0].table_off >= 0) {
    const TcItem it0 = cache[0];
    const int np0 = (it0.tok_end - it0.tok_begin + kPage - 1) / kPage;
    if (lane < kSlots && lane < np0) {
      const int page = p.suffix_bt[it0.table_off + it0.tok_begin / kPage + lane];
      if (page >= 0 && page < p.num_pages) {
        const size_t blk = ((size_t)page * p.hkv + it0.kv_head) * (kPage * D);
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(p.k_pages + blk),
                     "r"(L::kBlk)
                     : "memory");
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(p.v_pages + blk),
                     "r"(L::kBlk)
                     : "memory");
      }
    } else if (lane == kSlots) {
      asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(
                       p.q + ((size_t)it0.fork0 * p.hq + (size_t)it0.kv_head * G) * D),
                   "r"((uint32_t)G * D * 2u)
                   : "memory");
    }
  }
  // Inputs (device lengths, tables, Q, K/V) may be written by the stream's
  // previous kernel, and the partial buffers still read by it: this grid waits
  // for it here.  With the prefix kernel behind it, that kernel is released
  // only now (so it needs no wait of its own for the inputs).
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  if (p.late_trigger && threadIdx.x == 0)
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  if (lane < n_cached) cache[lane] = clamp_item(cache[lane], p.suffix_lens);
  __syncwarp();

  // item k: from the cache (cut to the device lengths), or read and cut here
  auto item = [&](int k) {
    return k < L::kCache ? cache[k] : clamp_item(p.items[ib + k], p.suffix_lens);
  };
  auto npages = [](const TcItem& it) { return (it.tok_end - it.tok_begin + kPage - 1) / kPage; };
  // page ids pb + lane of an item (0 past its end)
  auto ids = [&](const TcItem& it, int pb) -> int {
    if (pb + lane >= npages(it)) return 0;
    const int off = it.table_off >= 0 ? it.table_off : p.suffix_bt_off[it.seq];
    return p.suffix_bt[off + it.tok_begin / kPage + pb + lane];
  };
  // the first item at or after `from` with tokens (n_items if none)
  auto next_nonempty = [&](int from, TcItem& it) {
    int k = from;
    for (; k < n_items; ++k) {
      it = item(k);
      if (it.tok_end > it.tok_begin) break;
    }
    return k;
  };

  // ---- producer cursor: the item whose pages are being issued (pk), its page
  // ids 32 at a time, and the next non-empty item with its first ids loaded
  TcItem pit{}, nit{};
  int pk = n_items, pj = 0, pnp = 0, pb = 0, pid = 0;
  int nk = next_nonempty(0, nit);
  int npid = nk < n_items ? ids(nit, 0) : 0;
  auto advance_producer = [&]() {
    pk = nk;
    pit = nit;
    pid = npid;
    pj = 0;
    pb = 0;
    pnp = pk < n_items ? npages(pit) : 0;
    if (pk < n_items) {
      nk = next_nonempty(pk + 1, nit);
      npid = nk < n_items ? ids(nit, 0) : 0;
    }
  };
  advance_producer();
  int issued = 0, used = 0;
  auto issue = [&]() {  // page pj of item pk into slot issued % kSlots
    const int s = issued % kSlots;
    const int page = __shfl_sync(0xffffffffu, pid, pj - pb);
    const bool ok = page >= 0 && page < p.num_pages;
    if (lane == 0) {
      sflag[s] = ok ? 1 : 0;
      if (!ok) atomicOr(p.status, kStatusIndex);
      mbar_arrive_expect_tx(full(s), ok ? L::kSlot : 0u);
    }
    __syncwarp();
    if (ok && lane < 2) {  // lane 0 the K block, lane 1 the V block, in one instruction
      const uint32_t dst = wslot + (uint32_t)s * L::kSlot + (uint32_t)lane * L::kBlk;
      if constexpr (TL) {
        const __nv_bfloat16* src =
            (lane == 0 ? p.k_pages : p.v_pages) + ((size_t)page * p.hkv + pit.kv_head) * (kPage * D);
        bulk_load(dst, src, L::kBlk, full(s));
      } else {
        const CUtensorMap* m = lane == 0 ? tmk : tmv;
        if constexpr (D == 128)
          tma_load_5d(dst, m, 0, 0, 0, pit.kv_head, page, full(s));
        else
          tma_load_4d(dst, m, 0, 0, pit.kv_head, page, full(s));
      }
    }
    ++issued;
    if (++pj == pnp) {
      advance_producer();
    } else if (pj - pb == 32) {
      pb += 32;
      pid = ids(pit, pb);
    }
  };
  // the query rows of an item (G rows of D, contiguous in q) into the buffer
  int q_issued = 0, q_used = 0;
  auto issue_q = [&](const TcItem& it) {
    if (lane == 0) {
      const uint32_t bytes = (uint32_t)G * D * 2u;
      mbar_arrive_expect_tx(qbar, bytes);
      bulk_load(sQ, p.q + ((size_t)it.fork0 * p.hq + (size_t)it.kv_head * G) * D, bytes, qbar);
    }
    ++q_issued;
  };

  // prologue: the first item's Q and the first kSlots pages
  TcItem cnext{};  // consumer lookahead: the next non-empty item whose Q is still to be issued
  int cnk = next_nonempty(0, cnext);
  if (cnk < n_items) {
    issue_q(cnext);
    cnk = next_nonempty(cnk + 1, cnext);
  }
  for (int i = 0; i < kSlots && pk < n_items; ++i) issue();

  // per-lane parts of the ldmatrix addresses: K as the A operand of S^T (rows =
  // tokens, k = columns), V as the transposed A operand of O^T (rows = columns,
  // k = tokens), Q as the B operand of S^T
  const int mi = lane >> 3, mr = lane & 7;
  const int tk = (mi & 1) * 8 + mr, ck = mi >> 1;  // K: token, chunk offset within a k-step
  const int tv = (mi >> 1) * 8 + mr, cv = mi & 1;  // V: token, chunk offset within an m-tile
  const float sl2 = p.scale_log2;
  const uint32_t kZero = 0u;

  bool ok = true;
  TcItem it_next = n_items > 0 ? item(0) : TcItem{};
  for (int k = 0; ok && k < n_items; ++k) {
    const TcItem it = it_next;  // asked for at the previous item's start
    if (k + 1 < n_items) it_next = item(k + 1);
    const int np = npages(it);
    const int pslot = p.part_base[it.fork0] + it.part;
    if (np == 0) {
      // an item cut to nothing by the device lengths: an empty partial
      for (int x = lane; x < G * (p.dv / 4); x += 32) {
        const int r = x / (p.dv / 4), c4 = x % (p.dv / 4);
        reinterpret_cast<float4*>(p.part_o)[part_o_f4(pslot, it.kv_head * G + r, c4, p.hq, p.dv)] =
            make_float4(0.f, 0.f, 0.f, 0.f);
      }
      for (int r = lane; r < G; r += 32)
        p.part_lse[(size_t)pslot * p.hq + it.kv_head * G + r] = -INFINITY;
      continue;
    }
    // this item's query rows: into registers as B fragments (rows past G zero)
    if (!__all_sync(0xffffffffu, mbar_wait(qbar, q_used & 1, abort_flag, p.status))) {
      ok = false;
      break;
    }
    ++q_used;
    uint32_t qf[NT][KS][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
      const uint32_t rowa = sQ + (uint32_t)(8 * nt + mr) * (D * 2u);
#pragma unroll
      for (int kk = 0; kk < KS / 2; ++kk) {
        uint32_t r0, r1, r2, r3;
        ldmatrix_x4(rowa + (uint32_t)(4 * kk + mi) * 16u, r0, r1, r2, r3);
        const bool live = 8 * nt + g8 < G;
        qf[nt][2 * kk][0] = live ? r0 : kZero;
        qf[nt][2 * kk][1] = live ? r1 : kZero;
        qf[nt][2 * kk + 1][0] = live ? r2 : kZero;
        qf[nt][2 * kk + 1][1] = live ? r3 : kZero;
      }
    }
    // The next item's query rows go into the buffer only after the first page's
    // S^T MMAs have consumed these fragments: an ldmatrix result that no
    // instruction has used yet may still be in flight, and the bulk copy could
    // overwrite the buffer before it is read (seen as run-to-run differences in
    // the second n-tile's rows).
    bool next_q = cnk < n_items;

    float acc[NT][KS][4];
    float m[NT][2], l[NT][2];
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int mt = 0; mt < KS; ++mt)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[nt][mt][e] = 0.f;
      m[nt][0] = m[nt][1] = -INFINITY;
      l[nt][0] = l[nt][1] = 0.f;
    }

    for (int j = 0; j < np; ++j, ++used) {
      const int s = used % kSlots;
      if (!__all_sync(0xffffffffu, mbar_wait(full(s), (used / kSlots) & 1, abort_flag, p.status))) {
        ok = false;
        break;
      }
      const uint32_t sK = wslot + (uint32_t)s * L::kSlot, sV = sK + L::kBlk;
      const bool valid = sflag[s] != 0;
      const int rem = it.tok_end - (it.tok_begin + j * kPage);
      const int ntok = rem < kPage ? rem : kPage;
      const bool zeroed = !valid || ntok < kPage;
      if (zeroed) {
        // value rows this item does not own (past its end) or of an invalid
        // page: zero them, so that P = 0 never meets NaN or stale data
        const int first = valid ? ntok : 0;
        for (int x = lane; x < (kPage - first) * (D / 8); x += 32) {
          const int t = first + x / (D / 8), c = x % (D / 8);
          asm volatile("st.shared.v4.b32 [%0], {%1, %1, %1, %1};\n" ::"r"(sV + piece<D, TL>(t, c)),
                       "r"(0u)
                       : "memory");
        }
        __syncwarp();
      }
      // S^T = K Q^T (16 tokens x 8 heads per n-tile); with one n-tile the
      // k-steps run in two independent accumulator chains (even and odd k-steps,
      // added at the end), with two the n-tiles are the two chains
      float sc[NT][4], sc2[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        sc2[e] = 0.f;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) sc[nt][e] = 0.f;
      }
#pragma unroll
      for (int ks = 0; ks < KS; ++ks) {
        uint32_t a[4];
        ldmatrix_x4(sK + piece<D, TL>(tk, 2 * ks + ck), a[0], a[1], a[2], a[3]);
        if constexpr (NT == 1) {
          mma_bf16_16816((ks & 1) ? sc2 : sc[0], a, qf[0][ks][0], qf[0][ks][1]);
        } else {
#pragma unroll
          for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(sc[nt], a, qf[nt][ks][0], qf[nt][ks][1]);
        }
      }
      if constexpr (NT == 1) {
#pragma unroll
        for (int e = 0; e < 4; ++e) sc[0][e] += sc2[e];
      }
      if (next_q) {  // every Q fragment has been consumed by an MMA issued above
        __syncwarp();
        issue_q(cnext);
        cnk = next_nonempty(cnk + 1, cnext);
        next_q = false;
      }
      // tokens g8 and g8 + 8 of the page, heads 2*tig and 2*tig + 1 (+ 8 nt)
      const bool v0 = valid && g8 < ntok, v1 = valid && g8 + 8 < ntok;
      uint32_t pb0[NT], pb1[NT];
#pragma unroll
      for (int nt = 0; nt < NT; ++nt) {
        if (!v0) sc[nt][0] = sc[nt][1] = -INFINITY;
        if (!v1) sc[nt][2] = sc[nt][3] = -INFINITY;
        float alpha[2];
        bool grow = false;
#pragma unroll
        for (int r = 0; r < 2; ++r) {
          float mx = fmaxf(sc[nt][r], sc[nt][r + 2]);
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 4));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
          mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
          const float mt = mx * sl2;  // scale > 0
          alpha[r] = 1.f;
          if (mt > m[nt][r] + kRescale || (m[nt][r] == -INFINITY && mt != -INFINITY)) {
            alpha[r] = m[nt][r] == -INFINITY ? 0.f : fast_exp2(m[nt][r] - mt);
            l[nt][r] *= alpha[r];
            m[nt][r] = mt;
            grow = true;
          }
        }
        if (__any_sync(0xffffffffu, grow)) {
#pragma unroll
          for (int mt = 0; mt < KS; ++mt) {
            acc[nt][mt][0] *= alpha[0];
            acc[nt][mt][1] *= alpha[1];
            acc[nt][mt][2] *= alpha[0];
            acc[nt][mt][3] *= alpha[1];
          }
        }
        const float sub0 = m[nt][0] == -INFINITY ? 0.f : m[nt][0];
        const float sub1 = m[nt][1] == -INFINITY ? 0.f : m[nt][1];
        const float p00 = fast_exp2(fmaf(sc[nt][0], sl2, -sub0));
        const float p01 = fast_exp2(fmaf(sc[nt][1], sl2, -sub1));
        const float p10 = fast_exp2(fmaf(sc[nt][2], sl2, -sub0));
        const float p11 = fast_exp2(fmaf(sc[nt][3], sl2, -sub1));
        l[nt][0] += p00 + p10;
        l[nt][1] += p01 + p11;
        // P^T (tokens x heads) as the B operand: transpose each 8x8 block
        pb0[nt] = movmatrix_trans(pack_bf16x2(p00, p01));
        pb1[nt] = movmatrix_trans(pack_bf16x2(p10, p11));
      }
      // O^T += V^T P^T (16 columns x 8 heads per m-tile and n-tile)
#pragma unroll
      for (int mt = 0; mt < KS; ++mt) {
        uint32_t a[4];
        ldmatrix_x4_trans(sV + piece<D, TL>(tv, 2 * mt + cv), a[0], a[1], a[2], a[3]);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) mma_bf16_16816(acc[nt][mt], a, pb0[nt], pb1[nt]);
      }
      __syncwarp();  // every lane has read the slot
      if (pk < n_items) {
        if (zeroed) fence_proxy_async_smem();  // generic writes before the next async write
        issue();
      }
    }
    if (!ok) break;
    // ---- end of item: row sums over the eight lanes of a head, partial store
#pragma unroll
    for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
      for (int r = 0; r < 2; ++r) {
        float ls = l[nt][r];
        ls += __shfl_xor_sync(0xffffffffu, ls, 4);
        ls += __shfl_xor_sync(0xffffffffu, ls, 8);
        ls += __shfl_xor_sync(0xffffffffu, ls, 16);
        const int row = 8 * nt + 2 * tig + r;
        if (row < G) {
          const int head = it.kv_head * G + row;
          const float inv = ls > 0.f ? 1.f / ls : 0.f;
#pragma unroll
          for (int mt = 0; mt < KS; ++mt)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              const int c = 16 * mt + 8 * h + g8;
              p.part_o[part_o_f4(pslot, head, c >> 2, p.hq, p.dv) * 4 + (c & 3)] =
                  acc[nt][mt][2 * h + r] * inv;
            }
          if (g8 == 0)
            p.part_lse[(size_t)pslot * p.hq + head] =
                ls > 0.f ? (m[nt][r] + log2f(ls)) * kLn2 : -INFINITY;
        }
      }
    }
  }
  // never leave a copy in flight into this warp's shared memory
  if (lane == 0) {
    for (int u = used; u < issued; ++u) mbar_wait_drain(full(u % kSlots), (u / kSlots) & 1, p.status);
    if (q_issued > q_used) mbar_wait_drain(qbar, q_used & 1, p.status);
  }
  __syncwarp();
}

template <int D, bool TL, int NT>
__global__ void __launch_bounds__(kSuffixWarps * 32, kSuffixCtasPerSm)
    fork_suffix_kernel(const __grid_constant__ SfxParams p, const __grid_constant__ CUtensorMap tmk,
                       const __grid_constant__ CUtensorMap tmv) {
  // tmk / tmv: the key and value pools with one whole (page, head) block per box
  // (token-major pools); the tiled layout reads the pools with bulk copies.
  using L = Layout<D, NT>;
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t sb = (raw + 1023u) & ~1023u;  // 128B-swizzled boxes: 1024-byte aligned
  unsigned char* gb = smem_raw + (sb - raw);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gb + L::kAbort);
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    // alone, the merge (a programmatic dependent) may be launched now: it waits
    // for this grid's completion before it reads any partial (with the prefix
    // kernel behind this grid, the trigger comes after the wait instead)
    if (!p.late_trigger) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  }
  __syncthreads();
  suffix_warp<D, TL, NT>(p, &tmk, &tmv, sb, gb, threadIdx.x >> 5, abort_flag);
}

template <int D, bool TL, int NT>
cudaError_t launch_k(const SfxParams& p, const CUtensorMap& mk, const CUtensorMap& mv, int grid,
                     cudaStream_t stream) {
  constexpr int smem = (int)(Layout<D, NT>::kBytes + 1024u);
  static_assert(smem <= 232448, "suffix stage shared memory exceeds 227 KB");
  static_assert(kSuffixCtasPerSm * (smem + 1024) <= 233472, "suffix-stage CTAs per SM");
  auto kern = fork_suffix_kernel<D, TL, NT>;
  static thread_local int configured = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured != dev) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kSuffixWarps * 32);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, p, mk, mv);
}

template <bool TL, int NT>
cudaError_t launch_dim(const SfxParams& p, const CUtensorMap& mk, const CUtensorMap& mv, int grid,
                       int dqk, cudaStream_t stream) {
  if (dqk == 128) return launch_k<128, TL, NT>(p, mk, mv, grid, stream);
  if (dqk == 64) return launch_k<64, TL, NT>(p, mk, mv, grid, stream);
  return cudaErrorInvalidValue;
}

}  // namespace

bool suffix_stage_supported(int dqk, int dv, bool latent, int page_size, int G) {
  return fork_tc_supported(dqk, dv, latent, page_size, G) && G <= kSuffixMaxG;
}

cudaError_t launch_suffix_stage(const SfxParams& p, const void* k_pages, const void* v_pages,
                                int grid, int dqk, bool tiled, cudaStream_t stream) {
  if (grid == 0) return cudaSuccess;
  CUtensorMap mk, mv;
  if (tiled) {
    memset(&mk, 0, sizeof(mk));
    memset(&mv, 0, sizeof(mv));
    if (reinterpret_cast<uintptr_t>(k_pages) % 16 || reinterpret_cast<uintptr_t>(v_pages) % 16)
      return cudaErrorInvalidValue;
    return p.G <= 8 ? launch_dim<true, 1>(p, mk, mv, grid, dqk, stream)
                    : launch_dim<true, 2>(p, mk, mv, grid, dqk, stream);
  }
  // the maps depend only on the pools' addresses and shapes (cached per thread)
  struct MapKey {
    const void* k;
    const void* v;
    int dqk, hkv, num_pages;
    bool operator==(const MapKey& o) const {
      return k == o.k && v == o.v && dqk == o.dqk && hkv == o.hkv && num_pages == o.num_pages;
    }
  };
  static thread_local MapKey cached{nullptr, nullptr, 0, 0, 0};
  static thread_local CUtensorMap cached_k, cached_v;
  const MapKey key{k_pages, v_pages, dqk, p.hkv, p.num_pages};
  if (!(key == cached)) {
    cached = MapKey{nullptr, nullptr, 0, 0, 0};
    if (!fork_tc_block_map(&cached_k, k_pages, dqk, p.hkv, p.num_pages) ||
        !fork_tc_block_map(&cached_v, v_pages, dqk, p.hkv, p.num_pages))
      return cudaErrorInvalidValue;
    cached = key;
  }
  mk = cached_k;
  mv = cached_v;
  return p.G <= 8 ? launch_dim<false, 1>(p, mk, mv, grid, dqk, stream)
                  : launch_dim<false, 2>(p, mk, mv, grid, dqk, stream);
}

}  // namespace specgen
