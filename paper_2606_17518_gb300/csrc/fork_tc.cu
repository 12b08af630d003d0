// Fork-decode attention on the 5th-generation tensor cores (tcgen05 + TMA).
//
// One persistent CTA per SM walks its list of TcItems.  An item is either a
// chunk of a trace's shared prefix (the query rows of all the trace's forks for
// one kv head, gathered into one M = nforks * G <= 128 row tile, so each prefix
// page is fetched from HBM once for every fork) or a chunk of one fork's
// private suffix (M = G rows).  Each item writes a partial (O / l, LSE) per row.
//
// Per 128-token tile t (8 pages of 16 tokens), with t counted across items:
//   warp 0 (TMA)     K_t pages -> K ring, byte-counted on k_full[t%ST]
//   warp 10 (TMA)    V_t pages -> V ring, byte-counted on v_full[t%ST]
//   warp 1 (MMA)     S_t = Q K_t^T -> TMEM S[t%2]   (M=128, N=16*pages, K=D);
//                    the K stage is released as soon as S_t has finished
//                    O  += P_t V_t -> TMEM O         (M=128, N=D,  K=16*pages);
//                    then the V stage is released
//   warps 2-9        two groups of 4 warps on alternate tiles, one thread per
//                    row (= TMEM lane): the 128 scores of the tile in
//                    registers, masked where needed, running max kept in log2
//                    units; P_t = exp2(s*scale*log2e - m) back to TMEM as bf16;
//                    the TMEM output is rescaled only when a row's max grows
//                    by more than 2^8 (lazy rescaling), otherwise P may exceed 1.
// S is double-buffered in TMEM so S_{t+1} runs while tile t is in softmax.
// Separate K and V rings keep more bytes in flight: a K stage is held only
// until its score MMA is done, a V stage until its PV product is done.  Every
// copy issue costs the issuing warp a roughly fixed time, so the copies are as
// large as the layouts allow and all copies of a tile leave in one warp
// instruction.
//
// Two KV pool layouts.  Rows: every (page, head) block is 16 token rows of D
// contiguous elements.  K is gathered with one 64-column TMA box per panel and
// page into 128B-swizzled panels of the whole tile (the score MMA needs every
// panel's tokens at one stride); V with one box per page that holds all its
// panels ([page][panel][16 rows], which the PV MMA reads page by page).
// Tiled: every block is stored as the tensor cores' 8-token x 8-element core
// matrices, ((t/8)*(D/8) + d/8)*64 + (t%8)*8 + d%8, so one contiguous bulk copy
// (D*32 bytes) lands it in the layout the MMA reads directly (no swizzle): K is
// then K-major with 128-byte steps along d and D*16-byte steps per 8 tokens, V
// is MN-major with the same two strides.
// Warps whose 32 rows are all padding skip the softmax work.  Tokens past the
// item, past the sequence or on an invalid page are masked to -inf, and value
// rows past the sequence inside its last page are zeroed in shared memory
// before the PV product, so nothing stored there (even NaN) reaches the output.
// Head dim 64 uses 64-token tiles (four pages) with six stages per ring.  A
// causal instantiation serves prefill plans, whose suffix items hold several
// query rows of one fork, each masked at its own length.  The kernel is a
// programmatic dependent of the previous kernel of the stream: its prologue
// (and an L2 prefetch of its first tiles) runs before it waits for that kernel.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>
#include <string.h>

#include "common.cuh"
#include "fork_tc.h"
#include "plan.h"
#include "tc_common.cuh"

namespace specgen {

namespace {

using namespace tc;

constexpr int kPB = 16;                      // page size (tokens)
constexpr int kWG = 2;                       // softmax warpgroups (alternating tiles)
constexpr int kVWarp = 2 + 4 * kWG;          // the V copy warp, after the softmax groups
constexpr int kThreads = 32 * (kVWarp + 1);  // warp 0 K copies, warp 1 MMA, 4 warps per softmax group, V copies
constexpr uint32_t kTmemCols = 512;          // S[0] [0,TT) S[1] [TT,2TT) O[0] [256,..) O[1] [384,..)
constexpr uint32_t kTmemO = 256;
constexpr float kRescaleLog2 = 8.0f;         // lazy-rescale threshold (factor 256)
constexpr int kMaxStages = 6;
// tokens per pipeline tile: 8 pages for D = 128 (three stages per ring); 4 pages
// for D = 64 (six stages), where the shorter tiles fill the pipeline sooner
constexpr int kTile128 = 128;
constexpr int kTile64 = 64;

// Shared memory of one CTA: Q (128 rows x D, non-swizzled 8x8 core matrices:
// LBO 128 B along d, SBO D*16 B per 8 rows), a ring of `ST` K stages and one of
// `ST` V stages of TT tokens each (rows layout: 128B-swizzled 64-column panels,
// K as [panel][TT rows], V as [page][panel][16 rows]; tiled layout: the pool's
// own core-matrix blocks, page after page), barriers, the per-stage valid-page
// masks, the second group's (m, l) and the CTA's first items.
constexpr int kItemCache = 14;

template <int D, int TT, int ST, bool TL>
struct Smem {
  static constexpr int kPanels = D / 64;
  static constexpr uint32_t kQ = 128u * D * 2u;
  static constexpr uint32_t kRowsTile = TT * 128u;        // one 64-column panel of TT rows
  static constexpr uint32_t kKV = kPanels * kRowsTile;    // one K or V tile (TT x D bf16)
  static constexpr uint32_t kBlk = kPB * D * 2u;          // one (page, head) block
  static constexpr uint32_t kOffK = kQ;
  static constexpr uint32_t kOffV = kOffK + ST * kKV;
  static constexpr uint32_t kOffBar = kOffV + ST * kKV;
  static constexpr uint32_t kOffML = kOffBar + 384;        // 128 x (m, l) of the second group
  static constexpr uint32_t kOffItems = kOffML + 128 * 8;
  static constexpr uint32_t kAlign = TL ? 128u : 1024u;    // 128B-swizzled tiles: 1024-B aligned
  static constexpr uint32_t kBytes = kOffItems + kItemCache * (uint32_t)sizeof(TcItem) + kAlign;
};

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}
struct ItemView {
  const int32_t* table;
  int ntiles, page0, M;
};

template <int TT>
__device__ __forceinline__ ItemView view(const TcParams& p, const TcItem& it) {
  ItemView v;
  const int32_t* bt = it.table_kind == 0 ? p.prefix_bt : p.suffix_bt;
  v.table = bt + (it.table_off >= 0 ? it.table_off
                                    : (it.table_kind == 0 ? p.prefix_bt_off : p.suffix_bt_off)[it.seq]);
  v.ntiles = (it.tok_end - it.tok_begin + TT - 1) / TT;
  v.page0 = it.tok_begin / kPB;
  v.M = it.nforks * p.G;
  return v;
}

template <int TT>
__device__ __forceinline__ int tile_tokens(const TcItem& it, int j) {
  const int n = it.tok_end - (it.tok_begin + j * TT);
  return n < TT ? n : TT;
}

// Item k of this CTA: the first kItemCache come from shared memory (already
// cut to the current suffix lengths), the rest are read and cut here.
__device__ __forceinline__ TcItem get_item(const TcItem* cache, const TcParams& p, int it_begin,
                                           int k) {
  return k < kItemCache ? cache[k] : clamp_item(p.items[it_begin + k], p.suffix_lens);
}

// Page ids pb + lane of an item (lane-strided batch of 32); 0 past the item.
__device__ __forceinline__ int page_batch(const TcParams& p, const TcItem& it, int pb, int lane) {
  const int npages = (it.tok_end - it.tok_begin + kPB - 1) / kPB;
  if (pb + lane >= npages) return 0;
  const int32_t* bt = it.table_kind == 0 ? p.prefix_bt : p.suffix_bt;
  const int off = it.table_off >= 0
                      ? it.table_off
                      : (it.table_kind == 0 ? p.prefix_bt_off : p.suffix_bt_off)[it.seq];
  return bt[off + it.tok_begin / kPB + pb + lane];
}

// CAUSAL: the plan has causal suffix items (prefill chunks), each row masked at
// its own length; decode plans take the kernel without that per-row limit.
template <int D, int TT, int ST, bool TL, bool CAUSAL>
__global__ void __launch_bounds__(kThreads, 1)
    fork_tc_kernel(const __grid_constant__ TcParams p, const __grid_constant__ CUtensorMap tmk,
                   const __grid_constant__ CUtensorMap tmv) {
  // tmk: 4-D map, one 64-column panel of one (page, head) block per box;
  // tmv: the same for D = 64, else a 5-D map whose box is a whole block.
  using L = Smem<D, TT, ST, TL>;
  constexpr int kPagesPerTile = TT / kPB;
  static_assert(32 % kPagesPerTile == 0, "a batch of 32 page ids holds whole tiles");
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + L::kAlign - 1u) & ~(L::kAlign - 1u);
  unsigned char* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base;
  const uint32_t bar0 = base + L::kOffBar;
  // barrier block: k_full[4] k_empty[4] v_full[4] v_empty[4] s_full[2] p_full[2]
  // o_full[2] q_ready mma_done ml_ready q_free merge_done ml_back, then the TMEM
  // address, the abort flag, the per-stage valid-page masks (K copy warp -> MMA)
  // and the per-score-buffer masks (MMA -> softmax)
  auto k_full = [&](int s) { return bar0 + 8u * s; };
  auto k_empty = [&](int s) { return bar0 + 8u * (kMaxStages + s); };
  auto v_full = [&](int s) { return bar0 + 8u * (2 * kMaxStages + s); };
  auto v_empty = [&](int s) { return bar0 + 8u * (3 * kMaxStages + s); };
  constexpr int kB = 4 * kMaxStages;
  auto s_full = [&](int b) { return bar0 + 8u * (kB + b); };
  auto p_full = [&](int b) { return bar0 + 8u * (kB + 2 + b); };
  auto o_full = [&](int b) { return bar0 + 8u * (kB + 4 + b); };
  const uint32_t q_ready = bar0 + 8u * (kB + 6);     // Q of the next item stored
  const uint32_t mma_done = bar0 + 8u * (kB + 7);
  const uint32_t ml_ready = bar0 + 8u * (kB + 8);    // group 1's (m, l) written
  const uint32_t q_free = bar0 + 8u * (kB + 9);      // an item's last S finished
  const uint32_t merge_done = bar0 + 8u * (kB + 10); // group 1 read its O halves
  const uint32_t ml_back = bar0 + 8u * (kB + 11);    // group 0's weights written
  constexpr int kMisc = 8 * (kB + 12);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + L::kOffBar + kMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + L::kOffBar + kMisc + 4);
  volatile uint32_t* smask = reinterpret_cast<volatile uint32_t*>(gbase + L::kOffBar + kMisc + 8);
  volatile uint32_t* smask_s =
      reinterpret_cast<volatile uint32_t*>(gbase + L::kOffBar + kMisc + 8 + 4 * kMaxStages);
  // K tiles issued so far: the V copy warp never runs ahead of it, so that at
  // the start the copies leave in the order the tiles are consumed
  volatile int* k_issued =
      reinterpret_cast<volatile int*>(gbase + L::kOffBar + kMisc + 16 + 4 * kMaxStages);
  static_assert(kMisc + 20 + 4 * kMaxStages <= 384, "barrier block");
  float2* ml1 = reinterpret_cast<float2*>(gbase + L::kOffML);  // second group's (m, l) per row
  TcItem* items = reinterpret_cast<TcItem*>(gbase + L::kOffItems);
  auto sK = [&](int s) { return base + L::kOffK + s * L::kKV; };
  auto sV = [&](int s) { return base + L::kOffV + s * L::kKV; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int it_begin = p.cta_offsets[blockIdx.x], it_end = p.cta_offsets[blockIdx.x + 1];
  const int n_items = it_end - it_begin;
  // dependents (the merge) released at the start: they wait for this grid's
  // completion before they read anything it writes
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  // the CTA's first items, one per lane (40-byte records): the plan is written
  // by a host copy, never by a kernel, so it is read before the wait below
  constexpr int kWords = sizeof(TcItem) / 4;
  const int n_cached = n_items < kItemCache ? n_items : kItemCache;
  if (warp == 0) {
    const int32_t* src = reinterpret_cast<const int32_t*>(p.items + it_begin);
    int32_t* dst = reinterpret_cast<int32_t*>(items);
    for (int x = lane; x < n_cached * kWords; x += 32) dst[x] = src[x];
  }
  if (threadIdx.x == 32) {
    for (int i = 0; i < ST; ++i) {
      mbar_init(k_full(i), 1);
      mbar_init(k_empty(i), 1);
      mbar_init(v_full(i), 1);
      mbar_init(v_empty(i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      // the score MMAs' commit, and the MMA thread once it has stored the tile's mask
      mbar_init(s_full(i), 2);
      mbar_init(p_full(i), 128);
      mbar_init(o_full(i), 1);
    }
    mbar_init(q_ready, 128);
    mbar_init(mma_done, 1);
    mbar_init(ml_ready, 128);
    mbar_init(q_free, 1);
    mbar_init(merge_done, 128);
    mbar_init(ml_back, 128);
    *abort_flag = 0;
    *k_issued = 0;
    mbar_init_fence();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  // Launched as a programmatic dependent, this grid may start while the previous
  // kernel of the stream is still running: everything above touches only this
  // CTA's own resources and the plan.  The inputs (device lengths, block tables,
  // Q, K/V, possibly written by that kernel) and the partial buffers (possibly
  // still read by it) are used only after this wait.  (Behind the suffix stage
  // there is no wait here: see wait_at_end.)  Before it, the two copy
  // warps only ask L2 for the first item's first two tiles: the page ids they
  // read here serve as prefetch addresses (in-range ids only) and nothing else,
  // so a table the previous kernel rewrites costs bandwidth, never correctness.
  // Only plans with host-resolved table offsets take part: then every read
  // here is of the plan or of table entries at positions the plan was built
  // for.  Behind the suffix stage there is no wait to overlap, and the copies
  // themselves follow at once: no prefetch (measured 0.5 us faster).
  if (!p.wait_at_end && (warp == 0 || warp == kVWarp) && n_items > 0) {
    const TcItem it = p.items[it_begin];  // from the plan itself, not the cache
    const int npages = (it.tok_end - it.tok_begin + kPB - 1) / kPB;
    if (it.table_off >= 0 && lane < 2 * kPagesPerTile && lane < npages) {
      const int page = page_batch(p, it, 0, lane);
      if (page >= 0 && page < p.num_pages) {
        const __nv_bfloat16* blk = (warp == 0 ? p.k_pages : p.v_pages) +
                                   ((size_t)page * p.hkv + it.kv_head) * (kPB * D);
        asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;\n" ::"l"(blk), "r"(L::kBlk)
                     : "memory");
      }
    }
  }
  if (!p.wait_at_end) asm volatile("griddepcontrol.wait;\n" ::: "memory");
  if (warp == 0) {
    __syncwarp();
    for (int k = lane; k < n_cached; k += 32) items[k] = clamp_item(items[k], p.suffix_lens);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 || warp == kVWarp) {
    // ------------------------------------------------------------ copy warps
    // Warp 0 copies K tiles, warp kVWarp V tiles, each through its own ring.
    // Both fetch page ids 32 at a time (one coalesced load, one batch ahead, and
    // the next item's first batch one item ahead).  Lane 0 waits for a free
    // stage (the K warp also publishes the tile's valid-page mask); then one
    // lane per copy issues all copies of the tile in one instruction.
    const bool is_v = warp == kVWarp;
    const int pg = lane % kPagesPerTile;  // the page this lane copies
    int t = 0;                            // tiles issued so far (across items)
    bool ok = true;
    int first_next = n_items > 0 ? page_batch(p, get_item(items, p, it_begin, 0), 0, lane) : 0;
    for (int k = 0; ok && k < n_items; ++k) {
      const TcItem it = get_item(items, p, it_begin, k);
      const int npages = (it.tok_end - it.tok_begin + kPB - 1) / kPB;
      int cur = first_next;
      first_next = k + 1 < n_items ? page_batch(p, get_item(items, p, it_begin, k + 1), 0, lane) : 0;
      for (int pb = 0; ok && pb < npages; pb += 32) {
        const int nxt = page_batch(p, it, pb + 32, lane);
        const int batch_pages = npages - pb < 32 ? npages - pb : 32;
        for (int tp = 0; tp < batch_pages; tp += kPagesPerTile, ++t) {
          const int j = (pb + tp) / kPagesPerTile;  // tile index within the item
          const int np = (tile_tokens<TT>(it, j) + kPB - 1) / kPB;
          const int page = __shfl_sync(0xffffffffu, cur, tp + pg);
          const bool page_ok = pg < np && page >= 0 && page < p.num_pages;
          const uint32_t valid = __ballot_sync(0xffffffffu, page_ok && lane < kPagesPerTile);
          const uint32_t bad = ((1u << np) - 1u) & ~valid;
          const int s = t % ST;
          const uint32_t fbar = is_v ? v_full(s) : k_full(s);
          if (lane == 0) {
            ok = mbar_wait(is_v ? v_empty(s) : k_empty(s), ((t / ST) & 1) ^ 1, abort_flag,
                           p.status);
            if (ok && !is_v) smask[s] = valid;
            if (bad && !is_v) atomicOr(p.status, kStatusIndex);
            if (ok && is_v && *k_issued <= t) {  // bounded wait for K_t to be issued
              const unsigned long long w0 = globaltimer();
              while (*k_issued <= t) {
                if (*abort_flag) {
                  ok = false;
                  break;
                }
                if (globaltimer() - w0 > kWaitLimitNs) {
                  atomicOr(p.status, kStatusTimeout);
                  *abort_flag = 1;
                  ok = false;
                  break;
                }
              }
            }
          }
          ok = __shfl_sync(0xffffffffu, ok, 0);
          if (!ok) break;
          if constexpr (TL) {
            // one bulk copy per page; an invalid page's value block is zeroed
            // here instead (its scores are masked)
            if (is_v && bad) {
              for (int q = 0; q < np; ++q)
                if ((bad >> q) & 1u)
                  for (uint32_t x = lane * 16u; x < L::kBlk; x += 32u * 16u)
                    st_shared_v4(sV(s) + q * L::kBlk + x, 0u, 0u, 0u, 0u);
              fence_proxy_async_smem();
              __syncwarp();
            }
            if (lane == 0) mbar_arrive_expect_tx(fbar, (uint32_t)__popc(valid) * L::kBlk);
            __syncwarp();
            if (lane < kPagesPerTile && ((valid >> pg) & 1u)) {
              const __nv_bfloat16* src = (is_v ? p.v_pages : p.k_pages) +
                                         ((size_t)page * p.hkv + it.kv_head) * (kPB * D);
              bulk_load((is_v ? sV(s) : sK(s)) + pg * L::kBlk, src, L::kBlk, fbar);
            }
          } else {
            // TMA zero-fills out-of-range pages, so every box counts
            if (lane == 0) mbar_arrive_expect_tx(fbar, (uint32_t)np * L::kBlk);
            __syncwarp();
            if (is_v) {
              if (lane < kPagesPerTile && pg < np) {
                if constexpr (L::kPanels > 1)
                  tma_load_5d(sV(s) + pg * L::kBlk, &tmv, 0, 0, 0, it.kv_head, page, fbar);
                else
                  tma_load_4d(sV(s) + pg * L::kBlk, &tmv, 0, 0, it.kv_head, page, fbar);
              }
            } else {
              const int pn = lane / kPagesPerTile;  // this lane's 64-column panel
              if (pn < L::kPanels && pg < np)
                tma_load_4d(sK(s) + pn * L::kRowsTile + pg * (kPB * 128u), &tmk, pn * 64, 0,
                            it.kv_head, page, fbar);
            }
          }
          __syncwarp();
          if (!is_v && lane == 0) *k_issued = t + 1;
          // with an item's last V tile (about a ring of tiles before the item's
          // end is consumed) ask L2 for the next item's Q rows, which the
          // softmax loads on the path to that item's first score MMA; asked at
          // the item's start they could be evicted by the KV streamed meanwhile
          if (!CAUSAL && is_v && pb + tp + kPagesPerTile >= npages && k + 1 < n_items) {
            const TcItem nx = get_item(items, p, it_begin, k + 1);
            for (int r = lane; r < nx.nforks * p.G; r += 32) {
              const char* qrow = reinterpret_cast<const char*>(
                  p.q + ((size_t)(nx.fork0 + r / p.G) * p.hq + nx.kv_head * p.G + r % p.G) * D);
#pragma unroll
              for (int c = 0; c < D * 2; c += 128)
                asm volatile("prefetch.global.L2 [%0];\n" ::"l"(qrow + c));
            }
          }
        }
        cur = nxt;
      }
    }
    // never leave a copy in flight into this CTA's shared memory
    if (lane == 0)
      for (int u = t - ST < 0 ? 0 : t - ST; u < t; ++u)
        mbar_wait_drain(is_v ? v_full(u % ST) : k_full(u % ST), (u / ST) & 1, p.status);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      // descriptors are built once; every MMA only adds a constant offset
      // (in 16-byte units) to the start-address field
      const uint64_t dq = smem_desc_interleave(sQ, 128, D * 16);
      // tiled: K-major K (LBO = next 8 columns, SBO = next 8 tokens); MN-major V
      // (LBO = next 8 tokens, SBO = next 8 columns)
      const uint64_t dk0 = TL ? smem_desc_interleave(sK(0), 128, D * 16)
                              : smem_desc_sw128(sK(0), 16, 1024);
      // rows: V panels of one page are 16 rows x 128 B apart (LBO), 8-token
      // groups 1024 B apart (SBO)
      const uint64_t dv0 = TL ? smem_desc_interleave(sV(0), D * 16, 128)
                              : smem_desc_sw128(sV(0), kPB * 128u, 1024);
      // byte step of V per page (one 16-token k-step): one block in both layouts
      constexpr uint32_t kVPage = L::kBlk;
      constexpr uint64_t kStageDesc = L::kKV >> 4;
      constexpr uint32_t idesc_pv = idesc_bf16(128, D, true);
      // Ready-first issue: PV_v goes out as soon as its P is ready; S_u goes
      // out when its K tile has landed, its score buffer is free (PV_{u-2}
      // issued, so in-order execution has consumed P_{u-2}) and, for an item's
      // first tile, its Q is in shared memory.  After an item's last S, q_free
      // tells the Q loader that the buffer may be overwritten.  s_*: the next
      // S to issue, v_*: the next PV (item index, tile within item, global tile).
      int s_k = 0, s_j = 0, s_u = 0, v_k = 0, v_j = 0, v_u = 0;
      TcItem s_it = n_items > 0 ? get_item(items, p, it_begin, 0) : TcItem{};
      TcItem v_it = s_it;
      int s_nt = view<TT>(p, s_it).ntiles, v_nt = s_nt;
      bool q_ok = false;
      bool ok = true;
      unsigned long long t0 = 0;
      // items cut to nothing by the current suffix lengths have no tiles: the
      // PV cursor steps over them, the S cursor still takes their Q phase and
      // releases the Q buffer (q_free) so the item sequence stays in step
      while (v_k < n_items && v_nt == 0 && ++v_k < n_items) {
        v_it = get_item(items, p, it_begin, v_k);
        v_nt = view<TT>(p, v_it).ntiles;
      }
      while (ok && (v_k < n_items || s_k < n_items)) {
        bool did = false;
        if (s_k < n_items && s_nt == 0 && mbar_test_wait(q_ready, s_k & 1)) {
          mma_commit(q_free);  // an empty item: its Q phase taken, the buffer released
          q_ok = false;
          if (++s_k < n_items) {
            s_it = get_item(items, p, it_begin, s_k);
            s_nt = view<TT>(p, s_it).ntiles;
          }
          did = true;
        } else if (v_u < s_u && mbar_test_wait(p_full(v_u & 1), (v_u >> 1) & 1) &&
                   mbar_test_wait(v_full(v_u % ST), (v_u / ST) & 1)) {
          tc_fence_after();
          const int b = v_u & 1, s = v_u % ST;
          const int np = (tile_tokens<TT>(v_it, v_j) + kPB - 1) / kPB;
          const uint64_t dv = dv0 + (uint64_t)s * kStageDesc;
          const uint32_t o_tmem = tmem + kTmemO + (uint32_t)(v_j & 1) * 128u;
          const uint32_t p_tmem = tmem + (uint32_t)b * TT;
          const uint32_t acc0 = v_j >= 2 ? 1u : 0u;
          if (np == kPagesPerTile) {
#pragma unroll
            for (int kk = 0; kk < kPagesPerTile; ++kk)  // one page (16 tokens) per k-step
              mma_bf16_ts(o_tmem, p_tmem + kk * 8u, dv + (uint64_t)((kk * kVPage) >> 4),
                          idesc_pv, (acc0 | (kk > 0)) ? 1u : 0u);
          } else {
            for (int kk = 0; kk < np; ++kk)
              mma_bf16_ts(o_tmem, p_tmem + kk * 8u, dv + (uint64_t)((kk * kVPage) >> 4),
                          idesc_pv, (acc0 | (kk > 0)) ? 1u : 0u);
          }
          mma_commit(o_full(b));
          mma_commit(v_empty(s));
          ++v_u;
          if (++v_j == v_nt) {
            v_j = 0;
            do {
              if (++v_k < n_items) {
                v_it = get_item(items, p, it_begin, v_k);
                v_nt = view<TT>(p, v_it).ntiles;
              }
            } while (v_k < n_items && v_nt == 0);
          }
          did = true;
        } else if (s_k < n_items && s_nt > 0 && s_u - v_u < 2) {
          if (!q_ok && mbar_test_wait(q_ready, s_k & 1)) q_ok = true;
          if (q_ok && mbar_test_wait(k_full(s_u % ST), (s_u / ST) & 1)) {
            tc_fence_after();
            const int b = s_u & 1, s = s_u % ST;
            // the tile's page mask for the softmax (its previous reader, two
            // tiles back, is done: PV_{u-2} has been issued)
            smask_s[b] = smask[s];
            mbar_arrive(s_full(b));
            const int np = (tile_tokens<TT>(s_it, s_j) + kPB - 1) / kPB;
            const uint32_t idesc = idesc_bf16(128, np * kPB, false);
            const uint64_t dk = dk0 + (uint64_t)s * kStageDesc;
            const uint32_t d_s = tmem + (uint32_t)b * TT;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint64_t ko =
                  (TL ? kk * 256u : (kk >> 2) * L::kRowsTile + (kk & 3) * 32u) >> 4;
              mma_bf16(d_s, dq + (uint64_t)((kk * 256u) >> 4), dk + ko, idesc, kk > 0 ? 1u : 0u);
            }
            mma_commit(s_full(b));
            mma_commit(k_empty(s));
            ++s_u;
            if (++s_j == s_nt) {
              mma_commit(q_free);
              s_j = 0;
              q_ok = false;
              if (++s_k < n_items) {
                s_it = get_item(items, p, it_begin, s_k);
                s_nt = view<TT>(p, s_it).ntiles;
              }
            }
            did = true;
          }
        }
        if (did) {
          t0 = 0;
        } else if (t0 == 0) {
          t0 = globaltimer();
        } else if (*abort_flag) {
          ok = false;
        } else if (globaltimer() - t0 > kWaitLimitNs) {
          atomicOr(p.status, kStatusTimeout);
          *abort_flag = 1;
          ok = false;
        }
      }
      // every MMA issued by this thread has finished before TMEM is released
      mma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, p.status);
    }
  } else {
    // ------------------------------------------------------------ softmax groups
    // Group g (warps 2+4g .. 5+4g) takes the tiles j = g, g+2, ... of every item
    // with its own running max/sum and its own TMEM output O[g].  Group 1 also
    // stages Q: it loads the next item's rows (asked of L2 by the V copy warp)
    // into registers after its last tile and stores them once the MMA reports
    // the current item's last S finished.  At the end of every item the groups combine their halves,
    // each writing half of the value columns.
    const int grp = (warp - 2) >> 2;
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int gtid = (threadIdx.x - 64) & 127;  // 0..127 within the group
    const uint32_t lane_addr = (uint32_t)(q4 * 32) << 16;
    const uint32_t s_base = tmem + lane_addr;
    const uint32_t o_mine = tmem + lane_addr + kTmemO + (uint32_t)grp * 128u;
    const float sl2 = p.scale_log2;
    int t = 0;
    bool ok = true;
    uint4 qr[D / 8];  // group 1: the next item's Q row (zero for padding rows)
    // (re)defines qr on every path, so it is never live across a tile loop
    auto load_q = [&](bool want, const TcItem& it) {
      const bool rok = want && row < it.nforks * p.G;
      const int fl = row / p.G, gi = row % p.G;
      const uint4* src = reinterpret_cast<const uint4*>(
          p.q + ((size_t)(it.fork0 + (rok ? fl : 0)) * p.hq + (rok ? it.kv_head * p.G + gi : 0)) *
                    D);
#pragma unroll
      for (int c = 0; c < D / 8; ++c) qr[c] = rok ? __ldg(src + c) : make_uint4(0, 0, 0, 0);
    };
    load_q(grp == 1 && n_items > 0, get_item(items, p, it_begin, 0));
    auto store_q = [&]() {
#pragma unroll
      for (int c = 0; c < D / 8; ++c)
        st_shared_v4(sQ + ((row >> 3) * (D / 8) + c) * 128u + (row & 7) * 16u, qr[c].x, qr[c].y,
                     qr[c].z, qr[c].w);
      fence_proxy_async_smem();
      mbar_arrive(q_ready);
    };

    for (int k = 0; ok && k < n_items; ++k) {
      const TcItem it = get_item(items, p, it_begin, k);
      const int ntiles = (it.tok_end - it.tok_begin + TT - 1) / TT;
      const int M = it.nforks * p.G;
      const bool warp_live = q4 * 32 < M;  // some real row in this warp
      const bool row_ok = row < M;
      const int fl = row / p.G, gi = row % p.G;
      const int head = it.kv_head * p.G + gi;
      // this row's partial slot base, fetched now and used at the item's end
      const int pbase = p.part_base[it.fork0 + (row_ok ? fl : 0)];
      // causal items: tokens past this row's own length (relative to the item)
      // are masked; everything else sees the whole item
      const int row_end = CAUSAL && it.row_limit0 > 0 ? it.row_limit0 + fl - it.tok_begin
                                                      : 0x7fffffff;

      // group 1 stores Q of the first item here, of every later item at the end
      // of the previous one (as soon as that item's last S has finished)
      if (grp == 1 && k == 0) store_q();
      // prefill items are short: there group 1 asks L2 for the next item's Q
      // rows itself, at this item's start
      if constexpr (CAUSAL) {
        if (grp == 1 && k + 1 < n_items) {
          const TcItem nx = get_item(items, p, it_begin, k + 1);
          if (row < nx.nforks * p.G) {
            const char* qrow = reinterpret_cast<const char*>(
                p.q + ((size_t)(nx.fork0 + row / p.G) * p.hq + nx.kv_head * p.G + row % p.G) * D);
#pragma unroll
            for (int c = 0; c < D * 2; c += 128)
              asm volatile("prefetch.global.L2 [%0];\n" ::"l"(qrow + c));
          }
        }
      }

      float m = -INFINITY, l = 0.f;  // this group's running max (log2 units) and sum
      for (int j = grp; j < ntiles; j += 2) {
        const int u = t + j, b = u & 1, s = u % ST;
        const bool w = mbar_wait(s_full(b), (u >> 1) & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) {
          ok = false;
          break;
        }
        tc_fence_after();
        // S_u done implies every earlier MMA is done, in particular PV_{u-2}
        // (this group's previous tile): consume that o_full phase now
        if (j >= 2) mbar_wait(o_full(b), ((u - 2) >> 1) & 1, abort_flag, p.status);
        const int nt = tile_tokens<TT>(it, j);
        const int np = (nt + kPB - 1) / kPB;
        if (warp_live) {
          const uint32_t pv = smask_s[b];  // valid pages of this tile
          float sc[TT];
          {
            uint32_t r[TT / 32][32];
            const uint32_t sa = s_base + (uint32_t)b * TT;
#pragma unroll
            for (int c = 0; c < TT / 32; ++c) tmem_ld32(sa + c * 32u, r[c]);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < TT / 32; ++c)
#pragma unroll
              for (int i = 0; i < 32; ++i) sc[c * 32 + i] = __uint_as_float(r[c][i]);
          }
          // tokens this row may see in the tile: the item's, and for a causal
          // item (prefill chunk) those before the row's own limit
          int lim = nt;
          if constexpr (CAUSAL) lim = max(0, min(nt, row_end - j * TT));
          const bool full_tile = lim == TT && pv == (1u << kPagesPerTile) - 1u;
          if (!full_tile) {
#pragma unroll
            for (int i = 0; i < TT; ++i)
              if (!(i < lim && ((pv >> (i / kPB)) & 1u))) sc[i] = -INFINITY;
          }
          float mx0 = sc[0], mx1 = sc[1], mx2 = sc[2], mx3 = sc[3];
#pragma unroll
          for (int i = 4; i < TT; i += 4) {
            mx0 = fmaxf(mx0, sc[i]);
            mx1 = fmaxf(mx1, sc[i + 1]);
            mx2 = fmaxf(mx2, sc[i + 2]);
            mx3 = fmaxf(mx3, sc[i + 3]);
          }
          const float m_tile = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * sl2;  // scale > 0
          bool rescale = false;
          float alpha = 1.f;
          if (m_tile > m + kRescaleLog2 || (m == -INFINITY && m_tile != -INFINITY)) {
            alpha = m == -INFINITY ? 0.f : fast_exp2(m - m_tile);
            rescale = m != -INFINITY;
            l *= alpha;
            m = m_tile;
          }
          const float sub = m == -INFINITY ? 0.f : m;
          float ps0 = 0.f, ps1 = 0.f;
          // P_u (bf16 pairs) over the first TT/2 columns of S_u's TMEM buffer
#pragma unroll
          for (int c = 0; c < TT / 64; ++c) {
            uint32_t pk[32];
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              const float p0 = fast_exp2(fmaf(sc[c * 64 + 2 * i], sl2, -sub));
              const float p1 = fast_exp2(fmaf(sc[c * 64 + 2 * i + 1], sl2, -sub));
              ps0 += p0;
              ps1 += p1;
              pk[i] = pack_bf16x2(p0, p1);
            }
            tmem_st32(s_base + (uint32_t)b * TT + c * 32u, pk);
          }
          l += ps0 + ps1;
          // a row whose max grew: rescale this group's output (its previous PV is done)
          if (j >= 2 && __any_sync(0xffffffffu, rescale)) {
            const float a = rescale ? alpha : 1.f;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
              uint32_t r[32];
              tmem_ld32(o_mine + c * 32u, r);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * a);
              tmem_st32(o_mine + c * 32u, r);
            }
          }
          tmem_wait_st();
        }
        // value rows past the sequence inside its last page: zero them before PV
        // (once the V tile has landed; its stage cannot be refilled before this
        // group's p_full, so the phase is still the current one)
        if (j == ntiles - 1 && (nt % kPB) != 0) {
          if (!mbar_wait(v_full(s), (u / ST) & 1, abort_flag, p.status)) ok = false;
          const int pg = np - 1, first = nt % kPB;
          const int units = (kPB - first) * L::kPanels * 8;  // 16-byte pieces
          for (int x = gtid; x < units; x += 128) {
            const int rr = first + x / (L::kPanels * 8);
            const int rem = x % (L::kPanels * 8);  // 8-column chunk of the row
            const int tt = pg * kPB + rr;
            const uint32_t off = TL ? ((tt >> 3) * (D / 8) + rem) * 128u + (tt & 7) * 16u
                                    : pg * L::kBlk + (rem >> 3) * (kPB * 128u) + rr * 128u +
                                          ((rem & 7) << 4);
            st_shared_v4(sV(s) + off, 0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
        }
        tc_fence_before();
        mbar_arrive(p_full(b));
      }
      if (!ok) break;
      // ---- end of item: both groups wait for their last PV, exchange (m, l)
      // through ml1 in two steps (group 1's (m, l) to group 0, the two final
      // weights back), and each writes half of the value columns
      const int last = grp + ((ntiles - 1 - grp) >> 1) * 2;  // this group's last tile (if any)
      const bool has = grp < ntiles;
      load_q(grp == 1 && k + 1 < n_items, get_item(items, p, it_begin, k + 1 < n_items ? k + 1 : k));
      if (has) {
        const int u = t + last, b = u & 1;
        const bool w = mbar_wait(o_full(b), (u >> 1) & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) ok = false;
        tc_fence_after();
      }
      float a0 = 0.f, a1 = 0.f;  // O = a0 O[0] + a1 O[1] (weights already divided by the sum)
      if (grp == 1) {
        ml1[row] = make_float2(has ? m : -INFINITY, has ? l : 0.f);
        tc_fence_before();  // O[1] complete before group 0 reads it
        mbar_arrive(ml_ready);
        if (k + 1 < n_items) {
          // the next item's Q, once this item's last S has finished with the buffer
          const bool wq = mbar_wait(q_free, k & 1, abort_flag, p.status);
          if (__any_sync(0xffffffffu, !wq)) ok = false;
          if (ok) store_q();
        }
        const bool w = mbar_wait(ml_back, k & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) ok = false;
        tc_fence_after();
        const float2 wg = ml1[row];
        a0 = wg.x;
        a1 = wg.y;
      } else {
        const bool w = mbar_wait(ml_ready, k & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) ok = false;
        tc_fence_after();
        const float2 o1 = ml1[row];
        const float mm = fmaxf(m, o1.x);
        const float w0 = m == -INFINITY ? 0.f : fast_exp2(m - mm);
        const float w1 = o1.x == -INFINITY ? 0.f : fast_exp2(o1.x - mm);
        const float lsum = l * w0 + o1.y * w1;
        const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
        a0 = w0 * inv;
        a1 = w1 * inv;
        ml1[row] = make_float2(a0, a1);
        tc_fence_before();  // O[0] complete before group 1 reads it
        mbar_arrive(ml_back);
        if (ok && row_ok)
          p.part_lse[(size_t)(pbase + it.part) * p.hq + head] =
              mm == -INFINITY ? -INFINITY : (mm + log2f(lsum)) * kLn2;
      }
      if (ok && warp_live) {
        // one 32-column chunk of O[0] and O[1] per TMEM round trip (group 1
        // holds the next item's Q row in registers meanwhile)
        const uint32_t o0 = tmem + lane_addr + kTmemO + (uint32_t)grp * (D / 2), o1 = o0 + 128u;
        float4* dst = reinterpret_cast<float4*>(p.part_o) +
                      part_o_f4((size_t)pbase + it.part, head, grp * (D / 8), p.hq, p.dv);
#pragma unroll
        for (int c = 0; c < D / 64; ++c) {
          uint32_t r0[32], r1[32];
          tmem_ld32(o0 + c * 32u, r0);
          tmem_ld32(o1 + c * 32u, r1);
          tmem_wait_ld();
          if (row_ok) {
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              float x[4];
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                // an unused output buffer (weight 0) may hold anything: never multiply it
                const float v0 = a0 == 0.f ? 0.f : __uint_as_float(r0[i + e]) * a0;
                const float v1 = a1 == 0.f ? 0.f : __uint_as_float(r1[i + e]) * a1;
                x[e] = v0 + v1;
              }
              dst[(size_t)(c * 8 + i / 4) * p.hq] = make_float4(x[0], x[1], x[2], x[3]);
            }
          }
        }
      }
      tc_fence_before();
      if (grp == 1) {
        mbar_arrive(merge_done);
      } else {
        // group 1 has read its half of O[0] before the next item's first PV
        // (issued after this group's next p_full) overwrites it
        const bool w = mbar_wait(merge_done, k & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) ok = false;
        tc_fence_after();
      }
      if (__any_sync(0xffffffffu, !ok)) ok = false;
      t += ntiles;
    }
  }

  tc_fence_before();
  // non-aligned CTA barrier: it counts every thread, so the lanes of a warp may
  // arrive apart (lanes 1-31 of the MMA warp come here at once, its lane 0 and
  // the copy lanes only after their drains).  An aligned __syncthreads() there
  // could complete before the softmax warps' last TMEM loads.
  asm volatile("barrier.sync 0;\n" ::: "memory");
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
  // behind the suffix stage: complete only after it has (see wait_at_end)
  if (p.wait_at_end) asm volatile("griddepcontrol.wait;\n" ::: "memory");
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(ptr);
  }
  return fn;
}

// Paged pool [num_pages][hkv][page][D] bf16 as a 4-D tensor (D, page, hkv, pages);
// one box = 64 columns x one page of one head, 128-byte swizzled.
bool make_pool_map(CUtensorMap* map, const void* pool, int D, int page, int hkv, int num_pages) {
  EncodeTiledFn enc = encode_fn();
  if (!enc || !pool || num_pages < 1) return false;
  const cuuint64_t dims[4] = {(cuuint64_t)D, (cuuint64_t)page, (cuuint64_t)hkv,
                              (cuuint64_t)num_pages};
  const cuuint64_t strides[3] = {(cuuint64_t)D * 2, (cuuint64_t)page * D * 2,
                                 (cuuint64_t)hkv * page * D * 2};
  const cuuint32_t box[4] = {64, (cuuint32_t)page, 1, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(pool), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Value map of the rows layout: (64 columns, page rows, D/64 panels, hkv, pages)
// with the panel stride (128 B) inside the row stride, so one box is one whole
// (page, head) block, landing in shared memory as [panel][page rows], 128-byte
// swizzled.  D = 64 has one panel: the key map serves.
bool make_pool_map_v(CUtensorMap* map, const void* pool, int D, int page, int hkv, int num_pages) {
  if (D == 64) return make_pool_map(map, pool, D, page, hkv, num_pages);
  EncodeTiledFn enc = encode_fn();
  if (!enc || !pool || num_pages < 1) return false;
  const cuuint64_t dims[5] = {64, (cuuint64_t)page, (cuuint64_t)(D / 64), (cuuint64_t)hkv,
                              (cuuint64_t)num_pages};
  const cuuint64_t strides[4] = {(cuuint64_t)D * 2, 128, (cuuint64_t)page * D * 2,
                                 (cuuint64_t)hkv * page * D * 2};
  const cuuint32_t box[5] = {64, (cuuint32_t)page, (cuuint32_t)(D / 64), 1, 1};
  const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  return enc(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(pool), dims, strides, box,
             estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D, int TT, int ST, bool TL, bool CAUSAL>
cudaError_t launch_d(const TcParams& p, const CUtensorMap& mk, const CUtensorMap& mv, int grid,
                     cudaStream_t stream) {
  constexpr int smem = (int)Smem<D, TT, ST, TL>::kBytes;
  static_assert(smem <= 232448, "fork_tc kernel shared memory exceeds 227 KB");
  static_assert(ST <= kMaxStages && (TT == 64 || TT == 128), "unsupported pipeline shape");
  static_assert(kTmemO + 128u * kWG <= kTmemCols && 2 * TT <= (int)kTmemO, "TMEM layout");
  auto kern = fork_tc_kernel<D, TT, ST, TL, CAUSAL>;
  static thread_local int configured = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured != dev) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(kern, cudaFuncAttributePreferredSharedMemoryCarveout,
                             (int)cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  // programmatic dependent launch: the grid may start while the previous kernel
  // of the stream finishes (the kernel waits for it before touching its inputs)
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, p, mk, mv);
}

}  // namespace

bool fork_tc_block_map(CUtensorMap* map, const void* pool, int D, int hkv, int num_pages) {
  return make_pool_map_v(map, pool, D, kPB, hkv, num_pages);
}

bool fork_tc_supported(int dqk, int dv, bool latent, int page_size, int G) {
  return !latent && dqk == dv && (dqk == 64 || dqk == 128) && page_size == kPB && G <= 128;
}

int fork_tc_tile_tokens(int dqk) { return dqk == 64 ? kTile64 : kTile128; }
int fork_tc_page_size() { return kPB; }

template <bool CAUSAL>
static cudaError_t launch_layout(const TcParams& p, const void* k_pages, const void* v_pages, int grid,
                          int dqk, bool tiled, cudaStream_t stream) {
  if (grid == 0) return cudaSuccess;
  CUtensorMap mk, mv;
  if (tiled) {
    // bulk copies read the pools directly; the tensor maps stay unused
    memset(&mk, 0, sizeof(mk));
    memset(&mv, 0, sizeof(mv));
    if (reinterpret_cast<uintptr_t>(k_pages) % 16 || reinterpret_cast<uintptr_t>(v_pages) % 16)
      return cudaErrorInvalidValue;
    if (dqk == 128) return launch_d<128, kTile128, 3, true, CAUSAL>(p, mk, mv, grid, stream);
    if (dqk == 64) return launch_d<64, kTile64, 6, true, CAUSAL>(p, mk, mv, grid, stream);
    return cudaErrorInvalidValue;
  }
  // the maps depend only on the pools' addresses and shapes: encode them again
  // only when those change (a decode loop launches over the same pools)
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
    if (!make_pool_map(&cached_k, k_pages, dqk, kPB, p.hkv, p.num_pages) ||
        !make_pool_map_v(&cached_v, v_pages, dqk, kPB, p.hkv, p.num_pages))
      return cudaErrorInvalidValue;
    cached = key;
  }
  mk = cached_k;
  mv = cached_v;
  if (dqk == 128) return launch_d<128, kTile128, 3, false, CAUSAL>(p, mk, mv, grid, stream);
  if (dqk == 64) return launch_d<64, kTile64, 6, false, CAUSAL>(p, mk, mv, grid, stream);
  return cudaErrorInvalidValue;
}

cudaError_t launch_fork_tc(const TcParams& p, const void* k_pages, const void* v_pages, int grid,
                           int dqk, bool tiled, bool causal, cudaStream_t stream) {
  return causal ? launch_layout<true>(p, k_pages, v_pages, grid, dqk, tiled, stream)
                : launch_layout<false>(p, k_pages, v_pages, grid, dqk, tiled, stream);
}

}  // namespace specgen
