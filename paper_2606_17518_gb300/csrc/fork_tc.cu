// Fork-decode attention on the 5th-generation tensor cores (tcgen05 + TMA).
//
// One persistent CTA per SM walks its list of TcItems.  An item is either a
// chunk of a trace's shared prefix (the query rows of all the trace's forks for
// one kv head, gathered into one M = nforks * G <= 128 row tile, so each prefix
// page is fetched from HBM once for every fork) or a chunk of one fork's
// private suffix (M = G rows).  Each item writes a partial (O / l, LSE) per row.
//
// Per 128-token tile t (8 pages of 16 tokens), with t counted across items:
//   warp 0 (TMA)     K_t, V_t pages -> 2-stage shared-memory ring (two 64-column
//                    boxes per page, 128B swizzle), byte-counted on full[t%2]
//   warp 1 (MMA)     S_t = Q K_t^T -> TMEM S[t%2]   (M=128, N=16*pages, K=D)
//                    O  += P_t V_t -> TMEM O         (M=128, N=D,  K=16*pages)
//   warps 2-5        one thread per row (= TMEM lane): the 128 scores of the
//                    tile in registers, masked where needed, running max kept
//                    in log2 units; P_t = exp2(s*scale*log2e - m) to shared
//                    memory as bf16 (128B-swizzled, K-major); the TMEM output
//                    is rescaled only when a row's max grows by more than
//                    2^8 (lazy rescaling), otherwise P may exceed 1.
// S is double-buffered in TMEM so S_{t+1} runs while tile t is in softmax.
//
// Two KV pool layouts.  Rows: every (page, head) block is 16 token rows of D
// contiguous elements; the TMA engine gathers it with 64-column boxes into
// 128B-swizzled panels.  Tiled: every block is stored as the tensor cores'
// 8-token x 8-element core matrices, ((t/8)*(D/8) + d/8)*64 + (t%8)*8 + d%8,
// so one contiguous bulk copy (D*32 bytes) lands it in the layout the MMA
// reads directly (no swizzle): K is then K-major with 128-byte steps along d
// and D*16-byte steps per 8 tokens, V is MN-major with the same two strides.
// Warps whose 32 rows are all padding skip the softmax work.  Tokens past the
// item, past the sequence or on an invalid page are masked to -inf, and value
// rows past the sequence inside its last page are zeroed in shared memory
// before the PV product, so nothing stored there (even NaN) reaches the output.
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
constexpr int kThreads = 64 + 128 * kWG;     // warp 0 TMA, warp 1 MMA, 4 warps per softmax group
constexpr uint32_t kTmemCols = 512;          // S[0] [0,TT) S[1] [TT,2TT) O[0] [256,..) O[1] [384,..)
constexpr uint32_t kTmemO = 256;
constexpr float kRescaleLog2 = 8.0f;         // lazy-rescale threshold (factor 256)
constexpr int kMaxStages = 8;
constexpr int kTile = 128;                   // tokens per pipeline tile (8 pages)

// Shared memory of one CTA: Q (128 rows x D) and a ring of `ST` (K, V) stages of
// TT tokens.  Every operand tile is made of 64-column panels (128-byte rows,
// 128B-swizzled), 1024-byte aligned.  P lives in tensor memory.
template <int D, int TT, int ST>
struct Smem {
  static constexpr int kPanels = D / 64;
  static constexpr uint32_t kQPanel = 128 * 128u;         // 128 rows x 128 B
  static constexpr uint32_t kQ = kPanels * kQPanel;
  static constexpr uint32_t kRowsTile = TT * 128u;        // one 64-column panel of TT rows
  static constexpr uint32_t kKV = kPanels * kRowsTile;    // one K or V tile
  static constexpr uint32_t kStage = 2 * kKV;
  static constexpr uint32_t kOffKV = kQ;
  static constexpr uint32_t kOffBar = kOffKV + ST * kStage;
  static constexpr uint32_t kOffML = kOffBar + 256;        // 128 x (m, l) of the second group
  static constexpr uint32_t kBytes = kOffML + 128 * 8 + 1024;
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

template <int D, int TT, int ST, bool TL>
__global__ void __launch_bounds__(kThreads, 1)
    fork_tc_kernel(const __grid_constant__ TcParams p, const __grid_constant__ CUtensorMap tmk,
                   const __grid_constant__ CUtensorMap tmv) {
  using L = Smem<D, TT, ST>;
  constexpr int kPagesPerTile = TT / kPB;
  static_assert(32 % kPagesPerTile == 0, "a batch of 32 page ids holds whole tiles");
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;  // 128B-swizzled tiles: 1024-B aligned
  unsigned char* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base;
  const uint32_t bar0 = base + L::kOffBar;
  // barrier block: full[ST] empty[ST] s_full[2] p_full[2] o_full[2] q_ready mma_done
  auto full = [&](int s) { return bar0 + 8u * s; };
  auto empty = [&](int s) { return bar0 + 8u * (kMaxStages + s); };
  auto s_full = [&](int b) { return bar0 + 8u * (2 * kMaxStages + b); };
  auto p_full = [&](int b) { return bar0 + 8u * (2 * kMaxStages + 2 + b); };
  auto o_full = [&](int b) { return bar0 + 8u * (2 * kMaxStages + 4 + b); };
  const uint32_t q_ready = bar0 + 8u * (2 * kMaxStages + 6);
  const uint32_t mma_done = bar0 + 8u * (2 * kMaxStages + 7);
  const uint32_t ml_ready = bar0 + 8u * (2 * kMaxStages + 8);  // group 1's (m, l) written
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + L::kOffBar + 8 * (2 * kMaxStages + 9));
  volatile int* abort_flag =
      reinterpret_cast<volatile int*>(gbase + L::kOffBar + 8 * (2 * kMaxStages + 9) + 4);
  float2* ml1 = reinterpret_cast<float2*>(gbase + L::kOffML);  // second group's (m, l) per row
  auto sK = [&](int s) { return base + L::kOffKV + s * L::kStage; };
  auto sV = [&](int s) { return base + L::kOffKV + s * L::kStage + L::kKV; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int it_begin = p.cta_offsets[blockIdx.x], it_end = p.cta_offsets[blockIdx.x + 1];
  // let the merge grid (a programmatic dependent) get launched early; it waits
  // for this grid's completion before it reads anything
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");

  if (threadIdx.x == 0) {
    for (int i = 0; i < ST; ++i) {
      mbar_init(full(i), 1);
      mbar_init(empty(i), 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(s_full(i), 1);
      mbar_init(p_full(i), 128);
      mbar_init(o_full(i), 1);
    }
    mbar_init(q_ready, 128);
    mbar_init(mma_done, 1);
    mbar_init(ml_ready, 128);
    *abort_flag = 0;
    mbar_init_fence();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    // The whole warp fetches page ids 32 at a time (one coalesced load, one
    // batch ahead).  Lane 0 waits for a free stage; then lanes 0..2*D/64-1
    // each issue one box of every page (K and V, one 64-column panel each).
    constexpr int kIssuers = TL ? 2 * kPagesPerTile : 2 * L::kPanels;
    const bool issuer = lane < kIssuers;
    const bool is_v = lane >= L::kPanels;
    const int pn = is_v ? lane - L::kPanels : lane;
    const void* tmap = is_v ? static_cast<const void*>(&tmv) : static_cast<const void*>(&tmk);
    int t = 0;  // tiles issued so far (across items)
    bool ok = true;
    for (int ii = it_begin; ok && ii < it_end; ++ii) {
      const TcItem it = p.items[ii];
      const ItemView v = view<TT>(p, it);
      const int npages = (it.tok_end - it.tok_begin + kPB - 1) / kPB;
      int cur = lane < npages ? v.table[v.page0 + lane] : 0;
      for (int pb = 0; ok && pb < npages; pb += 32) {
        const int nxt = pb + 32 + lane < npages ? v.table[v.page0 + pb + 32 + lane] : 0;
        const int batch_pages = npages - pb < 32 ? npages - pb : 32;
        for (int tp = 0; tp < batch_pages; tp += kPagesPerTile, ++t) {
          const int j = (pb + tp) / kPagesPerTile;  // tile index within the item
          const int np = (tile_tokens<TT>(it, j) + kPB - 1) / kPB;
          int pages[kPagesPerTile];
#pragma unroll
          for (int pg = 0; pg < kPagesPerTile; ++pg)
            pages[pg] = __shfl_sync(0xffffffffu, cur, tp + pg);
          const int s = t % ST;
          if constexpr (TL) {
            // one bulk copy per (page, K or V); an invalid page is reported and
            // its value block zeroed here instead (its scores are masked)
            constexpr uint32_t kBlk = kPB * D * 2u;
            uint32_t bad = 0;
#pragma unroll
            for (int pg = 0; pg < kPagesPerTile; ++pg)
              if (pg < np && (pages[pg] < 0 || pages[pg] >= p.num_pages)) bad |= 1u << pg;
            if (lane == 0) ok = mbar_wait(empty(s), ((t / ST) & 1) ^ 1, abort_flag, p.status);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            if (bad) {
              for (int pg = 0; pg < np; ++pg)
                if ((bad >> pg) & 1u)
                  for (uint32_t x = lane * 16u; x < kBlk; x += 32u * 16u)
                    st_shared_v4(sV(s) + pg * kBlk + x, 0u, 0u, 0u, 0u);
              fence_proxy_async_smem();
              __syncwarp();
              if (lane == 0) atomicOr(p.status, kStatusIndex);
            }
            if (lane == 0)
              mbar_arrive_expect_tx(full(s), (uint32_t)(np - __popc(bad)) * 2u * kBlk);
            __syncwarp();
            const int pg = lane % kPagesPerTile;
            if (issuer && pg < np && !((bad >> pg) & 1u)) {
              const bool v_side = lane >= kPagesPerTile;
              const __nv_bfloat16* src = (v_side ? p.v_pages : p.k_pages) +
                                         ((size_t)pages[pg] * p.hkv + it.kv_head) * (kPB * D);
              bulk_load((v_side ? sV(s) : sK(s)) + pg * kBlk, src, kBlk, full(s));
            }
            continue;
          }
          if (lane == 0) {
            ok = mbar_wait(empty(s), ((t / ST) & 1) ^ 1, abort_flag, p.status);
            if (ok) mbar_arrive_expect_tx(full(s), (uint32_t)np * 2u * L::kPanels * (kPB * 128u));
          }
          ok = __shfl_sync(0xffffffffu, ok, 0);
          if (!ok) break;
          if (issuer) {
            const uint32_t dst = (is_v ? sV(s) : sK(s)) + pn * L::kRowsTile;
#pragma unroll
            for (int pg = 0; pg < kPagesPerTile; ++pg) {
              if (pg >= np) break;
              tma_load_4d(dst + pg * (kPB * 128u), tmap, pn * 64, 0, it.kv_head, pages[pg], full(s));
            }
          }
          if (lane == 0)
            for (int pg = 0; pg < np; ++pg)
              if (pages[pg] < 0 || pages[pg] >= p.num_pages)
                atomicOr(p.status, kStatusIndex);  // TMA zero-fills out-of-range pages
        }
        cur = nxt;
      }
    }
    // never leave a copy in flight into this CTA's shared memory
    if (lane == 0)
      for (int u = t - ST < 0 ? 0 : t - ST; u < t; ++u)
        mbar_wait_drain(full(u % ST), (u / ST) & 1, p.status);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      // descriptors are built once; every MMA only adds a constant offset
      // (in 16-byte units) to the start-address field
      const uint64_t dq = smem_desc_sw128(sQ, 16, 1024);
      // tiled: K-major K (LBO = next 8 columns, SBO = next 8 tokens); MN-major V
      // (LBO = next 8 tokens, SBO = next 8 columns)
      const uint64_t dk0 = TL ? smem_desc_interleave(sK(0), 128, D * 16)
                              : smem_desc_sw128(sK(0), 16, 1024);
      const uint64_t dv0 = TL ? smem_desc_interleave(sV(0), D * 16, 128)
                              : smem_desc_sw128(sV(0), L::kRowsTile, 1024);
      // byte step of V per page (one 16-token k-step) and of K per 16 columns
      constexpr uint32_t kVPage = TL ? kPB * D * 2u : kPB * 128u;
      constexpr uint64_t kStageDesc = L::kStage >> 4;
      constexpr uint32_t idesc_pv = idesc_bf16(128, D, true);
      // Ready-first issue: PV_v goes out as soon as its P is ready; S_u goes
      // out when its K tile has landed, its score buffer is free (PV_{u-2}
      // issued, so in-order execution has consumed P_{u-2}) and, for an item's
      // first tile, its Q is in shared memory.  s_*: the next S to issue,
      // v_*: the next PV to issue (item cursor, tile within item, global tile).
      int s_ii = it_begin, s_j = 0, s_u = 0, v_ii = it_begin, v_j = 0, v_u = 0;
      TcItem s_it = s_ii < it_end ? p.items[s_ii] : TcItem{};
      TcItem v_it = s_it;
      int s_nt = view<TT>(p, s_it).ntiles, v_nt = s_nt;
      bool q_ok = false;
      bool ok = true;
      unsigned long long t0 = 0;
      while (ok && v_ii < it_end) {
        bool did = false;
        if (v_u < s_u && mbar_try_wait(p_full(v_u & 1), (v_u >> 1) & 1)) {
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
          mma_commit(empty(s));
          ++v_u;
          if (++v_j == v_nt) {
            v_j = 0;
            if (++v_ii < it_end) {
              v_it = p.items[v_ii];
              v_nt = view<TT>(p, v_it).ntiles;
            }
          }
          did = true;
        } else if (s_ii < it_end && s_u - v_u < 2) {
          if (!q_ok && mbar_try_wait(q_ready, (s_ii - it_begin) & 1)) q_ok = true;
          if (q_ok && mbar_try_wait(full(s_u % ST), (s_u / ST) & 1)) {
            tc_fence_after();
            const int b = s_u & 1, s = s_u % ST;
            const int np = (tile_tokens<TT>(s_it, s_j) + kPB - 1) / kPB;
            const uint32_t idesc = idesc_bf16(128, np * kPB, false);
            const uint64_t dk = dk0 + (uint64_t)s * kStageDesc;
            const uint32_t d_s = tmem + (uint32_t)b * TT;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              const uint64_t qo = ((kk >> 2) * L::kQPanel + (kk & 3) * 32u) >> 4;
              const uint64_t ko =
                  (TL ? kk * 256u : (kk >> 2) * L::kRowsTile + (kk & 3) * 32u) >> 4;
              mma_bf16(d_s, dq + qo, dk + ko, idesc, kk > 0 ? 1u : 0u);
            }
            mma_commit(s_full(b));
            ++s_u;
            if (++s_j == s_nt) {
              s_j = 0;
              q_ok = false;
              if (++s_ii < it_end) {
                s_it = p.items[s_ii];
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
    // with its own running max/sum and its own TMEM output O[g]; group 0 merges
    // the two halves at the end of the item.
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

    for (int ii = it_begin; ok && ii < it_end; ++ii) {
      const TcItem it = p.items[ii];
      const ItemView v = view<TT>(p, it);
      const bool warp_live = q4 * 32 < v.M;  // some real row in this warp
      const bool row_ok = row < v.M;
      const int fl = row / p.G, gi = row % p.G;
      const int head = it.kv_head * p.G + gi;

      if (grp == 0) {
        // Q row -> shared memory, 128B-swizzled K-major panels; padding rows are zero
        const uint4* src = reinterpret_cast<const uint4*>(
            p.q + ((size_t)(it.fork0 + (row_ok ? fl : 0)) * p.hq + (row_ok ? head : 0)) * D);
        if (warp_live) {
#pragma unroll
          for (int c = 0; c < D / 8; ++c) {
            const uint4 q = row_ok ? __ldg(src + c) : make_uint4(0, 0, 0, 0);
            st_shared_v4(sQ + (c >> 3) * L::kQPanel + row * 128u + (((c & 7) ^ (row & 7)) << 4),
                         q.x, q.y, q.z, q.w);
          }
        }
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(q_ready);
      } else {
        // group 1 starts an item only after group 0 has finished merging the
        // previous one (group 0 arrives on q_ready after that merge)
        const bool w = mbar_wait(q_ready, (ii - it_begin) & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) {
          ok = false;
          break;
        }
      }

      float m = -INFINITY, l = 0.f;  // this group's running max (log2 units) and sum
      // page ids: 32 per coalesced warp load (lane i holds page pb + i), one batch ahead
      const int npages_item = (it.tok_end - it.tok_begin + kPB - 1) / kPB;
      auto load_batch = [&](int pb) {
        return pb + lane < npages_item ? v.table[v.page0 + pb + lane] : 0;
      };
      int cur_batch = 0;
      int cur_pages = load_batch(0), nxt_pages = load_batch(32);
      for (int j = grp; j < v.ntiles; j += 2) {
        const int u = t + j, b = u & 1;
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
        const int batch = (j * kPagesPerTile) >> 5;
        while (cur_batch < batch) {  // at most one step per visited tile
          cur_pages = nxt_pages;
          ++cur_batch;
          nxt_pages = load_batch(cur_batch * 32 + 32);
        }
        const int tp0 = (j * kPagesPerTile) & 31;
        if (warp_live) {
          uint32_t pv = 0;  // valid pages of this tile
#pragma unroll
          for (int pg = 0; pg < kPagesPerTile; ++pg) {
            const int page = __shfl_sync(0xffffffffu, cur_pages, (tp0 + pg) & 31);
            if (pg < np && page >= 0 && page < p.num_pages) pv |= 1u << pg;
          }
          float s[TT];
          {
            uint32_t r[TT / 32][32];
            const uint32_t sa = s_base + (uint32_t)b * TT;
#pragma unroll
            for (int c = 0; c < TT / 32; ++c) tmem_ld32(sa + c * 32u, r[c]);
            tmem_wait_ld();
#pragma unroll
            for (int c = 0; c < TT / 32; ++c)
#pragma unroll
              for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(r[c][i]);
          }
          const bool full_tile = nt == TT && pv == (1u << kPagesPerTile) - 1u;
          if (!full_tile) {
#pragma unroll
            for (int i = 0; i < TT; ++i)
              if (!(i < nt && ((pv >> (i / kPB)) & 1u))) s[i] = -INFINITY;
          }
          float mx0 = s[0], mx1 = s[1], mx2 = s[2], mx3 = s[3];
#pragma unroll
          for (int i = 4; i < TT; i += 4) {
            mx0 = fmaxf(mx0, s[i]);
            mx1 = fmaxf(mx1, s[i + 1]);
            mx2 = fmaxf(mx2, s[i + 2]);
            mx3 = fmaxf(mx3, s[i + 3]);
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
              const float p0 = fast_exp2(fmaf(s[c * 64 + 2 * i], sl2, -sub));
              const float p1 = fast_exp2(fmaf(s[c * 64 + 2 * i + 1], sl2, -sub));
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
        if (j == v.ntiles - 1 && (nt % kPB) != 0) {
          const int pg = np - 1, first = nt % kPB;
          const int units = (kPB - first) * L::kPanels * 8;  // 16-byte pieces
          for (int x = gtid; x < units; x += 128) {
            const int rr = first + x / (L::kPanels * 8);
            const int rem = x % (L::kPanels * 8);  // 8-column chunk of the row
            const int tt = pg * kPB + rr;
            const uint32_t off = TL ? ((tt >> 3) * (D / 8) + rem) * 128u + (tt & 7) * 16u
                                    : (rem >> 3) * L::kRowsTile + tt * 128u + ((rem & 7) << 4);
            st_shared_v4(sV(u % ST) + off, 0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
        }
        tc_fence_before();
        mbar_arrive(p_full(b));
      }
      if (!ok) break;
      // ---- end of item: wait for this group's last PV, then merge the groups
      const int last = grp + ((v.ntiles - 1 - grp) >> 1) * 2;  // this group's last tile (if any)
      const bool has = grp < v.ntiles;
      if (has) {
        const int u = t + last, b = u & 1;
        const bool w = mbar_wait(o_full(b), (u >> 1) & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) ok = false;
        tc_fence_after();
      }
      if (grp == 1) {
        ml1[row] = make_float2(has ? m : -INFINITY, has ? l : 0.f);
        tc_fence_before();
        mbar_arrive(ml_ready);
      } else {
        const bool w = mbar_wait(ml_ready, (ii - it_begin) & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) ok = false;
        tc_fence_after();
        if (ok && warp_live) {
          const float2 o1 = ml1[row];
          const float mm = fmaxf(m, o1.x);
          const float w0 = m == -INFINITY ? 0.f : fast_exp2(m - mm);
          const float w1 = o1.x == -INFINITY ? 0.f : fast_exp2(o1.x - mm);
          const float lsum = l * w0 + o1.y * w1;
          const float inv = lsum > 0.f ? 1.f / lsum : 0.f;
          const int fork = it.fork0 + (row_ok ? fl : 0);
          const size_t prow_out = (size_t)(p.part_base[fork] + it.part) * p.hq + head;
          float4* dst = reinterpret_cast<float4*>(p.part_o + prow_out * p.dv);
          const uint32_t o0 = tmem + lane_addr + kTmemO, o1a = o0 + 128u;
#pragma unroll
          for (int c = 0; c < D / 32; ++c) {
            uint32_t r0[32], r1[32];
            tmem_ld32(o0 + c * 32u, r0);
            tmem_ld32(o1a + c * 32u, r1);
            tmem_wait_ld();
            if (row_ok) {
#pragma unroll
              for (int i = 0; i < 32; i += 4) {
                float x[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                  // an unused output buffer (weight 0) may hold anything: never multiply it
                  const float a0 = w0 == 0.f ? 0.f : __uint_as_float(r0[i + e]) * w0;
                  const float a1 = w1 == 0.f ? 0.f : __uint_as_float(r1[i + e]) * w1;
                  x[e] = (a0 + a1) * inv;
                }
                dst[c * 8 + i / 4] = make_float4(x[0], x[1], x[2], x[3]);
              }
            }
          }
          if (row_ok)
            p.part_lse[prow_out] = mm == -INFINITY ? -INFINITY : (mm + log2f(lsum)) * kLn2;
        }
        tc_fence_before();
      }
      if (__any_sync(0xffffffffu, !ok)) ok = false;
      t += v.ntiles;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
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

template <int D, int TT, int ST, bool TL>
cudaError_t launch_d(const TcParams& p, const CUtensorMap& mk, const CUtensorMap& mv, int grid,
                     cudaStream_t stream) {
  constexpr int smem = (int)Smem<D, TT, ST>::kBytes;
  static_assert(smem <= 232448, "fork_tc kernel shared memory exceeds 227 KB");
  static_assert(ST <= kMaxStages && (TT == 64 || TT == 128), "unsupported pipeline shape");
  static_assert(kTmemO + 128u * kWG <= kTmemCols && 2 * TT <= (int)kTmemO, "TMEM layout");
  auto kern = fork_tc_kernel<D, TT, ST, TL>;
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
  kern<<<grid, kThreads, smem, stream>>>(p, mk, mv);
  return cudaGetLastError();
}

}  // namespace

bool fork_tc_supported(int dqk, int dv, bool latent, int page_size, int G) {
  return !latent && dqk == dv && (dqk == 64 || dqk == 128) && page_size == kPB && G <= 128;
}

int fork_tc_tile_tokens() { return kTile; }
int fork_tc_page_size() { return kPB; }

cudaError_t launch_fork_tc(const TcParams& p, const void* k_pages, const void* v_pages, int grid,
                           int dqk, bool tiled, cudaStream_t stream) {
  if (grid == 0) return cudaSuccess;
  CUtensorMap mk, mv;
  if (tiled) {
    // bulk copies read the pools directly; the tensor maps stay unused
    memset(&mk, 0, sizeof(mk));
    memset(&mv, 0, sizeof(mv));
    if (reinterpret_cast<uintptr_t>(k_pages) % 16 || reinterpret_cast<uintptr_t>(v_pages) % 16)
      return cudaErrorInvalidValue;
    if (dqk == 128) return launch_d<128, kTile, 3, true>(p, mk, mv, grid, stream);
    if (dqk == 64) return launch_d<64, kTile, 4, true>(p, mk, mv, grid, stream);
    return cudaErrorInvalidValue;
  }
  if (!make_pool_map(&mk, k_pages, dqk, kPB, p.hkv, p.num_pages) ||
      !make_pool_map(&mv, v_pages, dqk, kPB, p.hkv, p.num_pages))
    return cudaErrorInvalidValue;
  if (dqk == 128) return launch_d<128, kTile, 3, false>(p, mk, mv, grid, stream);
  if (dqk == 64) return launch_d<64, kTile, 4, false>(p, mk, mv, grid, stream);
  return cudaErrorInvalidValue;
}

}  // namespace specgen
