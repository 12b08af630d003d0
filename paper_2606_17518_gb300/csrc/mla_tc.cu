// Fork decode over a latent (MLA-style) KV cache on tcgen05 tensor cores.
//
// Shape: 128 query heads attend to one latent KV head whose 576-wide row is
// both the key (512 latent + 64 rotary columns, absorbed scoring) and, in its
// first 512 columns, the value; pages hold 64 tokens.  Every fork has its own
// 128 query rows, so one item is one fork (M = 128 rows = heads) against a
// chunk of its prefix or suffix.  The forks of a trace read the same prefix
// chunks; the prefix stays resident in L2 while they do.
//
// Tensor memory cannot hold a 128 x 512 fp32 output next to the scores, so an
// item produces one half of the value columns (dv0 = 0 or 256); the score tile
// is computed for each half.  Q (128 x 576 bf16, 144 KB) does not fit in
// shared memory next to two 64-token K tiles (72 KB each), so its first 256
// columns live in tensor memory (the A operand of the first 16 k-steps) and
// the other 320 in shared memory.  Per 64-token tile t (one page):
//   warp 0 (TMA)   the page as one box (nine panels of 64 rows x 64 columns,
//                  128B swizzle) -> 2-stage ring
//   warp 1 (MMA)   S_t = Q K_t^T (36 k-steps, N = 64; A from TMEM, then shared
//                  memory), then O += P_t V_t[:, dv0:dv0+256] (A = P in TMEM, N = 256)
//   warps 2-5      one thread per head: the tile's scores, masked, online
//                  softmax in log2 units with lazy rescaling, P back to TMEM
//                  as bf16 pairs.
// Value rows past a sequence inside its last tile are zeroed in shared memory
// before the PV product; every wait is bounded.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "mla_tc.h"
#include "plan.h"
#include "tc_common.cuh"

namespace specgen {

namespace {

using namespace tc;

constexpr int kDqk = 576;
constexpr int kDv = 512;
constexpr int kDvHalf = 256;
constexpr int kPage = 64;
constexpr int kTT = 64;                      // tokens per tile (one page)
constexpr int kST = 2;                       // pipeline stages
constexpr int kPanels = kDqk / 64;           // 9 column panels of 64
constexpr int kSteps = kDqk / 16;            // 36 k-steps of 16 for the scores
constexpr int kThreads = 192;                // warp 0 TMA, warp 1 MMA, warps 2-5 softmax
constexpr uint32_t kTmemCols = 512;          // S[0] [0,64) S[1] [64,128) Q [128,256) O [256,512)
constexpr uint32_t kTmemQ = 128;
constexpr uint32_t kTmemO = 256;
constexpr int kQTmemPanels = 4;              // Q columns [0, 256) in TMEM: k-steps 0..15
constexpr float kRescaleLog2 = 8.0f;
constexpr uint32_t kQPanel = 128 * 128u;     // 128 rows x 128 B
constexpr uint32_t kKPanel = kTT * 128u;     // 64 rows x 128 B
constexpr uint32_t kOffKV = (kPanels - kQTmemPanels) * kQPanel;  // Q panels 4..8
constexpr uint32_t kStage = kPanels * kKPanel;
constexpr uint32_t kOffBar = kOffKV + kST * kStage;
constexpr uint32_t kSmemBytes = kOffBar + 256 + 1024;
static_assert(kSmemBytes <= 232448, "latent kernel shared memory exceeds 227 KB");

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    mla_tc_kernel(const __grid_constant__ MlaParams p, const __grid_constant__ CUtensorMap tmk) {
  extern __shared__ unsigned char smem_raw[];
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  unsigned char* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base;
  const uint32_t bar0 = base + kOffBar;
  auto full = [&](int s) { return bar0 + 8u * s; };
  auto empty = [&](int s) { return bar0 + 8u * (2 + s); };
  auto s_full = [&](int b) { return bar0 + 8u * (4 + b); };
  auto p_full = [&](int b) { return bar0 + 8u * (6 + b); };
  auto o_full = [&](int b) { return bar0 + 8u * (8 + b); };  // PV_u done -> o_full[u%2]
  const uint32_t q_ready = bar0 + 80u;
  const uint32_t mma_done = bar0 + 88u;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + kOffBar + 96);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + kOffBar + 100);
  auto sK = [&](int s) { return base + kOffKV + s * kStage; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  // the merge (a programmatic dependent) may be launched now: it waits for this
  // grid's completion before it reads any partial
  if (threadIdx.x == 0) asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
  const int it_begin = p.cta_offsets[blockIdx.x], it_end = p.cta_offsets[blockIdx.x + 1];
  auto table_of = [&](const TcItem& it) {
    const int32_t* bt = it.table_kind == 0 ? p.prefix_bt : p.suffix_bt;
    return bt + (it.table_off >= 0 ? it.table_off
                                   : (it.table_kind == 0 ? p.prefix_bt_off : p.suffix_bt_off)[it.seq]);
  };
  auto ntiles_of = [&](const TcItem& it) { return (it.tok_end - it.tok_begin + kTT - 1) / kTT; };
  auto tile_tokens = [&](const TcItem& it, int j) {
    const int n = it.tok_end - (it.tok_begin + j * kTT);
    return n < kTT ? n : kTT;
  };

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(full(i), 1);
      mbar_init(empty(i), 1);
      mbar_init(s_full(i), 1);
      mbar_init(p_full(i), 128);
      mbar_init(o_full(i), 1);
    }
    mbar_init(q_ready, 128);
    mbar_init(mma_done, 1);
    *abort_flag = 0;
    mbar_init_fence();
  }
  if (warp == 1) {
    tmem_alloc(smem_u32(tmem_slot), kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  // Launched as a programmatic dependent, the grid may start while the stream's
  // previous kernel is still running: everything above touches only this CTA's
  // own resources and the plan (written by a host copy).  Inputs (lengths,
  // tables, Q, the pool) and the partial buffers are used only after this wait.
  asm volatile("griddepcontrol.wait;\n" ::: "memory");
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    // A tile is one page; page ids are fetched 32 at a time by the warp, one
    // batch ahead.  Lane 0 issues the tile as one box: all nine 64-column
    // panels of the page, landing panel after panel.
    int t = 0;
    bool ok = true;
    for (int ii = it_begin; ok && ii < it_end; ++ii) {
      const TcItem it = clamp_item(p.items[ii], p.suffix_lens);
      const int32_t* table = table_of(it);
      const int ntiles = ntiles_of(it);
      const int page0 = it.tok_begin / kPage;
      const int npages = ntiles;  // one page per tile
      int cur = lane < npages ? table[page0 + lane] : 0;
      int nxt = 32 + lane < npages ? table[page0 + 32 + lane] : 0;
      int batch = 0;
      for (int j = 0; j < ntiles; ++j, ++t) {
        const int tok = it.tok_begin + j * kTT;
        const int pidx = tok / kPage - page0;
        while ((pidx >> 5) > batch) {
          cur = nxt;
          ++batch;
          nxt = batch * 32 + 32 + lane < npages ? table[page0 + batch * 32 + 32 + lane] : 0;
        }
        const int page = __shfl_sync(0xffffffffu, cur, pidx & 31);
        const int slot0 = tok % kPage;
        const int s = t % kST;
        if (lane == 0) {
          ok = mbar_wait(empty(s), ((t / kST) & 1) ^ 1, abort_flag, p.status);
          if (ok) mbar_arrive_expect_tx(full(s), kStage);
        }
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (!ok) break;
        if (lane == 0) tma_load_4d(sK(s), &tmk, 0, slot0, 0, page, full(s));
        if (lane == 0 && (page < 0 || page >= p.num_pages)) atomicOr(p.status, kStatusIndex);
      }
    }
    if (lane == 0)
      for (int u = t - kST < 0 ? 0 : t - kST; u < t; ++u)
        mbar_wait_drain(full(u % kST), (u / kST) & 1, p.status);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      // descriptors are built once; every MMA adds a constant offset to them
      const uint64_t dq = smem_desc_sw128(sQ, 16, 1024);  // Q panels 4..8 from panel 0 here
      const uint64_t dk0 = smem_desc_sw128(sK(0), 16, 1024);
      const uint64_t dvb0 = smem_desc_sw128(sK(0), kKPanel, 1024);
      constexpr uint64_t kStageDesc = kStage >> 4;
      constexpr uint32_t idesc_s = idesc_bf16(128, kTT, false);
      constexpr uint32_t idesc_pv = idesc_bf16(128, kDvHalf, true);
      // Ready-first issue: PV_v goes out as soon as its P is ready; S_u goes
      // out when its K tile has landed, its score buffer is free (PV_{u-2}
      // issued, so in-order execution has consumed P_{u-2}) and, for an item's
      // first tile, its Q is in shared memory.  s_*: the next S to issue,
      // v_*: the next PV to issue (item cursor, tile within item, global tile).
      int s_ii = it_begin, s_j = 0, s_u = 0, v_ii = it_begin, v_j = 0, v_u = 0;
      TcItem s_it = s_ii < it_end ? clamp_item(p.items[s_ii], p.suffix_lens) : TcItem{};
      TcItem v_it = s_it;
      bool q_ok = false;  // Q of the item at s_ii is known to be loaded
      bool ok = true;
      unsigned long long t0 = 0;
      // items cut to nothing by the current suffix lengths: the PV cursor steps
      // over them, the S cursor still takes their Q phase
      while (v_ii < it_end && ntiles_of(v_it) == 0 && ++v_ii < it_end)
        v_it = clamp_item(p.items[v_ii], p.suffix_lens);
      while (ok && (v_ii < it_end || s_ii < it_end)) {
        bool did = false;
        if (s_ii < it_end && ntiles_of(s_it) == 0 &&
            mbar_test_wait(q_ready, (s_ii - it_begin) & 1)) {
          q_ok = false;
          if (++s_ii < it_end) s_it = clamp_item(p.items[s_ii], p.suffix_lens);
          did = true;
        } else if (v_u < s_u && mbar_test_wait(p_full(v_u & 1), (v_u >> 1) & 1)) {
          tc_fence_after();
          const int b = v_u & 1, s = v_u % kST;
          const uint64_t vpanel = (uint64_t)((v_it.dv0 / 64) * kKPanel) >> 4;
          const uint64_t dv = dvb0 + (uint64_t)s * kStageDesc + vpanel;
#pragma unroll
          for (int kk = 0; kk < kTT / 16; ++kk)  // 16 tokens (16 rows x 128 B) a step
            mma_bf16_ts(tmem + kTmemO, tmem + (uint32_t)b * kTT + kk * 8u,
                        dv + (uint64_t)((kk * 2048u) >> 4), idesc_pv,
                        (v_j > 0 || kk > 0) ? 1u : 0u);
          mma_commit(o_full(b));
          mma_commit(empty(s));
          ++v_u;
          if (++v_j == ntiles_of(v_it)) {
            v_j = 0;
            do {
              if (++v_ii < it_end) v_it = clamp_item(p.items[v_ii], p.suffix_lens);
            } while (v_ii < it_end && ntiles_of(v_it) == 0);
          }
          did = true;
        } else if (s_ii < it_end && ntiles_of(s_it) > 0 && s_u - v_u < 2) {
          if (!q_ok && mbar_test_wait(q_ready, (s_ii - it_begin) & 1)) q_ok = true;
          if (q_ok && mbar_test_wait(full(s_u % kST), (s_u / kST) & 1)) {
            tc_fence_after();
            const int b = s_u & 1, s = s_u % kST;
            const uint64_t dk = dk0 + (uint64_t)s * kStageDesc;
            const uint32_t d_s = tmem + (uint32_t)b * kTT;
#pragma unroll
            for (int kk = 0; kk < kQTmemPanels * 4; ++kk) {  // A = Q from TMEM, 8 columns a step
              const uint64_t ko = ((kk >> 2) * kKPanel + (kk & 3) * 32u) >> 4;
              mma_bf16_ts(d_s, tmem + kTmemQ + kk * 8u, dk + ko, idesc_s, kk > 0 ? 1u : 0u);
            }
#pragma unroll
            for (int kk = kQTmemPanels * 4; kk < kSteps; ++kk) {  // A = Q from shared memory
              const uint64_t qo = (((kk >> 2) - kQTmemPanels) * kQPanel + (kk & 3) * 32u) >> 4;
              const uint64_t ko = ((kk >> 2) * kKPanel + (kk & 3) * 32u) >> 4;
              mma_bf16(d_s, dq + qo, dk + ko, idesc_s, 1u);
            }
            mma_commit(s_full(b));
            ++s_u;
            if (++s_j == ntiles_of(s_it)) {
              s_j = 0;
              q_ok = false;
              if (++s_ii < it_end) s_it = clamp_item(p.items[s_ii], p.suffix_lens);
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
      mma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, p.status);
    }
  } else {
    // ------------------------------------------------------------ softmax warps
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;  // query head
    const int tid = threadIdx.x - 64;
    const uint32_t lane_addr = (uint32_t)(q4 * 32) << 16;
    const uint32_t s_base = tmem + lane_addr;
    const uint32_t o_base = tmem + lane_addr + kTmemO;
    const float sl2 = p.scale_log2;
    int t = 0, oc = 0;  // tiles done; next o_full phase (tile index) to consume
    bool ok = true;
    for (int ii = it_begin; ok && ii < it_end; ++ii) {
      const TcItem it = clamp_item(p.items[ii], p.suffix_lens);
      // this fork's partial slot base, fetched now and used at the item's end
      const int pbase = p.part_base[it.fork0];
      const int32_t* table = table_of(it);
      const int ntiles = ntiles_of(it);
      const int page0 = it.tok_begin / kPage;

      {  // Q row of this head: columns [0, 256) -> TMEM (this thread's lane),
         // the rest -> shared memory as five 128B-swizzled panels.  The shared-
         // memory part goes out first as asynchronous 16-byte copies; the TMEM
         // part is loaded in two batches of 16 pieces meanwhile, so the whole
         // row costs about two memory round trips instead of one per 8 pieces.
        const uint4* src = reinterpret_cast<const uint4*>(p.q + ((size_t)it.fork0 * 128 + row) * kDqk);
#pragma unroll
        for (int c = kQTmemPanels * 8; c < kDqk / 8; ++c)
          cp_async_16(sQ + ((c >> 3) - kQTmemPanels) * kQPanel + row * 128u +
                          (((c & 7) ^ (row & 7)) << 4),
                      src + c, 16);
        cp_async_commit();
#pragma unroll
        for (int half = 0; half < 2; ++half) {  // 16 x 16 B = 64 TMEM columns a batch
          uint4 q[16];
#pragma unroll
          for (int e = 0; e < 16; ++e) q[e] = __ldg(src + half * 16 + e);
#pragma unroll
          for (int h2 = 0; h2 < 2; ++h2) {
            uint32_t v[32];
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              v[4 * e] = q[h2 * 8 + e].x;
              v[4 * e + 1] = q[h2 * 8 + e].y;
              v[4 * e + 2] = q[h2 * 8 + e].z;
              v[4 * e + 3] = q[h2 * 8 + e].w;
            }
            tmem_st32(s_base + kTmemQ + (uint32_t)((half * 16 + h2 * 8) * 4), v);
          }
        }
        cp_async_wait<0>();
        tmem_wait_st();
        fence_proxy_async_smem();
        tc_fence_before();
        mbar_arrive(q_ready);
      }

      float m = -INFINITY, l = 0.f;
      for (int j = 0; j < ntiles; ++j) {
        const int u = t + j, b = u & 1;
        const bool w = mbar_wait(s_full(b), (u >> 1) & 1, abort_flag, p.status);
        if (__any_sync(0xffffffffu, !w)) {
          ok = false;
          break;
        }
        tc_fence_after();
        while (oc <= u - 2) {  // S_u done => PV_{u-2} done
          mbar_wait(o_full(oc & 1), (oc >> 1) & 1, abort_flag, p.status);
          ++oc;
        }
        const int nt = tile_tokens(it, j);
        const int tok = it.tok_begin + j * kTT;
        const int page = table[tok / kPage];
        const bool page_ok = page >= 0 && page < p.num_pages;
        float s[kTT];
        {
          uint32_t r[kTT / 32][32];
#pragma unroll
          for (int c = 0; c < kTT / 32; ++c) tmem_ld32(s_base + (uint32_t)b * kTT + c * 32u, r[c]);
          tmem_wait_ld();
#pragma unroll
          for (int c = 0; c < kTT / 32; ++c)
#pragma unroll
            for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(r[c][i]);
        }
        if (nt < kTT || !page_ok) {
#pragma unroll
          for (int i = 0; i < kTT; ++i)
            if (!(i < nt && page_ok)) s[i] = -INFINITY;
        }
        float mx0 = s[0], mx1 = s[1], mx2 = s[2], mx3 = s[3];
#pragma unroll
        for (int i = 4; i < kTT; i += 4) {
          mx0 = fmaxf(mx0, s[i]);
          mx1 = fmaxf(mx1, s[i + 1]);
          mx2 = fmaxf(mx2, s[i + 2]);
          mx3 = fmaxf(mx3, s[i + 3]);
        }
        const float m_tile = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * sl2;
        bool rescale = false;
        float alpha = 1.f;
        if (m_tile > m + kRescaleLog2 || (m == -INFINITY && m_tile != -INFINITY)) {
          alpha = m == -INFINITY ? 0.f : fast_exp2(m - m_tile);
          rescale = m != -INFINITY;
          l *= alpha;
          m = m_tile;
        }
        const float sub = m == -INFINITY ? 0.f : m;
        {
          uint32_t pk[kTT / 2];
          float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
          for (int i = 0; i < kTT / 2; ++i) {
            const float p0 = fast_exp2(fmaf(s[2 * i], sl2, -sub));
            const float p1 = fast_exp2(fmaf(s[2 * i + 1], sl2, -sub));
            ps0 += p0;
            ps1 += p1;
            pk[i] = pack_bf16x2(p0, p1);
          }
          tmem_st32(s_base + (uint32_t)b * kTT, pk);
          l += ps0 + ps1;
        }
        // value rows past the sequence in this tile: zero them before PV
        if (nt < kTT) {
          const int units = (kTT - nt) * 4 * 8;  // rows x 4 value panels x 8 chunks
          for (int x = tid; x < units; x += 128) {
            const int rr = nt + x / 32, rem = x % 32;
            st_shared_v4(sK(u % kST) + (it.dv0 / 64 + (rem >> 3)) * kKPanel + rr * 128u +
                             ((rem & 7) << 4), 0u, 0u, 0u, 0u);
          }
          fence_proxy_async_smem();
        }
        if (j >= 1 && __any_sync(0xffffffffu, rescale)) {
          bool w2 = true;
          while (oc <= u - 1) {
            w2 = w2 && mbar_wait(o_full(oc & 1), (oc >> 1) & 1, abort_flag, p.status);
            ++oc;
          }
          if (__any_sync(0xffffffffu, !w2)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const float a = rescale ? alpha : 1.f;
          for (int c = 0; c < kDvHalf / 32; ++c) {
            uint32_t r[32];
            tmem_ld32(o_base + c * 32u, r);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) r[i] = __float_as_uint(__uint_as_float(r[i]) * a);
            tmem_st32(o_base + c * 32u, r);
          }
        }
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(p_full(b));
      }
      if (!ok) break;
      {  // end of item: last PV, then the partial (O / l, LSE) of this half
        const int u = t + ntiles - 1;
        bool w = true;
        while (oc <= u) {
          w = w && mbar_wait(o_full(oc & 1), (oc >> 1) & 1, abort_flag, p.status);
          ++oc;
        }
        if (__any_sync(0xffffffffu, !w)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const size_t prow = (size_t)(pbase + it.part) * p.hq + row;
        float4* dst = reinterpret_cast<float4*>(p.part_o) +
                      part_o_f4((size_t)pbase + it.part, row, it.dv0 / 4, p.hq, kDv);
        const float inv = l > 0.f ? 1.f / l : 0.f;
        for (int c = 0; c < kDvHalf / 32; ++c) {
          uint32_t r[32];
          tmem_ld32(o_base + c * 32u, r);
          tmem_wait_ld();
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            dst[(size_t)(c * 8 + i / 4) * p.hq] =
                make_float4(__uint_as_float(r[i]) * inv, __uint_as_float(r[i + 1]) * inv,
                            __uint_as_float(r[i + 2]) * inv, __uint_as_float(r[i + 3]) * inv);
        }
        if (it.dv0 == 0) p.part_lse[prow] = m == -INFINITY ? -INFINITY : (m + log2f(l)) * kLn2;
        tc_fence_before();
      }
      (void)page0;
      t += ntiles;
    }
  }

  tc_fence_before();
  // non-aligned CTA barrier: it counts every thread, so the lanes of a warp may
  // arrive apart (lanes 1-31 of the MMA warp come here at once, its lane 0 and
  // the copy lane only after their drains).  An aligned __syncthreads() there
  // could complete before the softmax warps' last TMEM loads.
  asm volatile("barrier.sync 0;\n" ::: "memory");
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

}  // namespace

bool mla_tc_supported(int dqk, int dv, bool latent, int page_size, int hq, int hkv) {
  return latent && dqk == kDqk && dv == kDv && page_size == kPage && hq == 128 && hkv == 1;
}

int mla_tc_tile_tokens() { return kTT; }

cudaError_t launch_mla_tc(const MlaParams& p, const void* k_pages, int grid, cudaStream_t stream) {
  if (grid == 0) return cudaSuccess;
  EncodeTiledFn enc = encode_fn();
  if (!enc || !k_pages || p.num_pages < 1) return cudaErrorInvalidValue;
  // latent pool [num_pages][64][576] as a 4-D tensor (64 columns, 64 rows, 9
  // panels, pages) with the panel stride (128 B) inside the row stride: one box
  // is a whole page, landing as [panel][row][128 B], 128-byte swizzled
  CUtensorMap mk;
  const cuuint64_t dims[4] = {64, (cuuint64_t)kPage, (cuuint64_t)kPanels, (cuuint64_t)p.num_pages};
  const cuuint64_t strides[3] = {(cuuint64_t)kDqk * 2, 128, (cuuint64_t)kPage * kDqk * 2};
  const cuuint32_t box[4] = {64, kTT, (cuuint32_t)kPanels, 1};
  const cuuint32_t estr[4] = {1, 1, 1, 1};
  if (enc(&mk, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(k_pages), dims, strides,
          box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) != CUDA_SUCCESS)
    return cudaErrorInvalidValue;
  static thread_local int configured = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured != dev) {
    e = cudaFuncSetAttribute(mla_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kSmemBytes);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(mla_tc_kernel, cudaFuncAttributePreferredSharedMemoryCarveout,
                             (int)cudaSharedmemCarveoutMaxShared);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  // programmatic dependent launch: the prologue overlaps the previous kernel
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)grid);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = (size_t)kSmemBytes;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, mla_tc_kernel, p, mk);
}

}  // namespace specgen
