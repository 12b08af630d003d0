// Shared-prefix stage on the 5th-generation tensor cores (tcgen05 + TMA).
//
// All forks of one reasoning trace attend to the same prefix pages.  One CTA
// takes one PrefixItem: the query rows of every fork of the trace for one kv
// head, gathered into a single M = nforks * G (<= 128) row tile, against a
// contiguous chunk of the prefix.  Each prefix page of the chunk is fetched
// from HBM exactly once by TMA and used for all M rows, so the prefix is read
// once per trace instead of once per fork.
//
// Per 128-token tile j (8 pages of 16 tokens):
//   producer warp : TMA K_j, V_j pages (two 64-column boxes per page) into a
//                   2-stage ring, completion counted in bytes on full[j%2]
//   MMA warp      : S_j = Q K_j^T  -> TMEM S[j%2]    (M=128, N=16*pages, K=D)
//                   O_j = P_j V_j  -> TMEM O[j%2]    (M=128, N=D, K=16*pages)
//   4 softmax warps (thread = row = TMEM lane): online softmax in fp32 (log2
//                   domain), P_j written to shared memory as bf16 in the
//                   128B-swizzled K-major layout, and the running output
//                   O <- O * exp2(m_old - m_new) + O_j accumulated in registers.
// S and O are double-buffered in TMEM (4 x 128 columns), so S_{j+1} runs on the
// tensor cores while the softmax warps work on tile j.  Tokens past the chunk,
// past the sequence, or on an invalid page are masked to -inf; value rows past
// the sequence inside its last page are zeroed in shared memory before the PV
// product, so nothing stored there (even NaN) reaches the output.
#include <cuda.h>
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "plan.h"
#include "prefix_tc.h"
#include "tc_common.cuh"

namespace specgen {

namespace {

using namespace tc;

constexpr int kPB = 16;                      // page size (tokens)
constexpr int kTileTok = 128;                // tokens per tile
constexpr int kPagesPerTile = kTileTok / kPB;
constexpr uint32_t kPanelBytes = 128 * 128;  // 128 rows x 128 B (64 bf16 columns)
constexpr int kThreads = 192;                // warp 0 TMA, warp 1 MMA, warps 2-5 softmax
constexpr uint32_t kTmemCols = 512;

template <int D>
struct PrefixSmem {
  static constexpr int kPanels = D / 64;
  static constexpr uint32_t kQ = kPanels * kPanelBytes;
  static constexpr uint32_t kKV = kPanels * kPanelBytes;  // one K or V tile
  static constexpr uint32_t kStage = 2 * kKV;
  static constexpr uint32_t kP = 2 * kPanelBytes;         // 128 rows x 128 tokens
  static constexpr uint32_t kOffKV = kQ;
  static constexpr uint32_t kOffP = kOffKV + 2 * kStage;
  static constexpr uint32_t kOffBar = kOffP + 2 * kP;
  static constexpr uint32_t kBytes = kOffBar + 128 + 1024;  // + barriers + alignment slack
};

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b, uint32_t c,
                                             uint32_t d) {
  asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "r"(a), "r"(b), "r"(c),
               "r"(d)
               : "memory");
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    prefix_tc_kernel(const __grid_constant__ PrefixParams p, const __grid_constant__ CUtensorMap tmk,
                     const __grid_constant__ CUtensorMap tmv) {
  using L = PrefixSmem<D>;
  extern __shared__ unsigned char smem_raw[];
  // 128B-swizzled operand tiles need 1024-byte aligned bases
  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  unsigned char* gbase = smem_raw + (base - raw);
  const uint32_t sQ = base;
  const uint32_t sKV = base + L::kOffKV;
  const uint32_t sP = base + L::kOffP;
  const uint32_t bar0 = base + L::kOffBar;
  auto full = [&](int s) { return bar0 + 8u * s; };
  auto empty = [&](int s) { return bar0 + 16u + 8u * s; };
  auto s_full = [&](int b) { return bar0 + 32u + 8u * b; };
  auto p_full = [&](int b) { return bar0 + 48u + 8u * b; };
  auto o_full = [&](int b) { return bar0 + 64u + 8u * b; };
  const uint32_t q_ready = bar0 + 80u;
  const uint32_t mma_done = bar0 + 88u;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(gbase + L::kOffBar + 96);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(gbase + L::kOffBar + 100);
  auto sK = [&](int s) { return sKV + s * L::kStage; };
  auto sV = [&](int s) { return sKV + s * L::kStage + L::kKV; };

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const PrefixItem it = p.items[blockIdx.x];
  const int32_t* table = p.prefix_bt + p.prefix_bt_off[it.trace];
  const int M = it.nforks * p.G;
  const int ntiles = (it.tok_end - it.tok_begin + kTileTok - 1) / kTileTok;
  const int page0 = it.tok_begin / kPB;

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
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  auto tile_tokens = [&](int j) {
    int n = it.tok_end - (it.tok_begin + j * kTileTok);
    return n < kTileTok ? n : kTileTok;
  };

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int issued = 0;
      for (int j = 0; j < ntiles; ++j) {
        const int s = j & 1;
        if (!mbar_wait(empty(s), ((j >> 1) & 1) ^ 1, abort_flag, p.status)) break;
        const int np = (tile_tokens(j) + kPB - 1) / kPB;
        int pages[kPagesPerTile];  // fetch the tile's page ids before issuing any copy
#pragma unroll
        for (int pg = 0; pg < kPagesPerTile; ++pg)
          pages[pg] = pg < np ? table[page0 + j * kPagesPerTile + pg] : 0;
        mbar_arrive_expect_tx(full(s), (uint32_t)np * 2u * L::kPanels * (kPB * 128u));
#pragma unroll
        for (int pg = 0; pg < kPagesPerTile; ++pg) {
          if (pg >= np) break;
          const int page = pages[pg];
          if (page < 0 || page >= p.num_pages) atomicOr(p.status, kStatusIndex);  // TMA zero-fills
#pragma unroll
          for (int pn = 0; pn < L::kPanels; ++pn) {
            const uint32_t off = pn * kPanelBytes + pg * (kPB * 128u);
            tma_load_4d(sK(s) + off, &tmk, pn * 64, 0, it.kv_head, page, full(s));
            tma_load_4d(sV(s) + off, &tmv, pn * 64, 0, it.kv_head, page, full(s));
          }
        }
        issued = j + 1;
      }
      // never leave a copy in flight into this CTA's shared memory
      for (int j = issued - 2 < 0 ? 0 : issued - 2; j < issued; ++j)
        mbar_wait_drain(full(j & 1), (j >> 1) & 1, p.status);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      bool ok = mbar_wait(q_ready, 0, abort_flag, p.status);
      tc_fence_after();
      for (int j = 0; ok && j <= ntiles; ++j) {
        if (j < ntiles) {
          const int s = j & 1;
          if (!(ok = mbar_wait(full(s), (j >> 1) & 1, abort_flag, p.status))) break;
          tc_fence_after();
          const int np = (tile_tokens(j) + kPB - 1) / kPB;
          const uint32_t idesc = idesc_bf16(128, np * kPB, false);
          const uint32_t d_tmem = tmem + (uint32_t)s * 128u;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk >> 2) * kPanelBytes + (kk & 3) * 32u;
            mma_bf16(d_tmem, smem_desc_sw128(sQ + off, 16, 1024),
                     smem_desc_sw128(sK(s) + off, 16, 1024), idesc, kk > 0 ? 1u : 0u);
          }
          mma_commit(s_full(s));
        }
        if (j >= 1) {
          const int jj = j - 1, b = jj & 1;
          if (!(ok = mbar_wait(p_full(b), (jj >> 1) & 1, abort_flag, p.status))) break;
          tc_fence_after();
          const int np = (tile_tokens(jj) + kPB - 1) / kPB;
          constexpr uint32_t idesc = idesc_bf16(128, D, true);
          const uint32_t d_tmem = tmem + 256u + (uint32_t)b * 128u;
          for (int kk = 0; kk < np; ++kk) {  // one page (16 tokens) per k-step
            const uint64_t a = smem_desc_sw128(sP + b * L::kP + (kk >> 2) * kPanelBytes +
                                                   (kk & 3) * 32u, 16, 1024);
            const uint64_t v = smem_desc_sw128(sV(b) + kk * (kPB * 128u), kPanelBytes, 1024);
            mma_bf16(d_tmem, a, v, idesc, kk > 0 ? 1u : 0u);
          }
          mma_commit(o_full(b));
          mma_commit(empty(b));
        }
      }
      // every MMA issued by this thread has finished before TMEM is released
      mma_commit(mma_done);
      mbar_wait_drain(mma_done, 0, p.status);
    }
  } else {
    // ------------------------------------------------------------ softmax warps
    const int q4 = warp & 3;
    const int row = q4 * 32 + lane;
    const int tid = threadIdx.x - 64;  // 0..127
    const uint32_t lane_addr = (uint32_t)(q4 * 32) << 16;
    const bool row_ok = row < M;
    const int fl = row / p.G, gi = row % p.G;
    const int head = it.kv_head * p.G + gi;

    // Q row -> shared memory, 128B-swizzled K-major panels; rows >= M are zero
    {
      const uint4* src = reinterpret_cast<const uint4*>(
          p.q + ((size_t)(it.fork0 + (row_ok ? fl : 0)) * p.hq + head) * D);
#pragma unroll
      for (int c = 0; c < D / 8; ++c) {
        uint4 v = row_ok ? __ldg(src + c) : make_uint4(0, 0, 0, 0);
        const uint32_t dst = sQ + (c >> 3) * kPanelBytes + row * 128u + (((c & 7) ^ (row & 7)) << 4);
        st_shared_v4(dst, v.x, v.y, v.z, v.w);
      }
      fence_proxy_async_smem();
      mbar_arrive(q_ready);
    }

    const float sl2 = p.scale_log2;
    float m = -INFINITY, l = 0.f, alpha_prev = 1.f;
    float o[D];
#pragma unroll
    for (int i = 0; i < D; ++i) o[i] = 0.f;
    bool ok = true;

    auto accumulate = [&](int jj, float alpha) -> bool {
      const int b = jj & 1;
      bool w = mbar_wait(o_full(b), (jj >> 1) & 1, abort_flag, p.status);
      if (__any_sync(0xffffffffu, !w)) return false;
      tc_fence_after();
#pragma unroll
      for (int c = 0; c < D / 16; ++c) {
        uint32_t v[16];
        tmem_ld16(tmem + lane_addr + 256u + (uint32_t)b * 128u + c * 16u, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 16; ++i) o[c * 16 + i] = o[c * 16 + i] * alpha + __uint_as_float(v[i]);
      }
      return true;
    };

    for (int j = 0; j < ntiles; ++j) {
      const int b = j & 1;
      bool w = mbar_wait(s_full(b), (j >> 1) & 1, abort_flag, p.status);
      if (__any_sync(0xffffffffu, !w)) {
        ok = false;
        break;
      }
      tc_fence_after();
      const int nt = tile_tokens(j);
      const int np = (nt + kPB - 1) / kPB;
      uint32_t pv = 0;  // valid pages of this tile
      for (int pg = 0; pg < np; ++pg) {
        const int page = table[page0 + j * kPagesPerTile + pg];
        if (page >= 0 && page < p.num_pages) pv |= 1u << pg;
      }
      const uint32_t s_addr = tmem + lane_addr + (uint32_t)b * 128u;

      // pass 1: row maximum of the masked, scaled scores
      float mx = -INFINITY;
#pragma unroll
      for (int c = 0; c < 8; ++c) {
        uint32_t v[16];
        tmem_ld16(s_addr + c * 16u, v);
        tmem_wait_ld();
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const int col = c * 16 + i;
          const bool valid = col < nt && ((pv >> (col / kPB)) & 1u);
          mx = fmaxf(mx, valid ? __uint_as_float(v[i]) * sl2 : -INFINITY);
        }
      }
      const float m_new = fmaxf(m, mx);
      const float alpha = m_new == -INFINITY ? 1.f : fast_exp2(m - m_new);
      const float sub = m_new == -INFINITY ? 0.f : m_new;

      // pass 2: probabilities -> bf16 P tile (row-owned, swizzled), row sum
      float psum = 0.f;
      const uint32_t prow = sP + b * L::kP + row * 128u;
#pragma unroll
      for (int c = 0; c < 8; ++c) {  // 16 columns = two 16-byte chunks of the P row
        uint32_t v[16];
        tmem_ld16(s_addr + c * 16u, v);
        tmem_wait_ld();
        uint32_t packed[8];
#pragma unroll
        for (int i = 0; i < 16; i += 2) {
          const int col = c * 16 + i;
          const bool v0 = col < nt && ((pv >> (col / kPB)) & 1u);
          const bool v1 = col + 1 < nt && ((pv >> ((col + 1) / kPB)) & 1u);
          const float p0 = v0 ? fast_exp2(__uint_as_float(v[i]) * sl2 - sub) : 0.f;
          const float p1 = v1 ? fast_exp2(__uint_as_float(v[i + 1]) * sl2 - sub) : 0.f;
          psum += p0 + p1;
          packed[i >> 1] = pack_bf16x2(p0, p1);
        }
#pragma unroll
        for (int t = 0; t < 2; ++t) {
          const int chunk = (c & 3) * 2 + t;
          st_shared_v4(prow + (c >> 2) * kPanelBytes + ((chunk ^ (row & 7)) << 4),
                       packed[4 * t], packed[4 * t + 1], packed[4 * t + 2], packed[4 * t + 3]);
        }
      }
      l = l * alpha + psum;
      m = m_new;

      // value rows past the sequence inside its last page: zero them before PV
      if (j == ntiles - 1 && (nt % kPB) != 0) {
        const int pg = np - 1, first = nt % kPB;
        const int units = (kPB - first) * L::kPanels * 8;
        for (int u = tid; u < units; u += 128) {
          const int rr = first + u / (L::kPanels * 8);
          const int rem = u % (L::kPanels * 8);
          st_shared_v4(sV(b) + (rem >> 3) * kPanelBytes + (pg * kPB + rr) * 128u + ((rem & 7) << 4),
                       0u, 0u, 0u, 0u);
        }
      }
      tc_fence_before();
      fence_proxy_async_smem();
      mbar_arrive(p_full(b));

      if (j >= 1 && !accumulate(j - 1, alpha_prev)) {
        ok = false;
        break;
      }
      alpha_prev = alpha;
    }
    if (ok && ntiles > 0) ok = accumulate(ntiles - 1, alpha_prev);

    if (ok && row_ok) {
      const int fork = it.fork0 + fl;
      const int slot = p.part_base[fork] + it.chunk;
      const size_t prow_out = (size_t)slot * p.hq + head;
      const float inv = l > 0.f ? 1.f / l : 0.f;
      float4* dst = reinterpret_cast<float4*>(p.part_o + prow_out * p.dv + it.dv0);
#pragma unroll
      for (int c = 0; c < D / 4; ++c)
        dst[c] = make_float4(o[4 * c] * inv, o[4 * c + 1] * inv, o[4 * c + 2] * inv,
                             o[4 * c + 3] * inv);
      p.part_lse[prow_out] = m == -INFINITY ? -INFINITY : (m + log2f(l)) * kLn2;
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

template <int D>
cudaError_t launch_d(const PrefixParams& p, const CUtensorMap& mk, const CUtensorMap& mv,
                     int n_items, cudaStream_t stream) {
  constexpr int smem = (int)PrefixSmem<D>::kBytes;
  static_assert(smem <= 232448, "prefix kernel shared memory exceeds 227 KB");
  auto kern = prefix_tc_kernel<D>;
  static thread_local int configured = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured != dev) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured = dev;
  }
  kern<<<n_items, kThreads, smem, stream>>>(p, mk, mv);
  return cudaGetLastError();
}

}  // namespace

bool prefix_tc_supported(int dqk, int dv, bool latent, int page_size, int G) {
  return !latent && dqk == dv && (dqk == 64 || dqk == 128) && page_size == kPB && G <= 128;
}

int prefix_tc_tile_tokens() { return kTileTok; }
int prefix_tc_page_size() { return kPB; }

cudaError_t launch_prefix_tc(const PrefixParams& p, const void* k_pages, const void* v_pages,
                             int n_items, int dqk, cudaStream_t stream) {
  if (n_items == 0) return cudaSuccess;
  CUtensorMap mk, mv;
  if (!make_pool_map(&mk, k_pages, dqk, kPB, p.hkv, p.num_pages) ||
      !make_pool_map(&mv, v_pages, dqk, kPB, p.hkv, p.num_pages))
    return cudaErrorInvalidValue;
  if (dqk == 128) return launch_d<128>(p, mk, mv, n_items, stream);
  if (dqk == 64) return launch_d<64>(p, mk, mv, n_items, stream);
  return cudaErrorInvalidValue;
}

}  // namespace specgen
