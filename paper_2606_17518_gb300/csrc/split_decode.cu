// Split-K paged decode kernel (the per-fork suffix stage).
//
// One CTA computes one SplitItem: up to 16 query rows of one fork (the G query
// heads of one kv head; 16 of the 128 heads for latent KV) against a
// contiguous range of logical tokens of one paged sequence, and writes the
// partial (O / l, LSE) of that range.  This is the memory-bound part of fork
// decode: each fork's private continuation is read by that fork alone, so the
// kernel is built to stream pages at HBM speed:
//   * 16-byte cp.async copies, one (page, kv-head) run of rows is contiguous in
//     the pool, so consecutive threads read consecutive 16-byte chunks;
//   * a STAGES-deep shared-memory ring (tiles of 64 tokens) keeps several tiles
//     of K and V in flight per CTA;
//   * rows past the range and pages with an invalid id are zero-filled by the
//     copy itself (src-size 0) and masked to -inf, so nothing past a
//     sequence's length is ever read;
//   * QK^T and PV run on mma.sync m16n8k16 (bf16 in, fp32 accumulate); the
//     online softmax keeps fp32 running max/sum per row with quad shuffles;
//   * the four warps split each tile's tokens and are combined by log-sum-exp
//     in shared memory at the end.
// Softmax is done in the log2 domain: s' = s * scale * log2(e), exp2, and the
// stored LSE is converted back to natural log.
#include <cuda_runtime.h>
#include <math.h>

#include "common.cuh"
#include "plan.h"
#include "split_decode.h"

namespace specgen {

namespace {

constexpr int kTile = 64;      // tokens per pipeline stage
constexpr int kWarps = 4;      // each warp owns 16 tokens of a tile
constexpr int kThreads = kWarps * 32;
constexpr int kRows = 16;      // mma M

template <int DQK, int DVT, bool LATENT>
struct SplitSmem {
  static constexpr int kRowK = DQK * 2;                    // bytes per K row
  static constexpr int kRowV = DVT * 2;                    // bytes per V row (separate pool)
  static constexpr int kTileK = kTile * kRowK;
  static constexpr int kTileV = LATENT ? 0 : kTile * kRowV;
  static constexpr int kStage = kTileK + kTileV;
  static constexpr int kQ = kRows * kRowK;
};

template <int DQK, int DVT, bool LATENT, int STAGES>
constexpr int split_smem_bytes() {
  using S = SplitSmem<DQK, DVT, LATENT>;
  int main = STAGES * S::kStage + S::kQ + STAGES * kTile;  // + token-valid flags
  int combine = kWarps * kRows * (DVT + 2) * 4;
  return main > combine ? main : combine;
}

template <int DQK, int DVT, bool LATENT, int STAGES>
__global__ void __launch_bounds__(kThreads, 2) split_decode_kernel(const SplitParams p) {
  using S = SplitSmem<DQK, DVT, LATENT>;
  extern __shared__ __align__(128) unsigned char smem[];
  unsigned char* s_kv = smem;                                  // STAGES * kStage
  unsigned char* s_q = smem + STAGES * S::kStage;              // kQ
  uint8_t* s_ok = reinterpret_cast<uint8_t*>(s_q + S::kQ);     // STAGES * kTile

  SplitItem it = p.items[blockIdx.x];
  if (p.suffix_lens != nullptr && it.table_kind == 1) {  // one plan, several decode steps
    const int n = p.suffix_lens[it.seq];
    it.tok_end = n < it.tok_begin ? it.tok_begin : (n < it.tok_end ? n : it.tok_end);
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int B = p.page_size;
  const int32_t* table = it.table_kind == 0 ? p.prefix_bt + p.prefix_bt_off[it.seq]
                                            : p.suffix_bt + p.suffix_bt_off[it.seq];
  const __nv_bfloat16* kpool = p.k_pages;
  const __nv_bfloat16* vpool = LATENT ? p.k_pages : p.v_pages;
  const int vdq = LATENT ? DQK : p.dv;  // row length (elements) of the V pool
  const int ntok = it.tok_end - it.tok_begin;
  const int ntiles = (ntok + kTile - 1) / kTile;

  // ---- query rows -> shared memory (rows >= nrows are zero) ----
  {
    constexpr int kChunks = DQK / 8;
    for (int i = tid; i < kRows * kChunks; i += kThreads) {
      int r = i / kChunks, c = i % kChunks;
      int src_bytes = r < it.nrows ? 16 : 0;
      const __nv_bfloat16* src =
          p.q + ((size_t)it.fork * p.hq + it.h0 + (r < it.nrows ? r : 0)) * DQK + c * 8;
      cp_async_16(smem_u32(s_q) + swz(r, c, S::kRowK), src, src_bytes);
    }
  }

  // ---- tile loader: K (and V) rows of tokens [base, base + kTile) ----
  auto load_tile = [&](int t, int stage) {
    unsigned char* sk = s_kv + stage * S::kStage;
    const int base = it.tok_begin + t * kTile;
    constexpr int kChunksK = DQK / 8;
    for (int i = tid; i < kTile * kChunksK; i += kThreads) {
      int r = i / kChunksK, c = i % kChunksK;
      int j = base + r;
      int page = j < it.tok_end ? table[j / B] : 0;
      bool ok = j < it.tok_end && page >= 0 && page < p.num_pages;
      if (j < it.tok_end && !ok && c == 0) atomicOr(p.status, kStatusIndex);
      size_t row = ok ? ((size_t)page * p.hkv + it.kv_head) * B + (j % B) : 0;
      cp_async_16(smem_u32(sk) + swz(r, c, S::kRowK), kpool + row * DQK + c * 8, ok ? 16 : 0);
      if (c == 0) s_ok[stage * kTile + r] = ok ? 1 : 0;
    }
    if constexpr (!LATENT) {
      unsigned char* sv = sk + S::kTileK;
      constexpr int kChunksV = DVT / 8;
      for (int i = tid; i < kTile * kChunksV; i += kThreads) {
        int r = i / kChunksV, c = i % kChunksV;
        int j = base + r;
        int page = j < it.tok_end ? table[j / B] : 0;
        bool ok = j < it.tok_end && page >= 0 && page < p.num_pages;
        size_t row = ok ? ((size_t)page * p.hkv + it.kv_head) * B + (j % B) : 0;
        cp_async_16(smem_u32(sv) + swz(r, c, S::kRowV), vpool + row * vdq + it.dv0 + c * 8,
                    ok ? 16 : 0);
      }
    }
  };

  // prologue: Q travels with the first tile's group
#pragma unroll
  for (int s = 0; s < STAGES - 1; ++s) {
    if (s < ntiles) load_tile(s, s);
    cp_async_commit();
  }

  // per-lane state: rows r0 = lane/4 and r1 = lane/4 + 8
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
  float o[DVT / 8][4];
#pragma unroll
  for (int n = 0; n < DVT / 8; ++n) o[n][0] = o[n][1] = o[n][2] = o[n][3] = 0.f;

  const float sl2 = p.scale_log2;
  const int tb = warp * 16;  // this warp's first token within a tile
  const uint32_t q_base = smem_u32(s_q);

  for (int t = 0; t < ntiles; ++t) {
    cp_async_wait<STAGES - 2>();
    __syncthreads();
    {
      int nt = t + STAGES - 1;
      if (nt < ntiles) load_tile(nt, nt % STAGES);
      cp_async_commit();
    }
    const int stage = t % STAGES;
    const uint32_t k_base = smem_u32(s_kv + stage * S::kStage);
    const uint8_t* ok = s_ok + stage * kTile;

    // ---- S = Q K^T for this warp's 16 tokens (two n-tiles of 8) ----
    float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll
    for (int ks = 0; ks < DQK / 16; ++ks) {
      uint32_t a[4], b[4];
      {
        int mi = lane >> 3;
        int r = ((mi & 1) << 3) + (lane & 7);
        int c = 2 * ks + (mi >> 1);
        ldmatrix_x4(q_base + swz(r, c, S::kRowK), a[0], a[1], a[2], a[3]);
      }
      {
        int mi = lane >> 3;
        int r = tb + ((mi >> 1) << 3) + (lane & 7);
        int c = 2 * ks + (mi & 1);
        ldmatrix_x4(k_base + swz(r, c, S::kRowK), b[0], b[1], b[2], b[3]);
      }
      mma_bf16_16816(s[0], a, b[0], b[1]);
      mma_bf16_16816(s[1], a, b[2], b[3]);
    }

    // ---- online softmax (log2 domain) ----
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        int tok = tb + nt * 8 + ((lane & 3) << 1) + e;
        bool v = ok[tok] != 0 && (it.tok_begin + t * kTile + tok) < it.tok_end;
        s[nt][e] = v ? s[nt][e] * sl2 : -INFINITY;
        s[nt][e + 2] = v ? s[nt][e + 2] * sl2 : -INFINITY;
        mx0 = fmaxf(mx0, s[nt][e]);
        mx1 = fmaxf(mx1, s[nt][e + 2]);
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float nm0 = fmaxf(m0, mx0), nm1 = fmaxf(m1, mx1);
    // an all-masked history keeps m = -inf: nothing to rescale, p = 0
    const float al0 = nm0 == -INFINITY ? 1.f : fast_exp2(m0 - nm0);
    const float al1 = nm1 == -INFINITY ? 1.f : fast_exp2(m1 - nm1);
    const float sub0 = nm0 == -INFINITY ? 0.f : nm0;
    const float sub1 = nm1 == -INFINITY ? 0.f : nm1;
    m0 = nm0;
    m1 = nm1;
    float ps0 = 0.f, ps1 = 0.f;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        s[nt][e] = fast_exp2(s[nt][e] - sub0);
        s[nt][e + 2] = fast_exp2(s[nt][e + 2] - sub1);
        ps0 += s[nt][e];
        ps1 += s[nt][e + 2];
      }
    }
    l0 = l0 * al0 + ps0;
    l1 = l1 * al1 + ps1;
#pragma unroll
    for (int n = 0; n < DVT / 8; ++n) {
      o[n][0] *= al0;
      o[n][1] *= al0;
      o[n][2] *= al1;
      o[n][3] *= al1;
    }

    // ---- O += P V ----
    uint32_t pa[4];
    pa[0] = pack_bf16x2(s[0][0], s[0][1]);
    pa[1] = pack_bf16x2(s[0][2], s[0][3]);
    pa[2] = pack_bf16x2(s[1][0], s[1][1]);
    pa[3] = pack_bf16x2(s[1][2], s[1][3]);
    const uint32_t v_base = LATENT ? k_base : k_base + S::kTileK;
    constexpr int kRowVb = LATENT ? S::kRowK : S::kRowV;
    const int vchunk0 = LATENT ? it.dv0 / 8 : 0;  // latent V = leading K columns
#pragma unroll
    for (int np = 0; np < DVT / 16; ++np) {
      uint32_t b[4];
      int mi = lane >> 3;
      int r = tb + ((mi & 1) << 3) + (lane & 7);
      int c = vchunk0 + 2 * np + (mi >> 1);
      ldmatrix_x4_trans(v_base + swz(r, c, kRowVb), b[0], b[1], b[2], b[3]);
      mma_bf16_16816(o[2 * np], pa, b[0], b[1]);
      mma_bf16_16816(o[2 * np + 1], pa, b[2], b[3]);
    }
  }
  cp_async_wait<0>();
  __syncthreads();  // every warp is done with the ring; reuse it for the combine

  // ---- quad-reduce the running sums, then combine the four warps ----
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  float* c_o = reinterpret_cast<float*>(smem);                   // [warp][row][DVT]
  float* c_m = c_o + kWarps * kRows * DVT;                       // [warp][row]
  float* c_l = c_m + kWarps * kRows;                             // [warp][row]
  {
    const int r0 = lane >> 2, r1 = r0 + 8, col = (lane & 3) << 1;
    float* ow = c_o + warp * kRows * DVT;
#pragma unroll
    for (int n = 0; n < DVT / 8; ++n) {
      ow[r0 * DVT + n * 8 + col] = o[n][0];
      ow[r0 * DVT + n * 8 + col + 1] = o[n][1];
      ow[r1 * DVT + n * 8 + col] = o[n][2];
      ow[r1 * DVT + n * 8 + col + 1] = o[n][3];
    }
    if ((lane & 3) == 0) {
      c_m[warp * kRows + r0] = m0;
      c_m[warp * kRows + r1] = m1;
      c_l[warp * kRows + r0] = l0;
      c_l[warp * kRows + r1] = l1;
    }
  }
  __syncthreads();
  for (int i = tid; i < it.nrows * DVT; i += kThreads) {
    const int r = i / DVT, col = i % DVT;
    float mm = -INFINITY;
#pragma unroll
    for (int w = 0; w < kWarps; ++w) mm = fmaxf(mm, c_m[w * kRows + r]);
    float acc = 0.f, lsum = 0.f;
    if (mm != -INFINITY) {
#pragma unroll
      for (int w = 0; w < kWarps; ++w) {
        float mw = c_m[w * kRows + r];
        float sc = mw == -INFINITY ? 0.f : fast_exp2(mw - mm);
        lsum += c_l[w * kRows + r] * sc;
        acc += c_o[(w * kRows + r) * DVT + col] * sc;
      }
    }
    const size_t row = (size_t)it.slot * p.hq + it.h0 + r;
    const int cc = it.dv0 + col;
    p.part_o[part_o_f4(it.slot, it.h0 + r, cc / 4, p.hq, p.dv) * 4 + cc % 4] =
        mm == -INFINITY ? 0.f : acc / lsum;
    if (col == 0 && it.dv0 == 0)
      p.part_lse[row] = mm == -INFINITY ? -INFINITY : (mm + log2f(lsum)) * kLn2;
  }
}

template <int DQK, int DVT, bool LATENT, int STAGES>
cudaError_t launch_variant(const SplitParams& p, int n_items, cudaStream_t stream) {
  constexpr int smem = split_smem_bytes<DQK, DVT, LATENT, STAGES>();
  auto kern = split_decode_kernel<DQK, DVT, LATENT, STAGES>;
  static thread_local int configured_device = -1;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (configured_device != dev) {
    e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    configured_device = dev;
  }
  kern<<<n_items, kThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

bool split_variant_supported(int dqk, int dv, bool latent) {
  if (!latent) return (dqk == 64 && dv == 64) || (dqk == 128 && dv == 128);
  return dqk == 576 && dv == 512;
}

int split_dv_tile(int dqk, int dv, bool latent) {
  (void)dqk;
  return latent ? 128 : dv;
}

cudaError_t launch_split_decode(const SplitParams& p, int n_items, bool latent,
                                cudaStream_t stream) {
  if (n_items == 0) return cudaSuccess;
  if (!latent && p.dqk == 64) return launch_variant<64, 64, false, 4>(p, n_items, stream);
  if (!latent && p.dqk == 128) return launch_variant<128, 128, false, 3>(p, n_items, stream);
  if (latent && p.dqk == 576) return launch_variant<576, 128, true, 2>(p, n_items, stream);
  return cudaErrorInvalidValue;
}

}  // namespace specgen
