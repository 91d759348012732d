// Grouped bf16 GEMM on the 5th-generation tensor cores (tcgen05, sm_103a)
// for the workers' dense layers (Eq. 4, "otherwise" branch: the forward and
// backward passes of x - lr * g(x)), with the step's elementwise work fused
// into the epilogue.
//
//   D[m][n] = sum_k A[m][k] * B[n][k]     A, B bf16 K-major, D fp32 in TMEM
//
// One CTA computes one 128 x BN tile of one active worker (grid z = worker).
// Warp 0 lane 0 streams K-blocks of 64 with TMA (128-byte swizzle, 3-D
// tensor maps whose z coordinate selects the worker's buffer or the
// parameter slot), warp 1 lane 0 issues tcgen05.mma (M=128, N=BN, K=16) into
// a TMEM accumulator and frees each stage with tcgen05.commit, warp 2 owns
// the TMEM allocation; then all four warps read their 32 TMEM lanes
// (one output row per thread) and run the epilogue:
//
//  kEpiFwd  hidden layer forward, m = output feature, n = sample:
//           h = relu(acc + bias[m]) -> bf16 H[n][m] and H^T[m][n].
//  kEpiDh   input gradient of a hidden layer, m = input feature, n = sample:
//           g = acc * (Hmask[n][m] > 0) -> bf16 G[n][m], G^T[m][n] and the
//           bias gradient gb[m] = sum_n g (fp32, whole batch in one tile).
//  kEpiDw   weight gradient + SGD, m = output feature, n = input feature:
//           W[dst] = fmaf(-lr, acc, W[src]) (fp32 master), bf16 shadow,
//           optional bf16 transposed shadow; column-tile 0 also updates the
//           bias b[dst] = fmaf(-lr, gb[m], b[src]).
//  kEpiStore plain C[m][n] = acc in fp32 (a library GEMM for tests and
//           callers that need one).
//
// All waits are bounded (see common.cuh) and report through a device word.
#include <cstdio>

#include "common.cuh"
#include "internal.h"

namespace oscars {

namespace {

constexpr int BM = 128;
constexpr int BK = 64;
constexpr int kABytes = BM * BK * 2;
constexpr int kBarrierBytes = 256;          // mbarriers + TMEM address slot
constexpr int kEpiTileFloats = 32 * 36;     // per-warp staging tile (row stride 36: conflict-free 16-byte accesses)

// Warps per CTA: the weight-gradient epilogue streams the fp32 master and
// runs two warpgroups (each warp owns its TMEM lane quarter, the two groups
// split the columns); the others use one warpgroup.
template <int EPI>
constexpr int warps_for() { return EPI == kEpiDw ? 8 : 4; }

template <int BN>
struct TileCfg {
  static constexpr int kBBytes = BN * BK * 2;
  static constexpr int kStageBytes = kABytes + kBBytes;
  static constexpr uint32_t kTmemCols = BN <= 32 ? 32 : BN <= 64 ? 64 : BN <= 128 ? 128 : 256;
};

template <int EPI>
__device__ __forceinline__ void epi_fwd(const GemmArgs& a, int wid, int src, int m, int n0,
                                        const float (&v)[32]) {
  const float bias = a.master[static_cast<int64_t>(src) * a.slot_stride + a.offB + m];
  __nv_bfloat16* out = a.out + static_cast<int64_t>(wid) * a.N * a.M;
  uint32_t pk[16];
#pragma unroll
  for (int c = 0; c < 32; c += 2) {
    const float h0 = fmaxf(v[c] + bias, 0.f);
    const float h1 = fmaxf(v[c + 1] + bias, 0.f);
    const __nv_bfloat162 p = __floats2bfloat162_rn(h0, h1);
    out[static_cast<int64_t>(n0 + c) * a.M + m] = p.x;
    out[static_cast<int64_t>(n0 + c + 1) * a.M + m] = p.y;
    pk[c >> 1] = *reinterpret_cast<const uint32_t*>(&p);
  }
  uint4* outT = reinterpret_cast<uint4*>(a.outT + (static_cast<int64_t>(wid) * a.M + m) * a.N + n0);
#pragma unroll
  for (int q = 0; q < 4; ++q) outT[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
}

// The input-gradient epilogue's ReLU mask for 32 columns: mk[c] = the raw
// bf16 bits of Hmask[n0 + c][m].  All 32 loads are issued before any is
// used, and the caller issues the next chunk's loads before it stores the
// current one, so the mask reads of a thread overlap instead of waiting
// one by one behind its stores.
__device__ __forceinline__ void epi_dh_mask(const GemmArgs& a, int wid, int m, int n0, unsigned short (&mk)[32]) {
  const unsigned short* hm = reinterpret_cast<const unsigned short*>(a.hmask) +
                             static_cast<int64_t>(wid) * a.N * a.M + static_cast<int64_t>(n0) * a.M + m;
#pragma unroll
  for (int c = 0; c < 32; ++c) mk[c] = __ldg(hm + static_cast<int64_t>(c) * a.M);
}

__device__ __forceinline__ float epi_dh(const GemmArgs& a, int wid, int m, int n0, const float (&v)[32],
                                        const unsigned short (&mk)[32]) {
  __nv_bfloat16* out = a.out ? a.out + static_cast<int64_t>(wid) * a.N * a.M : nullptr;
  uint32_t pk[16];
  float gsum = 0.f;
#pragma unroll
  for (int c = 0; c < 32; c += 2) {
    const int64_t e0 = static_cast<int64_t>(n0 + c) * a.M + m;
    const int64_t e1 = e0 + a.M;
    const float g0 = __bfloat162float(__ushort_as_bfloat16(mk[c])) > 0.f ? v[c] : 0.f;
    const float g1 = __bfloat162float(__ushort_as_bfloat16(mk[c + 1])) > 0.f ? v[c + 1] : 0.f;
    gsum += g0;
    gsum += g1;
    const __nv_bfloat162 p = __floats2bfloat162_rn(g0, g1);
    if (out) {   // the row-major copy only when a consumer reads it K-major
      out[e0] = p.x;
      out[e1] = p.y;
    }
    pk[c >> 1] = *reinterpret_cast<const uint32_t*>(&p);
  }
  uint4* outT = reinterpret_cast<uint4*>(a.outT + (static_cast<int64_t>(wid) * a.M + m) * a.N + n0);
#pragma unroll
  for (int q = 0; q < 4; ++q) outT[q] = make_uint4(pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
  return gsum;
}

// Weight gradient + SGD for one 32 x 32 block: rows m_base .. m_base + 31
// (thread `lane` holds row m_base + lane in v), columns n_base .. n_base + 31.
// `old` holds the block's fp32 master values in the column layout of the
// store pass: old[i] (i < 8) = 4 columns (n_base + 4 (lane % 8) ..) of row
// m_base + 4 i + lane / 8.  The accumulators go through a shared-memory tile
// (row stride 36: 16-byte accesses of 8 lanes hit distinct banks both along
// rows and along columns) so that the fp32 master and bf16 shadow writes move
// full lines, 4 rows per instruction.  (The persistent kernel of gemm_dw.cu
// serves every layer whose input count is a multiple of 8; this epilogue is
// the general fallback.)
__device__ __forceinline__ void epi_dw_block(const GemmArgs& a, int wid, int m_base, int n_base,
                                             const float (&v)[32], const float4 (&old)[8], float* T, int lane) {
#pragma unroll
  for (int q = 0; q < 8; ++q)
    *reinterpret_cast<float4*>(T + lane * 36 + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
  __syncwarp();
  const int cq = (lane & 7) * 4;
  const bool nok = n_base + cq < a.N;     // N % 8 == 0: a 4-column group is all in or all out
  const int64_t dof = static_cast<int64_t>(wid) * a.slot_stride + a.offW + n_base + cq;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = 4 * i + (lane >> 3);
    const float4 g = *reinterpret_cast<const float4*>(T + r * 36 + cq);
    float4 nw;
    nw.x = fmaf(-a.lr, g.x, old[i].x);
    nw.y = fmaf(-a.lr, g.y, old[i].y);
    nw.z = fmaf(-a.lr, g.z, old[i].z);
    nw.w = fmaf(-a.lr, g.w, old[i].w);
    if (nok) {
      const int64_t e = dof + static_cast<int64_t>(m_base + r) * a.N;
      *reinterpret_cast<float4*>(a.master_w + e) = nw;
      *reinterpret_cast<uint2*>(a.shadow + e) = make_uint2(pack_bf16x2(nw.x, nw.y), pack_bf16x2(nw.z, nw.w));
    }
  }
  __syncwarp();
}

// old[i] = master[src][m_base + 4 i + lane / 8][n_base + 4 (lane % 8) ..] as
// float4 (0 outside N): all 8 loads issued before any is used
__device__ __forceinline__ void epi_dw_load(const GemmArgs& a, int src, int m_base, int n_base, int lane,
                                            float4 (&old)[8]) {
  const int cq = (lane & 7) * 4;
  const bool nok = n_base + cq < a.N;
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride + a.offW + n_base + cq;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = 4 * i + (lane >> 3);
    old[i] = nok ? *reinterpret_cast<const float4*>(a.master + so + static_cast<int64_t>(m_base + r) * a.N)
                 : make_float4(0.f, 0.f, 0.f, 0.f);
  }
}

__device__ __forceinline__ void epi_store(const GemmArgs& a, int m, int n0, const float (&v)[32]) {
  float* c = a.c_out + static_cast<int64_t>(m) * a.N + n0;
  if (n0 + 32 <= a.N && (a.N & 3) == 0) {
    float4* c4 = reinterpret_cast<float4*>(c);
#pragma unroll
    for (int q = 0; q < 8; ++q) c4[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (n0 + j < a.N) c[j] = v[j];
  }
}

// Split-K (SPLIT > 1, forward and input-gradient epilogues): a cluster of
// SPLIT CTAs shares one output tile, CTA r multiplying K-blocks [r nk / SPLIT,
// (r + 1) nk / SPLIT).  Each CTA pushes its fp32 partial rows into the CTA
// that owns them (rows [r 128 / SPLIT, (r + 1) 128 / SPLIT) belong to CTA r)
// through distributed shared memory, one cluster barrier follows, and each
// owner sums the SPLIT partials in rank order and runs the epilogue on its
// rows.  Used when a launch has too few tiles to fill the GPU (the tail of a
// round, where one worker with many local steps runs alone).
constexpr int kRedLd = 4;   // padding of a partial row (floats)

__device__ __forceinline__ void st_dsmem_f32x4(float* local, uint32_t rank, float4 v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(remote), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w)
               : "memory");
}

template <int BN, int EPI, int SPLIT = 1>
__global__ void __launch_bounds__(warps_for<EPI>() * 32) gemm_tc_kernel(const __grid_constant__ CUtensorMap mapA,
                                                           const __grid_constant__ CUtensorMap mapB,
                                                           const __grid_constant__ GemmArgs a,
                                                           int stages) {
  static_assert(SPLIT == 1 || EPI == kEpiFwd || EPI == kEpiDh, "split-K serves the forward and input-gradient GEMMs");
  using Cfg = TileCfg<BN>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + stages * kABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sB + stages * Cfg::kBBytes);
  uint64_t* empty = full + stages;
  uint64_t* accum = empty + stages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  float* epi_tiles = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(full) + kBarrierBytes);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int li = blockIdx.z / SPLIT;
  const int rank = SPLIT > 1 ? static_cast<int>(cluster_ctarank()) : 0;
  const int wid = a.wid ? a.wid[li] : li, src = a.src ? a.src[li] : li;
  const int m0 = blockIdx.x * BM, n0 = blockIdx.y * BN;
  const int nk_all = (a.K + BK - 1) / BK;
  const int kb0 = rank * nk_all / SPLIT;                 // this CTA's K-blocks [kb0, kb0 + nk)
  const int nk = (rank + 1) * nk_all / SPLIT - kb0;

  if (threadIdx.x == 0) {
    prefetch_tmap(&mapA);
    prefetch_tmap(&mapB);
    for (int s = 0; s < stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, Cfg::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_wait();      // the previous kernel's outputs (operands, masks, biases) are complete
  pdl_trigger();

  if (warp == 0 && lane == 0) {
    // TMA producer
    const int za = a.a_z_src ? src : wid;
    const int zb = a.b_z_src ? src : wid;
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % stages;
      if (kb >= stages && !mbar_wait(&empty[s], ((kb / stages) + 1) & 1, a.err, kDevTimeoutEmpty)) break;
      mbar_arrive_expect_tx(&full[s], kABytes + Cfg::kBBytes);
      const int k = (kb0 + kb) * BK;   // global K coordinate
      if constexpr (EPI == kEpiDh) {
        // A = W^T read MN-major from W [K = out][M = in]: two boxes of 64 M x
        // 64 K, the second 64 M-elements further along (8 KB in shared memory)
        tma_load_3d(sA + s * kABytes, &mapA, m0, k, za, &full[s]);
        tma_load_3d(sA + s * kABytes + kABytes / 2, &mapA, m0 + 64, k, za, &full[s]);
      } else {
        tma_load_3d(sA + s * kABytes, &mapA, k, m0, za, &full[s]);
      }
      if (EPI == kEpiDh && a.b_mn) {
        // B = G read MN-major from G^T [K = out][N = batch]: boxes of 64 N x 64 K, 8 KB apart
        for (int nb = 0; nb < BN / 64; ++nb)
          tma_load_3d(sB + s * Cfg::kBBytes + nb * 8192, &mapB, n0 + 64 * nb, k, zb, &full[s]);
      } else {
        tma_load_3d(sB + s * Cfg::kBBytes, &mapB, k, n0, zb, &full[s]);
      }
    }
  } else if (warp == 1 && lane == 0) {
    // MMA issuer
    // A MN-major (transpose-A bit 15) for the input gradient, K-major otherwise;
    // B MN-major (bit 16) when the input gradient reads G^T
    const bool bmn = EPI == kEpiDh && a.b_mn;
    const uint32_t idesc = idesc_bf16_f32(BM, BN) | (EPI == kEpiDh ? (1u << 15) : 0u) | (bmn ? (1u << 16) : 0u);
    for (int kb = 0; kb < nk; ++kb) {
      const int s = kb % stages;
      if (!mbar_wait(&full[s], (kb / stages) & 1, a.err, kDevTimeoutFull)) break;
      tc_fence_after();
      const uint32_t a_base = smem_u32(sA + s * kABytes);
      const uint32_t b_base = smem_u32(sB + s * Cfg::kBBytes);
#pragma unroll
      for (int j = 0; j < BK / 16; ++j) {
        // K-major: 16 K-elements are 32 bytes along a row; MN-major: 16 rows of 128 bytes
        const uint64_t adesc = EPI == kEpiDh ? smem_desc_mn128(a_base + j * 2048, kABytes / 2)
                                             : smem_desc_k128(a_base + j * 32);
        const uint64_t bdesc = bmn ? smem_desc_mn128(b_base + j * 2048, 8192) : smem_desc_k128(b_base + j * 32);
        umma_bf16(tmem, adesc, bdesc, idesc, (kb | j) != 0 ? 1u : 0u);
      }
      umma_commit(&empty[s]);
    }
    umma_commit(accum);  // arrives once every issued MMA has completed
  }
  __syncwarp();

  if constexpr (SPLIT > 1) {
    // ---- split-K epilogue (4 warps): push the partial rows to their owners
    constexpr int R = BM / SPLIT;                   // rows owned per CTA
    constexpr int ld = BN + kRedLd;
    float* red = epi_tiles;                         // [SPLIT][R][ld] fp32: the partials of this CTA's rows
    int acc_ok = mbar_wait(accum, 0, a.err, kDevTimeoutAccum) ? 1 : 0;
    acc_ok = __all_sync(0xffffffffu, acc_ok);
    tc_fence_after();
    const int row = (warp & 3) * 32 + lane;        // accumulator row of this thread
    const int owner = row / R;
    float* dst = red + (rank * R + (row - owner * R)) * ld;
    const uint32_t trow = tmem + (static_cast<uint32_t>((warp & 3) * 32) << 16);
#pragma unroll 1
    for (int c0 = 0; c0 < BN; c0 += 32) {
      float v[32];
      if (acc_ok) tmem_ld_32x32b_x32(trow + c0, v);
      else
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = 0.f;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float4 p4 = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        if (owner == rank) *reinterpret_cast<float4*>(dst + c0 + 4 * q) = p4;
        else st_dsmem_f32x4(dst + c0 + 4 * q, owner, p4);
      }
    }
    tc_fence_before();
    cluster_sync();   // every partial has landed in its owner
    // own rows: item = (row, 32-column chunk); partials summed in rank order
    float* gpart = red + SPLIT * R * ld;            // [R][BN / 32] bias-gradient partials (input gradient)
    for (int it = threadIdx.x; it < R * (BN / 32); it += warps_for<EPI>() * 32) {
      const int rl = it / (BN / 32), c0 = (it % (BN / 32)) * 32;
      float v[32];
#pragma unroll
      for (int j = 0; j < 32; ++j) v[j] = 0.f;
#pragma unroll
      for (int p = 0; p < SPLIT; ++p) {
        const float* src_row = red + (p * R + rl) * ld + c0;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 x = *reinterpret_cast<const float4*>(src_row + 4 * q);
          v[4 * q] += x.x;
          v[4 * q + 1] += x.y;
          v[4 * q + 2] += x.z;
          v[4 * q + 3] += x.w;
        }
      }
      const int m = m0 + rank * R + rl;
      if constexpr (EPI == kEpiFwd) {
        epi_fwd<EPI>(a, wid, src, m, n0 + c0, v);
      } else {
        unsigned short mk[32];
        epi_dh_mask(a, wid, m, n0 + c0, mk);
        gpart[rl * (BN / 32) + c0 / 32] = epi_dh(a, wid, m, n0 + c0, v, mk);
      }
    }
    if constexpr (EPI == kEpiDh) {
      __syncthreads();
      for (int rl = threadIdx.x; rl < R; rl += warps_for<EPI>() * 32) {
        float g = 0.f;
        for (int c = 0; c < BN / 32; ++c) g += gpart[rl * (BN / 32) + c];
        a.gb_out[static_cast<int64_t>(wid) * a.M + m0 + rank * R + rl] = g;
      }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 2) {
      tc_fence_after();
      tmem_dealloc(tmem, Cfg::kTmemCols);
    }
    return;
  }

  // epilogue: thread = one accumulator row
  unsigned short mk[32];   // input-gradient mask of the next 32 columns, read while the MMAs run
  if constexpr (EPI == kEpiDh) epi_dh_mask(a, wid, m0 + (warp & 3) * 32 + lane, n0, mk);
  float4 old0[8], old1[8];  // weight-gradient epilogue: the fp32 master block, read while the MMAs run
  if constexpr (EPI == kEpiDw) {
    const int c_begin = (warp >> 2) * (BN / 2);
    const int mb = m0 + (warp & 3) * 32;
    epi_dw_load(a, src, mb, n0 + c_begin, lane, old0);
    epi_dw_load(a, src, mb, n0 + c_begin + 32, lane, old1);
  }
  int acc_ok = mbar_wait(accum, 0, a.err, kDevTimeoutAccum) ? 1 : 0;
  acc_ok = __all_sync(0xffffffffu, acc_ok);
  tc_fence_after();
  if (acc_ok) {
    const int quarter = warp & 3;
    const int m = m0 + quarter * 32 + lane;
    const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    if constexpr (EPI == kEpiDw) {
      static_assert(BN == 128, "the weight-gradient epilogue covers 2 x 32 columns per warp");
      const int c_begin = (warp >> 2) * (BN / 2);
      const int mb = m0 + quarter * 32;
      float* T = epi_tiles + warp * kEpiTileFloats;
      if (n0 + c_begin < a.N) {
        float v[32];
        tmem_ld_32x32b_x32(trow + c_begin, v);
        epi_dw_block(a, wid, mb, n0 + c_begin, v, old0, T, lane);
      }
      if (n0 + c_begin + 32 < a.N) {
        float v[32];
        tmem_ld_32x32b_x32(trow + c_begin + 32, v);
        epi_dw_block(a, wid, mb, n0 + c_begin + 32, v, old1, T, lane);
      }
      if (warp < 4 && blockIdx.y == 0) {
        const int64_t bo = a.offB + m;
        a.master_w[static_cast<int64_t>(wid) * a.slot_stride + bo] =
            fmaf(-a.lr, a.gb_in[static_cast<int64_t>(wid) * a.M + m], a.master[static_cast<int64_t>(src) * a.slot_stride + bo]);
      }
    } else if constexpr (EPI == kEpiDh) {
      float gsum = 0.f;
#pragma unroll
      for (int c0 = 0; c0 < BN; c0 += 32) {
        float v[32];
        tmem_ld_32x32b_x32(trow + c0, v);
        unsigned short cur[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) cur[c] = mk[c];
        if (c0 + 32 < BN) epi_dh_mask(a, wid, m, n0 + c0 + 32, mk);
        gsum += epi_dh(a, wid, m, n0 + c0, v, cur);
      }
      a.gb_out[static_cast<int64_t>(wid) * a.M + m] = gsum;
    } else {
#pragma unroll 1
      for (int c0 = 0; c0 < BN; c0 += 32) {
        float v[32];
        tmem_ld_32x32b_x32(trow + c0, v);
        if (EPI == kEpiFwd) {
          epi_fwd<EPI>(a, wid, src, m, n0 + c0, v);
        } else if (EPI == kEpiStore) {
          if (n0 + c0 < a.N) epi_store(a, m, n0 + c0, v);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

// Shared memory that keeps the number of resident CTAs per SM at or below
// 512 / (TMEM columns per CTA), so a tcgen05.alloc never has to wait.
size_t smem_floor_for_tmem(uint32_t cols) {
  const size_t per_sm = 233472;  // 228 KB
  const size_t max_ctas = 512 / cols;
  return per_sm / (max_ctas + 1) - 1024 + 16;
}

int device_sms() {
  static int sms = 0;
  if (sms == 0) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms < 1) sms = 1;
  }
  return sms;
}

template <int BN, int EPI, int SPLIT = 1>
cudaError_t launch_tile(const CUtensorMap& mA, const CUtensorMap& mB, const GemmArgs& a, int n_active,
                        cudaStream_t s) {
  using Cfg = TileCfg<BN>;
  const int nk = ((a.K + BK - 1) / BK + SPLIT - 1) / SPLIT;   // K-blocks of the CTA with the most
  dim3 grid(a.M / BM, (a.N + BN - 1) / BN, n_active * SPLIT);
  // A grid that fits one CTA per SM gets as many stages as K-blocks, within
  // ~200 KB of shared memory: the whole K extent of these skinny GEMMs is
  // then in flight at once.  A larger grid gets stages for ~100 KB, so two
  // CTAs share each SM and the grid runs in one wave instead of two (the
  // bytes in flight per SM stay the same).  A split grid keeps room for the
  // partial rows its CTAs exchange.
  const int sms = device_sms();
  const long long ctas = static_cast<long long>(grid.x) * grid.y * grid.z;
  const size_t red_bytes = SPLIT > 1 ? sizeof(float) * (static_cast<size_t>(BM) * (BN + kRedLd) + BM / SPLIT * (BN / 32))
                                     : 0;
  const int budget = SPLIT > 1 ? 150 * 1024 : ctas > sms ? 100 * 1024 : 200 * 1024;
  const int max_stages = static_cast<int>((budget - (EPI == kEpiDw ? 8 * 32 * 33 * 4 : 0)) / Cfg::kStageBytes);
  int stages = nk < max_stages ? nk : (max_stages < 8 ? max_stages : 8);
  if (stages < 2) stages = nk < 2 ? nk : 2;
  constexpr int kWarps = warps_for<EPI>();
  size_t smem = 1024 + static_cast<size_t>(stages) * Cfg::kStageBytes + kBarrierBytes +
                (EPI == kEpiDw ? sizeof(float) * kWarps * kEpiTileFloats : 0) + red_bytes;
  const size_t floor_b = smem_floor_for_tmem(Cfg::kTmemCols);
  if (smem < floor_b) smem = floor_b;
  cudaError_t e = cudaFuncSetAttribute(gemm_tc_kernel<BN, EPI, SPLIT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kWarps * 32, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  int n = 0;
  if (SPLIT > 1) {
    attr[n].id = cudaLaunchAttributeClusterDimension;
    attr[n].val.clusterDim.x = 1;
    attr[n].val.clusterDim.y = 1;
    attr[n].val.clusterDim.z = SPLIT;
    ++n;
  }
  if (a.pdl) {
    attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[n].val.programmaticStreamSerializationAllowed = 1;
    ++n;
  }
  cfg.attrs = attr;
  cfg.numAttrs = n;
  return cudaLaunchKernelEx(&cfg, gemm_tc_kernel<BN, EPI, SPLIT>, mA, mB, a, stages);
}

// K split of a forward or input-gradient launch: 4 or 2 CTAs per tile when
// the unsplit grid would leave most of the GPU idle and each CTA keeps at
// least 4 K-blocks
int split_for(int M, int N, int BN, int K, int n_active) {
  const long long tiles = static_cast<long long>(M / BM) * ((N + BN - 1) / BN) * n_active;
  const int nk = (K + BK - 1) / BK;
  const int sms = device_sms();
  if (tiles * 4 <= sms && nk >= 16) return 4;
  if (tiles * 2 <= sms && nk >= 8) return 2;
  return 1;
}

}  // namespace

int gemm_bn_for(int epi, int N) {
  if (epi == kEpiDw || epi == kEpiStore) return 128;
  return N;  // forward / input gradient: the whole batch in one tile
}

cudaError_t launch_gemm(int epi, const CUtensorMap& mA, const CUtensorMap& mB, const GemmArgs& a,
                        int n_active, cudaStream_t s) {
  if (a.M % BM != 0) return cudaErrorInvalidValue;
  if (epi == kEpiDw) return launch_tile<128, kEpiDw>(mA, mB, a, n_active, s);
  if (epi == kEpiStore) return launch_tile<128, kEpiStore>(mA, mB, a, n_active, s);
  const int bn = gemm_bn_for(epi, a.N);
  const int split = bn == 128 ? split_for(a.M, a.N, bn, a.K, n_active) : 1;
  if (epi == kEpiFwd) {
    if (split == 4) return launch_tile<128, kEpiFwd, 4>(mA, mB, a, n_active, s);
    if (split == 2) return launch_tile<128, kEpiFwd, 2>(mA, mB, a, n_active, s);
    switch (bn) {
      case 32: return launch_tile<32, kEpiFwd>(mA, mB, a, n_active, s);
      case 64: return launch_tile<64, kEpiFwd>(mA, mB, a, n_active, s);
      case 128: return launch_tile<128, kEpiFwd>(mA, mB, a, n_active, s);
      case 256: return launch_tile<256, kEpiFwd>(mA, mB, a, n_active, s);
      default: return cudaErrorInvalidValue;
    }
  }
  if (split == 4) return launch_tile<128, kEpiDh, 4>(mA, mB, a, n_active, s);
  if (split == 2) return launch_tile<128, kEpiDh, 2>(mA, mB, a, n_active, s);
  switch (bn) {
    case 32: return launch_tile<32, kEpiDh>(mA, mB, a, n_active, s);
    case 64: return launch_tile<64, kEpiDh>(mA, mB, a, n_active, s);
    case 128: return launch_tile<128, kEpiDh>(mA, mB, a, n_active, s);
    case 256: return launch_tile<256, kEpiDh>(mA, mB, a, n_active, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace oscars
