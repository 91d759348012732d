// A whole round of local steps of a two-layer bf16 MLP (input -> H hidden
// ReLU units -> 10 classes) in ONE launch (Eq. 4, "otherwise" branch: each
// worker runs tau_i SGD steps from the global model).
//
// One thread-block cluster serves one worker; its H/128 CTAs split the
// hidden units, CTA r owning units [128 r, 128 r + 128).  Every step of the
// worker runs inside the cluster:
//
//  F  forward of the hidden layer for the CTA's units:
//     z[o][b] = sum_k W0[o][k] X[b][k] on tcgen05 (TMA-fed, TMEM accumulator),
//     h = relu(z + b0[o]) kept as bf16 in shared memory;
//  H  last layer: partial logits over the CTA's units, summed over the
//     cluster in rank order through distributed shared memory, softmax
//     cross-entropy; the masked input gradient dz0[b][o] of the CTA's units is
//     written straight into a 128-byte-swizzled K-major shared-memory tile
//     (the A operand of step D); bias gradient and SGD of b0 (own units), of
//     the head weights (own columns) and, on rank 0, of the head bias;
//  D  weight gradient of the hidden layer, dW0[o][k] = sum_b dz0[b][o] X[b][k]
//     on tcgen05 (X^T tiles by TMA, two TMEM buffers so the MMA of one tile
//     overlaps the epilogue of the previous), with the SGD update of W0 rows
//     fused in the epilogue (fp32 master read-modify-write and bf16 shadow,
//     both through a padded staging tile so every global access is a full
//     line).
//
// A CTA only ever rewrites the W0 rows, b0 entries and head-weight columns it
// owns, so the next step reads its own writes; the head bias, written by rank
// 0, is ordered by the cluster barriers.  Generic-proxy writes that TMA or
// the tensor core read afterwards are fenced with fence.proxy.async.
// Arithmetic and rounding points are those of the multi-kernel path.
//
// Warp roles (384 threads): warp 0 lane 0 issues TMA, warp 1 lane 0 issues
// tcgen05.mma, warp 2 owns the TMEM allocation (all 512 columns: one CTA per
// SM), warps 4..11 read TMEM in the epilogues (two warpgroups, each covering
// the 128 accumulator lanes), all warps share the CUDA-core work of step H.
#include "common.cuh"
#include "internal.h"

namespace oscars {
namespace {

constexpr int kFT = 384;               // threads
constexpr int kFU = 128;               // hidden units per CTA
constexpr int kFC = 10;                // classes
constexpr int kFMaxCluster = 8;
constexpr int kFBK = 64;               // K-block (bf16 elements, 128 bytes)

__device__ __forceinline__ void tma_load_4d(void* smem_dst, const CUtensorMap* map, int c0, int c1, int c2, int c3,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

// Per-batch-size configuration (all sizes known at compile time).
template <int B>
struct FCfg {
  static constexpr int kStagesF = 4;
  static constexpr int kABytes = kFU * kFBK * 2;            // W0 tile: 128 rows x 64 k
  static constexpr int kBBytes = B * kFBK * 2;              // X tile: B rows x 64 k
  static constexpr int kND = 32;                            // columns (input features) per weight-gradient tile
  static constexpr int kNBD = 4;                            // weight-gradient buffers in flight
  static constexpr int kKB = (B + kFBK - 1) / kFBK;         // K-blocks of the weight gradient (K = batch)
  static constexpr int kXtBytes = kND * kFBK * 2 * kKB;     // one X^T tile (all K-blocks)
  static constexpr int kMsBytes = kFU * kND * 4;            // fp32 master tile: 128 rows x kND columns
  static constexpr int kBufD = kXtBytes + kMsBytes;
  static constexpr int kPipe = kStagesF * (kABytes + kBBytes);
  static constexpr int kPipeD = kNBD * kBufD;
  static constexpr int kRegion = kPipe > kPipeD ? kPipe : kPipeD;   // TMA area, reused by both steps
  static constexpr int kDzT = kFU * 128 * kKB;              // dz0^T tile: 128 rows x (64 k per block)
  static constexpr int kTpr = 256 / B;                      // threads per row, partial logits (256 threads)
  static constexpr int kHsd = kFU + 4 * kTpr;               // padded row stride of the float h tile
  // shared memory carve-up (bytes, from a 1024-aligned base)
  static constexpr int oRegion = 0;
  static constexpr int oDzT = oRegion + kRegion;
  static constexpr int oHs = oDzT + kDzT;                    // [B][kHsd] float
  static constexpr int oWc = oHs + B * kHsd * 4;             // [C][128] float
  static constexpr int oPl = oWc + kFC * kFU * 4;            // [B][C] float
  static constexpr int oDz = oPl + B * kFC * 4;              // [B][C] float
  static constexpr int oDzb = oDz + B * kFC * 4;             // [B][C] float
  static constexpr int oGbp = oDzb + B * kFC * 4;            // [8][128] float
  static constexpr int oRowLoss = oGbp + 8 * kFU * 4;        // [B] float
  static constexpr int oPre = (oRowLoss + B * 4 + 15) / 16 * 16;   // H inputs prefetched during F:
  static constexpr int kPreFloats = kFC * kFU + kFU + 16 + B;       //   W1 master cols, b0, b1, labels
  static constexpr int oEpi = (oPre + kPreFloats * 4 + 15) / 16 * 16;   // 8 x [32][36] float staging tiles
  static constexpr int oBar = oEpi + 8 * 32 * 36 * 4;
  static constexpr int kBarBytes = 256;
  static constexpr int kSmem = oBar + kBarBytes + 1024;      // + alignment slack
};

struct FusedArgs {
  const int32_t* tau;       // [W]
  int W, D, H;
  int global_slot;
  float lr;
  const float* master;
  float* master_w;
  __nv_bfloat16* shadow;
  int64_t slot_stride;
  int64_t offW0, offB0, offW1, offB1;
  const int32_t* labels;    // [max_tau][W][B]
  float* loss_part;         // [(w * max_tau + s) * (B / 16) + chunk]
  int max_tau;
  int* err;
  unsigned long long* phase_ts;   // [max_tau][4] phase start stamps of worker 0 (or null)
};

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long v;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(v));
  return v;
}

// byte offset of element (row, k) in a K-major 128-byte-swizzled tile of
// `rows` rows per 64-wide K-block (the layout TMA writes and UMMA reads)
__device__ __forceinline__ uint32_t sw128_offset(int row, int k, int rows) {
  const int kb = k >> 6, kk = k & 63;
  return static_cast<uint32_t>(kb * rows * 128 + (row >> 3) * 1024 + (row & 7) * 128 +
                               ((((kk >> 3) ^ (row & 7)) & 7) << 4) + (kk & 7) * 2);
}

template <int B>
__global__ void __launch_bounds__(kFT, 1) fused_mlp2_round_kernel(const __grid_constant__ CUtensorMap mW0,
                                                                 const __grid_constant__ CUtensorMap mX,
                                                                 const __grid_constant__ CUtensorMap mXT,
                                                                 const __grid_constant__ CUtensorMap mWm,
                                                                 const __grid_constant__ FusedArgs a) {
  using Cfg = FCfg<B>;
  extern __shared__ uint8_t fs_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(fs_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* region = sm + Cfg::oRegion;
  uint8_t* dzT = sm + Cfg::oDzT;
  float* hs = reinterpret_cast<float*>(sm + Cfg::oHs);
  float* wcs = reinterpret_cast<float*>(sm + Cfg::oWc);
  float* pl = reinterpret_cast<float*>(sm + Cfg::oPl);
  float* dz = reinterpret_cast<float*>(sm + Cfg::oDz);
  float* dzb = reinterpret_cast<float*>(sm + Cfg::oDzb);
  float* gbp = reinterpret_cast<float*>(sm + Cfg::oGbp);
  float* rowloss = reinterpret_cast<float*>(sm + Cfg::oRowLoss);
  float* epi = reinterpret_cast<float*>(sm + Cfg::oEpi);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::oBar);
  uint64_t* fullF = bars;                      // [kStagesF]
  uint64_t* emptyF = fullF + Cfg::kStagesF;    // [kStagesF]
  uint64_t* accF = emptyF + Cfg::kStagesF;     // [1]
  uint64_t* fullD = accF + 1;                  // [kNBD] X^T + master tile landed
  uint64_t* accD = fullD + Cfg::kNBD;          // [kNBD] TMEM buffer full
  uint64_t* tfreeD = accD + Cfg::kNBD;         // [kNBD] TMEM + shared buffer drained (128 arrivals)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tfreeD + Cfg::kNBD);
  float* pre = reinterpret_cast<float*>(sm + Cfg::oPre);
  float* w1m = pre;                            // [C][128] fp32 master W1 columns (src)
  float* b0m = w1m + kFC * kFU;                // [128] fp32 b0 of own units (src)
  float* b1m = b0m + kFU;                      // [16] fp32 b1 (src)
  int* labs = reinterpret_cast<int*>(b1m + 16);   // [B] labels of this step

  const int w = blockIdx.x;
  const int rank = static_cast<int>(cluster_ctarank());
  const int ncl = static_cast<int>(gridDim.y);
  const int u0 = rank * kFU;                    // first hidden unit of this CTA
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int D = a.D, H = a.H;
  const int tau = a.tau[w];
  const int nkF = (D + kFBK - 1) / kFBK;
  const int nD = (D + Cfg::kND - 1) / Cfg::kND;

  if (t == 0) {
    prefetch_tmap(&mW0);
    prefetch_tmap(&mX);
    prefetch_tmap(&mXT);
    prefetch_tmap(&mWm);
    for (int i = 0; i < Cfg::kStagesF; ++i) {
      mbar_init(&fullF[i], 1);
      mbar_init(&emptyF[i], 1);
    }
    mbar_init(accF, 1);
    for (int i = 0; i < Cfg::kNBD; ++i) {
      mbar_init(&fullD[i], 1);
      mbar_init(&accD[i], 1);
      mbar_init(&tfreeD[i], 128);
    }
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  // zero the dz0^T tile once: for B < 64 its K padding must stay zero
  for (int i = t; i < Cfg::kDzT / 16; i += kFT) reinterpret_cast<uint4*>(dzT)[i] = make_uint4(0, 0, 0, 0);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  int kcount = 0;   // F K-blocks issued so far (ring position)
  int dcount = 0;   // D tiles so far (TMEM / X^T double buffer position)

  const bool stamp = a.phase_ts && w == 0 && rank == 0 && t == 0;
  for (int s = 0; s < tau; ++s) {
    if (stamp) a.phase_ts[s * 4 + 0] = global_ns();
    const int src = s == 0 ? a.global_slot : w;
    const int64_t so = static_cast<int64_t>(src) * a.slot_stride;
    const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;

    // ------------------------------------------------------------ F: forward of the hidden layer
    if (warp == 0 && lane == 0) {
      fence_proxy_async_global();     // this CTA's generic writes of W0 rows precede these TMA reads
      for (int kb = 0; kb < nkF; ++kb) {
        const int c = kcount + kb, st = c % Cfg::kStagesF;
        if (c >= Cfg::kStagesF && !mbar_wait(&emptyF[st], ((c / Cfg::kStagesF) + 1) & 1, a.err, kDevTimeoutEmpty)) break;
        mbar_arrive_expect_tx(&fullF[st], Cfg::kABytes + Cfg::kBBytes);
        uint8_t* sa = region + st * (Cfg::kABytes + Cfg::kBBytes);
        tma_load_3d(sa, &mW0, kb * kFBK, u0, src, &fullF[st]);
        tma_load_4d(sa + Cfg::kABytes, &mX, kb * kFBK, 0, w, s, &fullF[st]);
      }
    } else if (warp == 1 && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, B);
      for (int kb = 0; kb < nkF; ++kb) {
        const int c = kcount + kb, st = c % Cfg::kStagesF;
        if (!mbar_wait(&fullF[st], (c / Cfg::kStagesF) & 1, a.err, kDevTimeoutFull)) break;
        tc_fence_after();
        const uint32_t sa = smem_u32(region + st * (Cfg::kABytes + Cfg::kBBytes));
#pragma unroll
        for (int j = 0; j < kFBK / 16; ++j)
          umma_bf16(tmem, smem_desc_k128(sa + j * 32), smem_desc_k128(sa + Cfg::kABytes + j * 32), idesc,
                    (kb | j) != 0 ? 1u : 0u);
        umma_commit(&emptyF[st]);
      }
      umma_commit(accF);
    }
    kcount += nkF;
    // every global input of step H, fetched while the tensor core runs F:
    // head weights of this CTA's columns (bf16 operand and fp32 master), b0 of
    // its units, the head bias and this step's labels
    for (int q = t; q < kFC * (kFU / 8); q += kFT) {
      const int c = q / (kFU / 8), c8 = (q % (kFU / 8)) * 8;
      const int64_t e = a.offW1 + static_cast<int64_t>(c) * H + u0 + c8;
      const uint4 v = *reinterpret_cast<const uint4*>(a.shadow + so + e);
      const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(p2[j]);
        wcs[c * kFU + c8 + 2 * j] = f.x;
        wcs[c * kFU + c8 + 2 * j + 1] = f.y;
      }
      *reinterpret_cast<float4*>(w1m + c * kFU + c8) = *reinterpret_cast<const float4*>(a.master + so + e);
      *reinterpret_cast<float4*>(w1m + c * kFU + c8 + 4) = *reinterpret_cast<const float4*>(a.master + so + e + 4);
    }
    if (t < kFU) b0m[t] = a.master[so + a.offB0 + u0 + t];
    if (t < kFC) b1m[t] = a.master[so + a.offB1 + t];
    for (int b = t; b < B; b += kFT) labs[b] = a.labels[(static_cast<int64_t>(s) * a.W + w) * B + b];
    __syncthreads();   // the prefetched b0 is read by the F epilogue below
    if (warp >= 4) {   // epilogue F: thread = hidden unit, columns = samples
      int ok = mbar_wait(accF, s & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
      ok = __all_sync(0xffffffffu, ok);
      tc_fence_after();
      if (ok) {
        const int quarter = warp & 3, grp = (warp - 4) >> 2;
        const int ul = quarter * 32 + lane;              // local unit
        const float bias = b0m[ul];
        const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        for (int c0 = grp * 32; c0 < B; c0 += 64) {
          float v[32];
          tmem_ld_32x32b_x32(trow + c0, v);
#pragma unroll
          for (int j = 0; j < 32; ++j) hs[(c0 + j) * Cfg::kHsd + ul] = bf16_round(fmaxf(v[j] + bias, 0.f));
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    if (stamp) a.phase_ts[s * 4 + 1] = global_ns();

    // ------------------------------------------------------------ H: last layer
    if (t < 256) {   // partial logits: kTpr threads per row, all classes in registers
      const int rb = t / Cfg::kTpr, q = t % Cfg::kTpr;
      float acc[kFC];
#pragma unroll
      for (int c = 0; c < kFC; ++c) acc[c] = 0.f;
      for (int k = 4 * q; k < kFU; k += 4 * Cfg::kTpr) {
        const float4 hv = *reinterpret_cast<const float4*>(hs + rb * Cfg::kHsd + k);
#pragma unroll
        for (int c = 0; c < kFC; ++c) {
          const float4 wv = *reinterpret_cast<const float4*>(wcs + c * kFU + k);
          acc[c] = fmaf(hv.x, wv.x, acc[c]);
          acc[c] = fmaf(hv.y, wv.y, acc[c]);
          acc[c] = fmaf(hv.z, wv.z, acc[c]);
          acc[c] = fmaf(hv.w, wv.w, acc[c]);
        }
      }
#pragma unroll
      for (int c = 0; c < kFC; ++c) {
        for (int o = Cfg::kTpr / 2; o > 0; o >>= 1) acc[c] += __shfl_xor_sync(0xffffffffu, acc[c], o);
        if (q == 0) pl[rb * kFC + c] = acc[c];
      }
    }
    cluster_sync();
    for (int q = t; q < B * kFC; q += kFT) {
      float part[kFMaxCluster];
#pragma unroll
      for (int r = 0; r < kFMaxCluster; ++r) part[r] = r < ncl ? ld_dsmem_f32(pl + q, r) : 0.f;
      float acc = 0.f;
#pragma unroll
      for (int r = 0; r < kFMaxCluster; ++r)
        if (r < ncl) acc += part[r];
      dz[q] = acc + b1m[q % kFC];
    }
    cluster_sync();   // all remote reads of pl and all reads of the head bias are done
    for (int b = t; b < B; b += kFT) {
      float z[kFC], e[kFC];
#pragma unroll
      for (int c = 0; c < kFC; ++c) z[c] = dz[b * kFC + c];
      float m = z[0];
#pragma unroll
      for (int c = 1; c < kFC; ++c) m = fmaxf(m, z[c]);
      const int y = labs[b];
      float se = 0.f, so_ = 0.f, zy = 0.f;
#pragma unroll
      for (int c = 0; c < kFC; ++c) {
        e[c] = expf(z[c] - m);
        se += e[c];
        if (c != y) so_ += e[c];
        else zy = z[c];
      }
      rowloss[b] = m + logf(se) - zy;
      const float inv = 1.0f / static_cast<float>(B);
#pragma unroll
      for (int c = 0; c < kFC; ++c) {
        const float g = (c == y ? -(so_ / se) : e[c] / se) * inv;
        dz[b * kFC + c] = g;
        dzb[b * kFC + c] = bf16_round(g);
      }
    }
    __syncthreads();
    if (rank == 0) {
      if (t < B / kRowsPerLossChunk) {
        float l = 0.f;
        for (int r = 0; r < kRowsPerLossChunk; ++r) l += rowloss[t * kRowsPerLossChunk + r];
        a.loss_part[(static_cast<int64_t>(w) * a.max_tau + s) * (B / kRowsPerLossChunk) + t] = l;
      }
      if (t < kFC * 16) {   // head bias
        const int c = t >> 4, j = t & 15;
        float g = 0.f;
        for (int b = j; b < B; b += 16) g += dz[b * kFC + c];
#pragma unroll
        for (int o = 8; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o, 16);
        if (j == 0) a.master_w[dof + a.offB1 + c] = fmaf(-a.lr, g, b1m[c]);
      }
    }
    // masked input gradient dz0[b][u] of this CTA's units: item = (row, 4 units);
    // 8 warps x 32 lanes x 4 units (warps 8..11 help with the head weight gradient)
    if (t < 256) {
      const int u4 = (t & 31) * 4, wg = t >> 5;
      float4 wc[kFC];
#pragma unroll
      for (int c = 0; c < kFC; ++c) wc[c] = *reinterpret_cast<const float4*>(wcs + c * kFU + u4);
      float4 gs = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int b = wg; b < B; b += 8) {
        const float4 hv = *reinterpret_cast<const float4*>(hs + b * Cfg::kHsd + u4);
        float4 dh = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int c = 0; c < kFC; ++c) {
          const float g = dzb[b * kFC + c];
          dh.x = fmaf(g, wc[c].x, dh.x);
          dh.y = fmaf(g, wc[c].y, dh.y);
          dh.z = fmaf(g, wc[c].z, dh.z);
          dh.w = fmaf(g, wc[c].w, dh.w);
        }
        dh.x = hv.x > 0.f ? dh.x : 0.f;
        dh.y = hv.y > 0.f ? dh.y : 0.f;
        dh.z = hv.z > 0.f ? dh.z : 0.f;
        dh.w = hv.w > 0.f ? dh.w : 0.f;
        gs.x += dh.x;
        gs.y += dh.y;
        gs.z += dh.z;
        gs.w += dh.w;
        const float dv[4] = {dh.x, dh.y, dh.z, dh.w};
#pragma unroll
        for (int j = 0; j < 4; ++j)
          *reinterpret_cast<__nv_bfloat16*>(dzT + sw128_offset(u4 + j, b, kFU)) = __float2bfloat16_rn(dv[j]);
      }
      *reinterpret_cast<float4*>(gbp + wg * kFU + u4) = gs;
    }
    fence_proxy_async_smem();   // dz0^T is read by the tensor core next
    __syncthreads();
    if (t < kFU) {   // b0 of this CTA's units
      float g = 0.f;
#pragma unroll
      for (int r = 0; r < 8; ++r) g += gbp[r * kFU + t];
      a.master_w[dof + a.offB0 + u0 + t] = fmaf(-a.lr, g, b0m[t]);
    }
    // head weight gradient + SGD of this CTA's columns: item = (class, 4 units)
    for (int q = t; q < kFC * (kFU / 4); q += kFT) {
      const int c = q / (kFU / 4), u4 = (q % (kFU / 4)) * 4;
      float4 dw = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int b = 0; b < B; ++b) {
        const float g = dzb[b * kFC + c];
        const float4 hv = *reinterpret_cast<const float4*>(hs + b * Cfg::kHsd + u4);
        dw.x = fmaf(g, hv.x, dw.x);
        dw.y = fmaf(g, hv.y, dw.y);
        dw.z = fmaf(g, hv.z, dw.z);
        dw.w = fmaf(g, hv.w, dw.w);
      }
      const int64_t e = a.offW1 + static_cast<int64_t>(c) * H + u0 + u4;
      const float4 o = *reinterpret_cast<const float4*>(w1m + c * kFU + u4);
      float4 nw;
      nw.x = fmaf(-a.lr, dw.x, o.x);
      nw.y = fmaf(-a.lr, dw.y, o.y);
      nw.z = fmaf(-a.lr, dw.z, o.z);
      nw.w = fmaf(-a.lr, dw.w, o.w);
      *reinterpret_cast<float4*>(a.master_w + dof + e) = nw;
      *reinterpret_cast<uint2*>(a.shadow + dof + e) = make_uint2(pack_bf16x2(nw.x, nw.y), pack_bf16x2(nw.z, nw.w));
    }

    if (stamp) a.phase_ts[s * 4 + 2] = global_ns();
    // ------------------------------------------------------------ D: weight gradient + SGD of W0 rows
    if (warp == 0 && lane == 0) {
      for (int tt = 0; tt < nD; ++tt) {
        const int c = dcount + tt, buf = c % Cfg::kNBD, use = c / Cfg::kNBD;
        // the buffer's previous tile must be fully consumed (MMA and epilogue)
        if (use >= 1 && !mbar_wait(&tfreeD[buf], (use - 1) & 1, a.err, kDevTimeoutEmpty)) break;
        mbar_arrive_expect_tx(&fullD[buf], Cfg::kBufD);
        uint8_t* dst = region + buf * Cfg::kBufD;
#pragma unroll
        for (int kb = 0; kb < Cfg::kKB; ++kb)
          tma_load_4d(dst + kb * Cfg::kND * 128, &mXT, kb * kFBK, tt * Cfg::kND, w, s, &fullD[buf]);
        tma_load_3d(dst + Cfg::kXtBytes, &mWm, tt * Cfg::kND, u0, src, &fullD[buf]);   // old W0 rows
      }
    } else if (warp == 1 && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, Cfg::kND);
      for (int tt = 0; tt < nD; ++tt) {
        const int c = dcount + tt, buf = c % Cfg::kNBD, use = c / Cfg::kNBD;
        if (!mbar_wait(&fullD[buf], use & 1, a.err, kDevTimeoutFull)) break;
        if (use >= 1 && !mbar_wait(&tfreeD[buf], (use - 1) & 1, a.err, kDevTimeoutAccum)) break;
        tc_fence_after();
        const uint32_t xa = smem_u32(region + buf * Cfg::kBufD);
        const uint32_t da = smem_u32(dzT);
        const uint32_t dcol = tmem + static_cast<uint32_t>(buf * Cfg::kND);
#pragma unroll
        for (int kb = 0; kb < Cfg::kKB; ++kb)
#pragma unroll
          for (int j = 0; j < kFBK / 16; ++j)
            umma_bf16(dcol, smem_desc_k128(da + kb * kFU * 128 + j * 32),
                      smem_desc_k128(xa + kb * Cfg::kND * 128 + j * 32), idesc, (kb | j) != 0 ? 1u : 0u);
        umma_commit(&accD[buf]);
      }
    } else if (warp >= 4) {
      // the two warpgroups take alternate tiles; a warp covers 32 rows x 32 columns
      const int quarter = warp & 3, grp = (warp - 4) >> 2;
      const int mb = quarter * 32;                       // local rows of this warp
      float* T = epi + (warp - 4) * 32 * 36;   // row stride 36: 16-byte accesses of 8 lanes hit distinct banks
      for (int tt = grp; tt < nD; tt += 2) {
        const int c = dcount + tt, buf = c % Cfg::kNBD, use = c / Cfg::kNBD;
        int ok = mbar_wait(&accD[buf], use & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
        ok = __all_sync(0xffffffffu, ok);
        tc_fence_after();
        if (ok) {
          const float* Ms = reinterpret_cast<const float*>(region + buf * Cfg::kBufD + Cfg::kXtBytes);
          const int n_base = tt * Cfg::kND;              // first input feature of the tile
          float v[32];
          tmem_ld_32x32b_x32(tmem + (static_cast<uint32_t>(quarter * 32) << 16) + buf * Cfg::kND, v);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            *reinterpret_cast<float4*>(T + lane * 36 + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          __syncwarp();
          // lane -> (row 4 i + lane / 8, columns 4 (lane % 8) .. + 3): 4 rows per instruction
          const int cq = (lane & 7) * 4;
          const bool nok = n_base + cq < D;   // D % 8 == 0: a 4-column group is all in or all out
#pragma unroll
          for (int i = 0; i < 8; ++i) {
            const int r = 4 * i + (lane >> 3);
            const float4 g = *reinterpret_cast<const float4*>(T + r * 36 + cq);
            const float4 o = *reinterpret_cast<const float4*>(Ms + (mb + r) * Cfg::kND + cq);
            float4 nw;
            nw.x = fmaf(-a.lr, g.x, o.x);
            nw.y = fmaf(-a.lr, g.y, o.y);
            nw.z = fmaf(-a.lr, g.z, o.z);
            nw.w = fmaf(-a.lr, g.w, o.w);
            if (nok) {
              const int64_t e = dof + a.offW0 + static_cast<int64_t>(u0 + mb + r) * D + n_base + cq;
              *reinterpret_cast<float4*>(a.master_w + e) = nw;
              *reinterpret_cast<uint2*>(a.shadow + e) = make_uint2(pack_bf16x2(nw.x, nw.y), pack_bf16x2(nw.z, nw.w));
            }
          }
          __syncwarp();
        }
        tc_fence_before();
        mbar_arrive(&tfreeD[buf]);
      }
    }
    dcount += nD;
    fence_proxy_async_global();   // W0 rows written here are read by TMA next step
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    cluster_sync();               // head bias (rank 0) visible; pl / dz0^T reusable
    if (stamp) a.phase_ts[s * 4 + 3] = global_ns();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int B>
cudaError_t launch_b(const CUtensorMap& mW0, const CUtensorMap& mX, const CUtensorMap& mXT, const CUtensorMap& mWm,
                     const FusedArgs& a, cudaStream_t s) {
  using Cfg = FCfg<B>;
  cudaError_t e = cudaFuncSetAttribute(fused_mlp2_round_kernel<B>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::kSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.W, a.H / kFU, 1);
  cfg.blockDim = dim3(kFT, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = a.H / kFU;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fused_mlp2_round_kernel<B>, mW0, mX, mXT, mWm, a);
}

}  // namespace

bool fused_round_supported(int L, int D, int H, int C, int B) {
  if (L != 2 || C != kFC || H % kFU != 0 || H / kFU > kFMaxCluster || D % 8 != 0) return false;
  if (B != 32 && B != 64) return false;   // a batch of 128 does not fit the shared-memory budget
  const int smem = B == 32 ? FCfg<32>::kSmem : FCfg<64>::kSmem;
  return smem <= 227 * 1024;
}

int fused_round_xt_rows(int B) { return FCfg<64>::kND; }

cudaError_t launch_fused_round(const CUtensorMap& mW0, const CUtensorMap& mX, const CUtensorMap& mXT,
                               const CUtensorMap& mWm, const FusedRoundArgs& r, cudaStream_t s) {
  FusedArgs a;
  a.tau = r.tau;
  a.W = r.W;
  a.D = r.D;
  a.H = r.H;
  a.global_slot = r.global_slot;
  a.lr = r.lr;
  a.master = r.master;
  a.master_w = r.master_w;
  a.shadow = r.shadow;
  a.slot_stride = r.slot_stride;
  a.offW0 = r.offW0;
  a.offB0 = r.offB0;
  a.offW1 = r.offW1;
  a.offB1 = r.offB1;
  a.labels = r.labels;
  a.loss_part = r.loss_part;
  a.max_tau = r.max_tau;
  a.err = r.err;
  a.phase_ts = r.phase_ts;
  switch (r.B) {
    case 32: return launch_b<32>(mW0, mX, mXT, mWm, a, s);
    case 64: return launch_b<64>(mW0, mX, mXT, mWm, a, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace oscars
