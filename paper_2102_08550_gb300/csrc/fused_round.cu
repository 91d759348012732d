// A whole round of local steps of a two-layer bf16 MLP (input -> H hidden
// ReLU units -> 10 classes) in ONE launch (Eq. 4, "otherwise" branch: each
// worker runs tau_i SGD steps from the global model).
//
// One thread-block cluster serves one worker.  The hidden units come in
// groups of 128 (one tensor-core tile of rows); each group is served by S
// CTAs (S = 1 or 2) that split the INPUT dimension: CTA h of the group owns
// input columns [c_h, c_{h+1}) of the group's 128 rows of W0 (a split on a
// 64-column K-block boundary).  Cluster rank = group * S + h.  Every step of
// the worker runs inside the cluster:
//
//  F  forward: each CTA computes the partial pre-activation of the group's
//     128 units over its own input columns on tcgen05 (TMA-fed, TMEM
//     accumulator).  With S = 2 the pair exchanges partials through
//     distributed shared memory and each CTA keeps 128/S of the units:
//     z = (part_0 + part_1) + b0, h = relu(z), bf16, in shared memory;
//  H  last layer for the CTA's units: partial logits, summed over the whole
//     cluster in rank order through distributed shared memory, softmax
//     cross-entropy; the masked input gradient dz0[b][u] of its units is
//     written (as bf16) into the 128-byte-swizzled K-major dz0^T tile of
//     every CTA of its group (the A operand of step D); bias gradient and SGD
//     of b0 (own units), of the head weights (own columns) and, on rank 0,
//     of the head bias;
//  D  weight gradient of the group's 128 rows over the CTA's own input
//     columns, dW0[o][k] = sum_b dz0[b][o] X[b][k] on tcgen05 (X^T tiles and
//     the fp32 master tiles by TMA, four buffers), with the SGD update fused
//     in the epilogue (16-byte staged accesses, full lines).
//
// Ownership: a CTA rewrites only its own (rows x columns) block of W0, its
// own b0 entries and head-weight columns, so its next step reads its own
// writes; everything it reads from other CTAs (partials, dz0 rows, logits,
// the head bias written by rank 0) is ordered by cluster barriers.
// Generic-proxy writes that TMA or the tensor core read afterwards are
// fenced with fence.proxy.async.  Arithmetic and rounding points are those of
// the per-layer path (the pair's two partial sums are added in rank order).
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
constexpr int kFU = 128;               // hidden units per group (tensor-core rows)
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

__device__ __forceinline__ float4 ld_dsmem_f32x4(const float* local, uint32_t rank) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(remote)
               : "memory");
  return v;
}

__device__ __forceinline__ void st_dsmem_b16(void* local, uint32_t rank, __nv_bfloat16 v) {
  uint32_t remote;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_u32(local)), "r"(rank));
  const unsigned short bits = *reinterpret_cast<const unsigned short*>(&v);
  asm volatile("st.shared::cluster.b16 [%0], %1;" ::"r"(remote), "h"(bits) : "memory");
}

__device__ __forceinline__ unsigned long long global_ns() {
  unsigned long long v;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(v));
  return v;
}

// Per-shape configuration (all sizes known at compile time).
template <int B, int S>
struct FCfg {
  static_assert(B == 32 || B == 64, "batch of 32 or 64");
  static_assert(S == 1 || S == 2, "one or two CTAs per group");
  static constexpr int kUPC = kFU / S;                      // units per CTA in steps F (kept) and H
  static constexpr int kStagesF = 4;
  static constexpr int kABytes = kFU * kFBK * 2;            // W0 tile: 128 rows x 64 k
  static constexpr int kBBytes = B * kFBK * 2;              // X tile: B rows x 64 k
  static constexpr int kND = 32;                            // columns per weight-gradient tile
  static constexpr int kNBD = 4;                            // weight-gradient buffers in flight
  static constexpr int kXtBytes = kND * kFBK * 2;           // X^T tile: 32 rows x 64 k (K padded)
  static constexpr int kMsBytes = kFU * kND * 4;            // fp32 master tile: 128 rows x 32 columns
  static constexpr int kBufD = kXtBytes + kMsBytes;
  static constexpr int kZs = B + 4;                         // row stride of the partial z exchange (floats)
  static constexpr int kPipe = kStagesF * (kABytes + kBBytes);
  static constexpr int kPipeD = kNBD * kBufD;
  static constexpr int kZBytes = S > 1 ? kFU * kZs * 4 : 0;
  static constexpr int kRegion0 = kPipe > kPipeD ? kPipe : kPipeD;
  static constexpr int kRegion = kRegion0 > kZBytes ? kRegion0 : kZBytes;   // TMA area / z exchange
  static constexpr int kDzT = kFU * 128;                    // dz0^T tile: 128 rows x 64 k (batch padded)
  static constexpr int kTpr = 256 / B;                      // threads per row, partial logits
  static constexpr int kHsd = kUPC + 4 * kTpr;              // padded row stride of the float h tile
  static constexpr int kGrpRows = 256 / (kUPC / 4);         // rows per pass of the input-gradient items
  // shared memory carve-up (bytes, from a 1024-aligned base)
  static constexpr int oRegion = 0;
  static constexpr int oDzT = oRegion + kRegion;
  static constexpr int oHs = oDzT + kDzT;                    // [B][kHsd] float
  static constexpr int oWc = oHs + B * kHsd * 4;             // [C][kUPC] float (bf16 operand)
  static constexpr int oW1m = oWc + kFC * kUPC * 4;          // [C][kUPC] fp32 master head columns
  static constexpr int oPl = oW1m + kFC * kUPC * 4;          // [B][C]
  static constexpr int oDz = oPl + B * kFC * 4;              // [B][C]
  static constexpr int oDzb = oDz + B * kFC * 4;             // [B][C]
  static constexpr int oGbp = oDzb + B * kFC * 4;            // [kGrpRows][kUPC]
  static constexpr int oRowLoss = oGbp + kGrpRows * kUPC * 4;   // [B]
  static constexpr int oB0 = oRowLoss + B * 4;               // [kFU] b0 of the group's units
  static constexpr int oB1 = oB0 + kFU * 4;                  // [16]
  static constexpr int oLab = oB1 + 16 * 4;                  // [B] int
  static constexpr int oEpi = (oLab + B * 4 + 15) / 16 * 16; // 8 x [32][36] float staging tiles
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
  float* loss_out;                // [W]
  int64_t* cursor;                // [W]
  const int64_t* shard_n;         // [W]
};

// byte offset of element (row, k) in a K-major 128-byte-swizzled tile of one
// 64-wide K-block (the layout TMA writes and UMMA reads)
__device__ __forceinline__ uint32_t sw128_offset(int row, int k) {
  return static_cast<uint32_t>((row >> 3) * 1024 + (row & 7) * 128 + ((((k >> 3) ^ (row & 7)) & 7) << 4) +
                               (k & 7) * 2);
}

template <int B, int S>
__global__ void __launch_bounds__(kFT, 1) fused_mlp2_round_kernel(const __grid_constant__ CUtensorMap mW0,
                                                                 const __grid_constant__ CUtensorMap mX,
                                                                 const __grid_constant__ CUtensorMap mXT,
                                                                 const __grid_constant__ CUtensorMap mWm,
                                                                 const __grid_constant__ FusedArgs a) {
  using Cfg = FCfg<B, S>;
  constexpr int UPC = Cfg::kUPC;
  extern __shared__ uint8_t fs_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(fs_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* region = sm + Cfg::oRegion;
  float* zx = reinterpret_cast<float*>(region);   // [128][kZs] partial z (S = 2), after F
  uint8_t* dzT = sm + Cfg::oDzT;
  float* hs = reinterpret_cast<float*>(sm + Cfg::oHs);
  float* wcs = reinterpret_cast<float*>(sm + Cfg::oWc);
  float* w1m = reinterpret_cast<float*>(sm + Cfg::oW1m);
  float* pl = reinterpret_cast<float*>(sm + Cfg::oPl);
  float* dz = reinterpret_cast<float*>(sm + Cfg::oDz);
  float* dzb = reinterpret_cast<float*>(sm + Cfg::oDzb);
  float* gbp = reinterpret_cast<float*>(sm + Cfg::oGbp);
  float* rowloss = reinterpret_cast<float*>(sm + Cfg::oRowLoss);
  float* b0m = reinterpret_cast<float*>(sm + Cfg::oB0);
  float* b1m = reinterpret_cast<float*>(sm + Cfg::oB1);
  int* labs = reinterpret_cast<int*>(sm + Cfg::oLab);
  float* epi = reinterpret_cast<float*>(sm + Cfg::oEpi);
  uint64_t* bars = reinterpret_cast<uint64_t*>(sm + Cfg::oBar);
  uint64_t* fullF = bars;                      // [kStagesF]
  uint64_t* emptyF = fullF + Cfg::kStagesF;    // [kStagesF]
  uint64_t* accF = emptyF + Cfg::kStagesF;     // [1]
  uint64_t* fullD = accF + 1;                  // [kNBD] X^T + master tile landed
  uint64_t* accD = fullD + Cfg::kNBD;          // [kNBD] TMEM buffer full
  uint64_t* tfreeD = accD + Cfg::kNBD;         // [kNBD] TMEM + shared buffer drained (128 arrivals)
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tfreeD + Cfg::kNBD);

  const int w = blockIdx.x;
  const int rank = static_cast<int>(cluster_ctarank());
  const int ncl = static_cast<int>(gridDim.y);
  const int grp = rank / S, half = rank % S;    // unit group, column half
  const int g0 = grp * kFU;                     // first unit of the group
  const int ku0 = half * UPC;                   // first kept unit within the group
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int D = a.D, H = a.H;
  const int tau = a.tau[w];
  const int nkF = (D + kFBK - 1) / kFBK;
  const int kb_split = S > 1 ? nkF / 2 : nkF;
  const int kb_begin = half == 0 ? 0 : kb_split, kb_end = half == 0 ? kb_split : nkF;
  const int col_begin = kb_begin * kFBK;
  const int col_end = half == S - 1 ? D : kb_end * kFBK;
  const int nkf = kb_end - kb_begin;
  const int nD = (col_end - col_begin + Cfg::kND - 1) / Cfg::kND;

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
  int dcount = 0;   // D tiles so far (buffer ring position)
  const bool stamp = a.phase_ts && w == 0 && rank == 0 && t == 0;

  for (int s = 0; s < tau; ++s) {
    if (stamp) a.phase_ts[s * 4 + 0] = global_ns();
    const int src = s == 0 ? a.global_slot : w;
    const int64_t so = static_cast<int64_t>(src) * a.slot_stride;
    const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;

    // ------------------------------------------------------------ F: partial forward of the group's units
    if (warp == 0 && lane == 0) {
      fence_proxy_async_global();     // this CTA's generic writes of W0 precede these TMA reads
      for (int kb = 0; kb < nkf; ++kb) {
        const int c = kcount + kb, st = c % Cfg::kStagesF;
        if (c >= Cfg::kStagesF && !mbar_wait(&emptyF[st], ((c / Cfg::kStagesF) + 1) & 1, a.err, kDevTimeoutEmpty)) break;
        mbar_arrive_expect_tx(&fullF[st], Cfg::kABytes + Cfg::kBBytes);
        uint8_t* sa = region + st * (Cfg::kABytes + Cfg::kBBytes);
        tma_load_3d(sa, &mW0, (kb_begin + kb) * kFBK, g0, src, &fullF[st]);
        tma_load_4d(sa + Cfg::kABytes, &mX, (kb_begin + kb) * kFBK, 0, w, s, &fullF[st]);
      }
    } else if (warp == 1 && lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, B);
      for (int kb = 0; kb < nkf; ++kb) {
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
    kcount += nkf;
    // every global input of the F epilogue and of step H, fetched while the tensor core works
    for (int q = t; q < kFC * (UPC / 8); q += kFT) {
      const int c = q / (UPC / 8), c8 = (q % (UPC / 8)) * 8;
      const int64_t e = a.offW1 + static_cast<int64_t>(c) * H + g0 + ku0 + c8;
      const uint4 v = *reinterpret_cast<const uint4*>(a.shadow + so + e);
      const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(p2[j]);
        wcs[c * UPC + c8 + 2 * j] = f.x;
        wcs[c * UPC + c8 + 2 * j + 1] = f.y;
      }
      *reinterpret_cast<float4*>(w1m + c * UPC + c8) = *reinterpret_cast<const float4*>(a.master + so + e);
      *reinterpret_cast<float4*>(w1m + c * UPC + c8 + 4) = *reinterpret_cast<const float4*>(a.master + so + e + 4);
    }
    if (t < kFU) b0m[t] = a.master[so + a.offB0 + g0 + t];
    if (t < kFC) b1m[t] = a.master[so + a.offB1 + t];
    for (int b = t; b < B; b += kFT) labs[b] = a.labels[(static_cast<int64_t>(s) * a.W + w) * B + b];
    __syncthreads();   // the prefetched b0 is read by the F epilogue below
    if (warp >= 4) {   // epilogue F: thread = unit of the group, columns = samples
      int ok = mbar_wait(accF, s & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
      ok = __all_sync(0xffffffffu, ok);
      tc_fence_after();
      if (ok) {
        const int quarter = warp & 3, eg = (warp - 4) >> 2;
        const int u = quarter * 32 + lane;
        const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
        for (int c0 = eg * 32; c0 < B; c0 += 64) {
          float v[32];
          tmem_ld_32x32b_x32(trow + c0, v);
          if (S == 1) {
            const float bias = b0m[u];
#pragma unroll
            for (int j = 0; j < 32; ++j) hs[(c0 + j) * Cfg::kHsd + u] = bf16_round(fmaxf(v[j] + bias, 0.f));
          } else {
#pragma unroll
            for (int q = 0; q < 8; ++q)
              *reinterpret_cast<float4*>(zx + u * Cfg::kZs + c0 + 4 * q) =
                  make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
    if (S > 1) {
      // pair exchange: z of this CTA's units = part(half 0) + part(half 1) + b0
      cluster_sync();
      for (int q = t; q < UPC * (B / 4); q += kFT) {
        const int ul = q / (B / 4), b4 = (q % (B / 4)) * 4;
        const int ug = ku0 + ul;                   // unit within the group
        float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int j = 0; j < S; ++j) {
          const float* p = zx + ug * Cfg::kZs + b4;
          const float4 v = j == half ? *reinterpret_cast<const float4*>(p) : ld_dsmem_f32x4(p, grp * S + j);
          z.x += v.x;
          z.y += v.y;
          z.z += v.z;
          z.w += v.w;
        }
        const float bias = b0m[ug];
        hs[(b4 + 0) * Cfg::kHsd + ul] = bf16_round(fmaxf(z.x + bias, 0.f));
        hs[(b4 + 1) * Cfg::kHsd + ul] = bf16_round(fmaxf(z.y + bias, 0.f));
        hs[(b4 + 2) * Cfg::kHsd + ul] = bf16_round(fmaxf(z.z + bias, 0.f));
        hs[(b4 + 3) * Cfg::kHsd + ul] = bf16_round(fmaxf(z.w + bias, 0.f));
      }
      __syncthreads();
    }
    if (stamp) a.phase_ts[s * 4 + 1] = global_ns();

    // ------------------------------------------------------------ H: last layer for this CTA's units
    if (t < 256) {   // partial logits: kTpr threads per row, all classes in registers
      const int rb = t / Cfg::kTpr, q = t % Cfg::kTpr;
      float acc[kFC];
#pragma unroll
      for (int c = 0; c < kFC; ++c) acc[c] = 0.f;
      for (int k = 4 * q; k < UPC; k += 4 * Cfg::kTpr) {
        const float4 hv = *reinterpret_cast<const float4*>(hs + rb * Cfg::kHsd + k);
#pragma unroll
        for (int c = 0; c < kFC; ++c) {
          const float4 wv = *reinterpret_cast<const float4*>(wcs + c * UPC + k);
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
    cluster_sync();   // all remote reads of pl (and of the partial z) are done
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
    // written into the dz0^T tile of every CTA of the group
    if (t < 256) {
      constexpr int kLanesPerRow = UPC / 4;
      const int u4 = (t % kLanesPerRow) * 4, rg = t / kLanesPerRow;
      float4 wc[kFC];
#pragma unroll
      for (int c = 0; c < kFC; ++c) wc[c] = *reinterpret_cast<const float4*>(wcs + c * UPC + u4);
      float4 gs = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int b = rg; b < B; b += Cfg::kGrpRows) {
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
        for (int j = 0; j < 4; ++j) {
          const __nv_bfloat16 g16 = __float2bfloat16_rn(dv[j]);
          uint8_t* dst = dzT + sw128_offset(ku0 + u4 + j, b);
          *reinterpret_cast<__nv_bfloat16*>(dst) = g16;
#pragma unroll
          for (int o = 0; o < S; ++o)
            if (o != half) st_dsmem_b16(dst, grp * S + o, g16);
        }
      }
      *reinterpret_cast<float4*>(gbp + rg * UPC + u4) = gs;
    }
    fence_proxy_async_smem();   // dz0^T is read by the tensor core next
    __syncthreads();
    if (t < UPC) {   // b0 of this CTA's units
      float g = 0.f;
#pragma unroll
      for (int r = 0; r < Cfg::kGrpRows; ++r) g += gbp[r * UPC + t];
      a.master_w[dof + a.offB0 + g0 + ku0 + t] = fmaf(-a.lr, g, b0m[ku0 + t]);
    }
    // head weight gradient + SGD of this CTA's columns: item = (class, 4 units)
    for (int q = t; q < kFC * (UPC / 4); q += kFT) {
      const int c = q / (UPC / 4), u4 = (q % (UPC / 4)) * 4;
      float4 dw = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int b = 0; b < B; ++b) {
        const float g = dzb[b * kFC + c];
        const float4 hv = *reinterpret_cast<const float4*>(hs + b * Cfg::kHsd + u4);
        dw.x = fmaf(g, hv.x, dw.x);
        dw.y = fmaf(g, hv.y, dw.y);
        dw.z = fmaf(g, hv.z, dw.z);
        dw.w = fmaf(g, hv.w, dw.w);
      }
      const int64_t e = a.offW1 + static_cast<int64_t>(c) * H + g0 + ku0 + u4;
      const float4 o = *reinterpret_cast<const float4*>(w1m + c * UPC + u4);
      float4 nw;
      nw.x = fmaf(-a.lr, dw.x, o.x);
      nw.y = fmaf(-a.lr, dw.y, o.y);
      nw.z = fmaf(-a.lr, dw.z, o.z);
      nw.w = fmaf(-a.lr, dw.w, o.w);
      *reinterpret_cast<float4*>(a.master_w + dof + e) = nw;
      *reinterpret_cast<uint2*>(a.shadow + dof + e) = make_uint2(pack_bf16x2(nw.x, nw.y), pack_bf16x2(nw.z, nw.w));
    }
    if (S > 1) {
      cluster_sync();             // the partner's dz0^T rows have landed
      fence_proxy_async_smem();
    }
    if (stamp) a.phase_ts[s * 4 + 2] = global_ns();

    // ------------------------------------------------------------ D: weight gradient + SGD of own W0 block
    if (warp == 0 && lane == 0) {
      for (int tt = 0; tt < nD; ++tt) {
        const int c = dcount + tt, buf = c % Cfg::kNBD, use = c / Cfg::kNBD;
        // the buffer's previous tile must be fully consumed (MMA and epilogue)
        if (use >= 1 && !mbar_wait(&tfreeD[buf], (use - 1) & 1, a.err, kDevTimeoutEmpty)) break;
        mbar_arrive_expect_tx(&fullD[buf], Cfg::kBufD);
        uint8_t* dst = region + buf * Cfg::kBufD;
        const int n0 = col_begin + tt * Cfg::kND;
        tma_load_4d(dst, &mXT, 0, n0, w, s, &fullD[buf]);
        tma_load_3d(dst + Cfg::kXtBytes, &mWm, n0, g0, src, &fullD[buf]);   // old W0 block
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
        for (int j = 0; j < kFBK / 16; ++j)
          umma_bf16(dcol, smem_desc_k128(da + j * 32), smem_desc_k128(xa + j * 32), idesc, j != 0 ? 1u : 0u);
        umma_commit(&accD[buf]);
      }
    } else if (warp >= 4) {
      // the two warpgroups take alternate tiles; a warp covers 32 rows x 32 columns
      const int quarter = warp & 3, eg = (warp - 4) >> 2;
      const int mb = quarter * 32;                       // rows of this warp within the group
      float* T = epi + (warp - 4) * 32 * 36;   // row stride 36: 16-byte accesses of 8 lanes hit distinct banks
      for (int tt = eg; tt < nD; tt += 2) {
        const int c = dcount + tt, buf = c % Cfg::kNBD, use = c / Cfg::kNBD;
        int ok = mbar_wait(&accD[buf], use & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
        ok = __all_sync(0xffffffffu, ok);
        tc_fence_after();
        if (ok) {
          const float* Ms = reinterpret_cast<const float*>(region + buf * Cfg::kBufD + Cfg::kXtBytes);
          const int n_base = col_begin + tt * Cfg::kND;  // first input column of the tile
          float v[32];
          tmem_ld_32x32b_x32(tmem + (static_cast<uint32_t>(quarter * 32) << 16) + buf * Cfg::kND, v);
#pragma unroll
          for (int q = 0; q < 8; ++q)
            *reinterpret_cast<float4*>(T + lane * 36 + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
          __syncwarp();
          // lane -> (row 4 i + lane / 8, columns 4 (lane % 8) .. + 3): 4 rows per instruction
          const int cq = (lane & 7) * 4;
          const bool nok = n_base + cq < col_end;   // column ends are multiples of 8
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
              const int64_t e = dof + a.offW0 + static_cast<int64_t>(g0 + mb + r) * D + n_base + cq;
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
    fence_proxy_async_global();   // W0 written here is read by TMA next step
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    cluster_sync();               // head bias (rank 0) visible; exchange buffers reusable
    if (stamp) a.phase_ts[s * 4 + 3] = global_ns();
  }
  // round bookkeeping of this worker: mean loss over its steps (sum in step
  // order, fp64) and the data cursor
  if (rank == 0 && t == 0) {
    constexpr int nc = B / kRowsPerLossChunk;
    double sum = 0.0;
    for (int st = 0; st < tau; ++st)
      for (int c = 0; c < nc; ++c) sum += a.loss_part[(static_cast<int64_t>(w) * a.max_tau + st) * nc + c];
    a.loss_out[w] = static_cast<float>(sum / (static_cast<double>(B) * tau));
    a.cursor[w] = (a.cursor[w] + static_cast<int64_t>(tau) * B) % a.shard_n[w];
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

template <int B, int S>
cudaError_t launch_bs(const CUtensorMap& mW0, const CUtensorMap& mX, const CUtensorMap& mXT, const CUtensorMap& mWm,
                      const FusedArgs& a, cudaStream_t s) {
  using Cfg = FCfg<B, S>;
  cudaError_t e = cudaFuncSetAttribute(fused_mlp2_round_kernel<B, S>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::kSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(a.W, S * (a.H / kFU), 1);
  cfg.blockDim = dim3(kFT, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = S * (a.H / kFU);
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, fused_mlp2_round_kernel<B, S>, mW0, mX, mXT, mWm, a);
}

// two CTAs per unit group when the cluster stays within 8 CTAs and the input
// has at least two K-blocks
int split_for(int D, int H) { return (2 * (H / kFU) <= kFMaxCluster && (D + kFBK - 1) / kFBK >= 2) ? 2 : 1; }

}  // namespace

bool fused_round_supported(int L, int D, int H, int C, int B) {
  if (L != 2 || C != kFC || H % kFU != 0 || H / kFU > kFMaxCluster || D % 8 != 0) return false;
  if (B != 32 && B != 64) return false;
  int smem = 0;
  const int S = split_for(D, H);
  if (B == 32) smem = S == 2 ? FCfg<32, 2>::kSmem : FCfg<32, 1>::kSmem;
  else smem = S == 2 ? FCfg<64, 2>::kSmem : FCfg<64, 1>::kSmem;
  return smem <= 227 * 1024;
}

int fused_round_xt_rows(int) { return 32; }

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
  a.loss_out = r.loss_out;
  a.cursor = r.cursor;
  a.shard_n = r.shard_n;
  const int S = split_for(r.D, r.H);
  if (r.B == 32) return S == 2 ? launch_bs<32, 2>(mW0, mX, mXT, mWm, a, s) : launch_bs<32, 1>(mW0, mX, mXT, mWm, a, s);
  if (r.B == 64) return S == 2 ? launch_bs<64, 2>(mW0, mX, mXT, mWm, a, s) : launch_bs<64, 1>(mW0, mX, mXT, mWm, a, s);
  return cudaErrorInvalidValue;
}

}  // namespace oscars
