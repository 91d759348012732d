// Forward and backward of the last layer (10 classes) of the per-layer path
// on the tensor cores (Eq. 4, "otherwise" branch: one SGD step of the
// worker's head).  A cluster of H/F CTAs serves one active worker; CTA r owns
// hidden features [F r, F r + F), F = 128 NH with NH = 1 or 2 halves of 128
// (NH = 2 keeps the cluster at 4 CTAs for H = 1024: only 15 clusters of 8
// are resident on the GPU at once).  With h = the layer input (bf16,
// [B][H]) and W2 the head weights ([C][H]):
//
//  1. partial logits of the CTA's features, P[b][c] = sum_f h[b][f] W2[c][f]:
//     tcgen05.mma M = 128 rows, N = 16 classes (rows >= B and classes >= C
//     are zero-filled by the TMA loads), K = F features;
//  2. cluster barrier; the logits are the partials of ranks 0..n-1 summed in
//     that order from distributed shared memory, plus the bias; softmax
//     cross-entropy per row (one thread per row); dz (fp32) and its bf16
//     copy, written into two shared tiles laid out as tensor-core operands;
//  3. head weight gradient dW2^T[f][c] = sum_b h[b][f] dz[b][c] (per half
//     M = 128 features, N = 16, K = B: the h tile read MN-major) and SGD of
//     the CTA's head columns;
//  4. input gradient of the layer below, transposed: dh^T[f][b] = sum_c
//     W2[c][f] dz[b][c] (per half M = 128 features, N = B, K = 16: the W2
//     tile read MN-major); masked by h > 0; G^T rows from registers, the fp32 bias
//     gradient per feature, and G rows through the h tile (overwritten in
//     place with the bf16 input gradient, then written as full 16-byte
//     chunks of each row).
// Rank 0 also writes the loss partials and updates the head bias.  One
// thread issues the TMA loads and the MMAs; the accumulators share 128 NH
// TMEM columns (the phases run one after another).  All mbarrier waits are
// bounded; the cluster barriers are unconditional, so a timeout cannot leave
// a CTA of the cluster behind at one.
#include "common.cuh"
#include "internal.h"

namespace oscars {

namespace {

constexpr int kHT = 128;                 // hidden features per half (tensor-core rows)
constexpr int kHTThreads = 256;
constexpr int kHTMaxCluster = 8;
constexpr int kHTC = 10;                 // classes
constexpr int kHTN = 16;                 // classes padded to the MMA's N
constexpr int kHTRows = 128;             // rows of the h tile (B <= 128; the rest zero)

// shared memory carve-up (bytes from a 1024-aligned base) for NH halves
template <int NH>
struct HTCfg {
  static constexpr int F = kHT * NH;                     // features per CTA
  static constexpr int oH = 0;                           // h tile: F/64 boxes [128 rows][64 features] bf16, 128-B swizzle
  static constexpr int oW2 = oH + (F / 64) * kHTRows * 128;   // W2 tile: F/64 boxes [16 classes][64 features]
  static constexpr int oDzT = oW2 + (F / 64) * kHTN * 128;    // dz^T: [16 classes][B rows] K-major (K = rows), 2 atoms
  static constexpr int oDzK = oDzT + 2 * kHTN * 128;     // dz: [B rows][16 classes] K-major, no swizzle
  static constexpr int oPl = oDzK + kHTRows * 32;        // [128][16] fp32 partial logits (read by the cluster)
  static constexpr int oDz = oPl + kHTRows * kHTN * 4;   // [128][16] fp32 dlogits
  static constexpr int oLoss = oDz + kHTRows * kHTN * 4; // [128]
  static constexpr int oGbp = oLoss + kHTRows * 4;       // [2][F]
  static constexpr int oLab = oGbp + 2 * F * 4;          // [128] int
  static constexpr int oB2 = oLab + kHTRows * 4;         // [16]
  static constexpr int oBar = oB2 + kHTN * 4;            // tma, mma barriers, TMEM slot
  static constexpr int kSmem = oBar + 64 + 1024;
  static constexpr uint32_t kTmemCols = 128 * NH;
};

// element (row b, feature f) of the h tile (K-major, 128-byte swizzle, one box per 64 features)
__device__ __forceinline__ uint32_t h_off(int b, int f) {
  return static_cast<uint32_t>((f >> 6) * (kHTRows * 128) + b * 128 + ((((f & 63) >> 3) ^ (b & 7)) << 4) + (f & 7) * 2);
}

// K-major no-swizzle descriptor: core matrices of 8 rows x 16 bytes, `lbo`
// bytes apart along K and `sbo` bytes apart along M/N.
__device__ __forceinline__ uint64_t smem_desc_none(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
  uint64_t d = 0;
  d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
  d |= static_cast<uint64_t>((lbo >> 4) & 0x3FFFu) << 16;
  d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;
  d |= static_cast<uint64_t>(1) << 46;
  return d;
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

__device__ __forceinline__ void tmem_ld_32x32b_x16(uint32_t taddr, float (&v)[16]) {
  uint32_t r[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr)
      : "memory");
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// columns [c, c + 32) of the warp's 32 lanes as two 16-column loads under one wait
__device__ __forceinline__ void tmem_ld_32x32b_x16x2(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%32];\n\t"
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%33];\n\t"
      "tcgen05.wait::ld.sync.aligned;"
      : "=&r"(r[0]), "=&r"(r[1]), "=&r"(r[2]), "=&r"(r[3]), "=&r"(r[4]), "=&r"(r[5]), "=&r"(r[6]), "=&r"(r[7]),
        "=&r"(r[8]), "=&r"(r[9]), "=&r"(r[10]), "=&r"(r[11]), "=&r"(r[12]), "=&r"(r[13]), "=&r"(r[14]), "=&r"(r[15]),
        "=&r"(r[16]), "=&r"(r[17]), "=&r"(r[18]), "=&r"(r[19]), "=&r"(r[20]), "=&r"(r[21]), "=&r"(r[22]), "=&r"(r[23]),
        "=&r"(r[24]), "=&r"(r[25]), "=&r"(r[26]), "=&r"(r[27]), "=&r"(r[28]), "=&r"(r[29]), "=&r"(r[30]), "=&r"(r[31])
      : "r"(taddr), "r"(taddr + 16u)
      : "memory");
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

template <int NH>
__global__ void __launch_bounds__(kHTThreads) head_tc_kernel(const __grid_constant__ CUtensorMap mH,
                                                              const __grid_constant__ CUtensorMap mW2,
                                                              const __grid_constant__ HeadArgs a) {
  using Cfg = HTCfg<NH>;
  constexpr int F = Cfg::F;
  extern __shared__ uint8_t ht_raw[];
  uint8_t* sm = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(ht_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* hT = sm + Cfg::oH;
  uint8_t* w2 = sm + Cfg::oW2;
  uint8_t* dzT = sm + Cfg::oDzT;
  uint8_t* dzK = sm + Cfg::oDzK;
  float* pl = reinterpret_cast<float*>(sm + Cfg::oPl);
  float* dz = reinterpret_cast<float*>(sm + Cfg::oDz);
  float* rowloss = reinterpret_cast<float*>(sm + Cfg::oLoss);
  float* gbp = reinterpret_cast<float*>(sm + Cfg::oGbp);
  int* labs = reinterpret_cast<int*>(sm + Cfg::oLab);
  float* b2 = reinterpret_cast<float*>(sm + Cfg::oB2);
  uint64_t* tma_bar = reinterpret_cast<uint64_t*>(sm + Cfg::oBar);
  uint64_t* mma_bar = tma_bar + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(mma_bar + 1);

  const int H = a.H, B = a.B;
  const int i = blockIdx.x;
  const int w = a.wid[i], src = a.src[i];
  const uint32_t rank = cluster_ctarank();
  const int ncl = static_cast<int>(gridDim.y);
  const int k0 = blockIdx.y * F;
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride;
  const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;

  if (t == 0) {
    prefetch_tmap(&mH);
    prefetch_tmap(&mW2);
    mbar_init(tma_bar, 1);
    mbar_init(mma_bar, 1);
    fence_barrier_init();
  }
  pdl_wait();      // the layer input (the previous kernel's output) is complete
  if (t == 0) {
    // the h and W2 tiles, requested first: the rest of the prologue overlaps them
    mbar_arrive_expect_tx(tma_bar, (F / 64) * (kHTRows * 128 + kHTN * 128));
#pragma unroll
    for (int q = 0; q < F / 64; ++q) {
      tma_load_3d(hT + q * kHTRows * 128, &mH, k0 + 64 * q, 0, w, tma_bar);
      tma_load_3d(w2 + q * kHTN * 128, &mW2, k0 + 64 * q, 0, src, tma_bar);
    }
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, Cfg::kTmemCols);
    tmem_relinquish();
  }
  // the dz tiles' padding (classes >= C, rows >= B) stays zero
  for (int q = t; q < (2 * kHTN * 128 + kHTRows * 32) / 16; q += kHTThreads)
    reinterpret_cast<uint4*>(dzT)[q] = make_uint4(0, 0, 0, 0);
  for (int b = t; b < B; b += kHTThreads) labs[b] = a.labels[static_cast<int64_t>(w) * B + b];
  if (t < kHTN) b2[t] = t < kHTC ? a.master[so + a.offB + t] : 0.f;
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  pdl_trigger();

  // ---- 1. partial logits
  if (t == 0) {
    if (mbar_wait(tma_bar, 0, a.err, kDevTimeoutFull)) {
      tc_fence_after();
      constexpr uint32_t idesc = idesc_bf16_f32(kHTRows, kHTN);
#pragma unroll
      for (int kb = 0; kb < F / 64; ++kb)
#pragma unroll
        for (int j = 0; j < 4; ++j)
          umma_bf16(tmem, smem_desc_k128(smem_u32(hT + kb * kHTRows * 128) + j * 32),
                    smem_desc_k128(smem_u32(w2 + kb * kHTN * 128) + j * 32), idesc, (kb | j) != 0 ? 1u : 0u);
    }
    umma_commit(mma_bar);   // arrives even with nothing issued, so the waits below end
  }
  bool ok = mbar_wait(mma_bar, 0, a.err, kDevTimeoutAccum);
  tc_fence_after();
  if (warp < 4) {
    float v[16];
    tmem_ld_32x32b_x16(tmem + (static_cast<uint32_t>(32 * warp) << 16), v);
    float4* row = reinterpret_cast<float4*>(pl + (32 * warp + lane) * kHTN);
#pragma unroll
    for (int q = 0; q < 4; ++q) row[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();

  // ---- 2. logits (cluster sum in rank order), softmax cross-entropy, dz tiles
  if (t < B) {
    const int b = t;
    float z[kHTC];
#pragma unroll
    for (int c = 0; c < kHTC; ++c) z[c] = 0.f;
    // every rank's partials are requested before the first is added (a
    // remote load waits a round trip across the cluster)
    float4 p[kHTMaxCluster][3];
#pragma unroll
    for (int r = 0; r < kHTMaxCluster; ++r)
      if (r < ncl) {
        p[r][0] = ld_dsmem_f32x4(pl + b * kHTN, r);
        p[r][1] = ld_dsmem_f32x4(pl + b * kHTN + 4, r);
        p[r][2] = ld_dsmem_f32x4(pl + b * kHTN + 8, r);
      }
#pragma unroll
    for (int r = 0; r < kHTMaxCluster; ++r)
      if (r < ncl) {
        z[0] += p[r][0].x; z[1] += p[r][0].y; z[2] += p[r][0].z; z[3] += p[r][0].w;
        z[4] += p[r][1].x; z[5] += p[r][1].y; z[6] += p[r][1].z; z[7] += p[r][1].w;
        z[8] += p[r][2].x; z[9] += p[r][2].y;
      }
#pragma unroll
    for (int c = 0; c < kHTC; ++c) z[c] += b2[c];
    float m = z[0];
#pragma unroll
    for (int c = 1; c < kHTC; ++c) m = fmaxf(m, z[c]);
    const int y = labs[b];
    float e[kHTC], s = 0.f, so_ = 0.f, zy = 0.f;
#pragma unroll
    for (int c = 0; c < kHTC; ++c) {
      e[c] = expf(z[c] - m);
      s += e[c];
      if (c != y) so_ += e[c];
      else zy = z[c];
    }
    rowloss[b] = m + logf(s) - zy;
    const float inv = 1.0f / static_cast<float>(B);
    float g[kHTC];
#pragma unroll
    for (int c = 0; c < kHTC; ++c) {
      g[c] = (c == y ? -(so_ / s) : e[c] / s) * inv;
      dz[b * kHTN + c] = g[c];
    }
    // dz as the K-major [rows][16 classes] operand: classes 0-7 one 16-byte
    // chunk of core matrix (b / 8, 0), classes 8-9 the start of core matrix (b / 8, 1)
    uint8_t* ck = dzK + (b >> 3) * 256 + (b & 7) * 16;
    *reinterpret_cast<uint4*>(ck) = make_uint4(pack_bf16x2(g[0], g[1]), pack_bf16x2(g[2], g[3]),
                                               pack_bf16x2(g[4], g[5]), pack_bf16x2(g[6], g[7]));
    *reinterpret_cast<uint32_t*>(ck + 128) = pack_bf16x2(g[8], g[9]);
    // dz^T as the K-major [16 classes][rows] operand (K = rows, atoms of 64 rows)
    uint8_t* at = dzT + (b >> 6) * (kHTN * 128);
    const int e64 = b & 63;
#pragma unroll
    for (int c = 0; c < kHTC; ++c)
      *reinterpret_cast<__nv_bfloat16*>(at + c * 128 + ((((e64 >> 3) ^ (c & 7)) & 7) << 4) + (e64 & 7) * 2) =
          __float2bfloat16_rn(g[c]);
  }
  fence_proxy_async_smem();   // the dz tiles are read by the tensor core
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // ---- 3. head weight gradient (M = features, N = classes, K = rows) + SGD
  if (t == 0) {
    if (ok) {
      constexpr uint32_t idesc = idesc_bf16_f32(kHT, kHTN) | (1u << 15);   // A (h^T) MN-major
#pragma unroll
      for (int mh = 0; mh < NH; ++mh)   // half mh: features [128 mh, 128 mh + 128) into columns [16 mh, 16 mh + 16)
        for (int j = 0; j < B / 16; ++j)
          umma_bf16(tmem + 16 * mh, smem_desc_mn128(smem_u32(hT + mh * 2 * kHTRows * 128) + j * 2048, kHTRows * 128),
                    smem_desc_k128(smem_u32(dzT + (j >> 2) * (kHTN * 128)) + (j & 3) * 32), idesc, j != 0 ? 1u : 0u);
    }
    umma_commit(mma_bar);
  }
  if (rank == 0 && warp >= 4) {   // loss partials and the head bias (CUDA cores, meanwhile)
    const int u = t - 128;
    if (u < B / kRowsPerLossChunk) {
      float l = 0.f;
      for (int r = 0; r < kRowsPerLossChunk; ++r) l += rowloss[u * kRowsPerLossChunk + r];
      const int64_t row = static_cast<int64_t>(w) * a.part_mul + a.part_add;
      a.loss_part[row * (B / kRowsPerLossChunk) + u] = l;
    }
    if (u >= 32) {   // warps 5-7: 8 lanes per class, then shuffles within each group of 8 (whole warps)
      const int c = (u - 32) >> 3, j = u & 7;
      float g = 0.f;
      if (c < kHTC)
        for (int b = j; b < B; b += 8) g += dz[b * kHTN + c];
#pragma unroll
      for (int o = 4; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o, 8);
      if (c < kHTC && j == 0) a.master_w[dof + a.offB + c] = fmaf(-a.lr, g, a.master[so + a.offB + c]);
    }
  }
  // the old master values of this thread's head column, requested while the
  // MMAs run and before any new value is stored (source and destination
  // slots may be the same slab)
  float old[kHTC];
  if (warp < 4 * NH) {
    const int f = kHT * (warp >> 2) + 32 * (warp & 3) + lane;
#pragma unroll
    for (int c = 0; c < kHTC; ++c) old[c] = a.master[so + a.offW + static_cast<int64_t>(c) * H + k0 + f];
  }
  ok = mbar_wait(mma_bar, 1, a.err, kDevTimeoutAccum) && ok;
  tc_fence_after();
  if (warp < 4 * NH && ok) {
    const int mh = warp >> 2, q = warp & 3;
    const int f = kHT * mh + 32 * q + lane;
    float v[16];
    tmem_ld_32x32b_x16(tmem + 16 * mh + (static_cast<uint32_t>(32 * q) << 16), v);
#pragma unroll
    for (int c = 0; c < kHTC; ++c) {
      const int64_t e = a.offW + static_cast<int64_t>(c) * H + k0 + f;
      const float nw = fmaf(-a.lr, v[c], old[c]);
      a.master_w[dof + e] = nw;
      a.shadow_w[dof + e] = __float2bfloat16_rn(nw);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();

  // ---- 4. input gradient, transposed (M = features, N = rows, K = 16 classes)
  if (t == 0) {
    if (ok) {
      const uint32_t idesc = idesc_bf16_f32(kHT, B) | (1u << 15);   // A (W2^T) MN-major
#pragma unroll
      for (int mh = 0; mh < NH; ++mh)   // half mh into columns [B mh, B mh + B)
        umma_bf16(tmem + B * mh, smem_desc_mn128(smem_u32(w2 + mh * 2 * kHTN * 128), kHTN * 128),
                  smem_desc_none(smem_u32(dzK), 128, 256), idesc, 0u);
    }
    umma_commit(mma_bar);
  }
  ok = mbar_wait(mma_bar, 0, a.err, kDevTimeoutAccum) && ok;
  tc_fence_after();
  {
    // warp quarter q: features 32 q .. of its half; NH = 1: the two warp
    // groups split the rows; NH = 2: warp group g takes half g, all rows
    const int q = warp & 3, g = warp >> 2;
    const int mh = NH == 2 ? g : 0;
    const int f = kHT * mh + 32 * q + lane;
    const int rows = NH == 2 ? B : B / 2;
    const int r0 = NH == 2 ? 0 : g * rows;
    float gsum = 0.f;
    if (ok) {
      for (int c0 = 0; c0 < rows; c0 += 32) {   // rows is a multiple of 16; a 32-row pass when it fits
        const int b0 = r0 + c0;
        const int nr = rows - c0 >= 32 ? 32 : 16;
        float v[32];
        const uint32_t ta = tmem + static_cast<uint32_t>(B * mh + b0) + (static_cast<uint32_t>(32 * q) << 16);
        if (nr == 32) {
          tmem_ld_32x32b_x16x2(ta, v);
        } else {
          float h16[16];
          tmem_ld_32x32b_x16(ta, h16);
#pragma unroll
          for (int j = 0; j < 16; ++j) v[j] = h16[j];
        }
        uint32_t pk[16];
#pragma unroll
        for (int j = 0; j < 32; j += 2) {
          if (j >= nr) break;
          __nv_bfloat16* h0 = reinterpret_cast<__nv_bfloat16*>(hT + h_off(b0 + j, f));
          __nv_bfloat16* h1 = reinterpret_cast<__nv_bfloat16*>(hT + h_off(b0 + j + 1, f));
          const float d0 = __bfloat162float(*h0) > 0.f ? v[j] : 0.f;
          const float d1 = __bfloat162float(*h1) > 0.f ? v[j + 1] : 0.f;
          gsum += d0;
          gsum += d1;
          const __nv_bfloat162 p = __floats2bfloat162_rn(d0, d1);
          if (a.G) {      // the h tile now holds the bf16 input gradient at (b, f), for the G rows below
            *h0 = p.x;
            *h1 = p.y;
          }
          pk[j >> 1] = *reinterpret_cast<const uint32_t*>(&p);
        }
        uint4* gt = reinterpret_cast<uint4*>(a.GT + (static_cast<int64_t>(w) * H + k0 + f) * B + b0);
        gt[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        gt[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        if (nr == 32) {
          gt[2] = make_uint4(pk[8], pk[9], pk[10], pk[11]);
          gt[3] = make_uint4(pk[12], pk[13], pk[14], pk[15]);
        }
      }
    }
    gbp[(NH == 2 ? 0 : g) * F + f] = gsum;
  }
  tc_fence_before();
  __syncthreads();
  if (t < F && ok) a.gb[static_cast<int64_t>(w) * H + k0 + t] = NH == 2 ? gbp[t] : gbp[t] + gbp[F + t];
  if (ok && a.G) {   // G rows: 16-byte chunks of 8 features (when a consumer reads G K-major)
    for (int q = t; q < B * (F / 8); q += kHTThreads) {
      const int b = q / (F / 8), j = q % (F / 8);
      *reinterpret_cast<uint4*>(a.G + (static_cast<int64_t>(w) * B + b) * H + k0 + 8 * j) =
          *reinterpret_cast<const uint4*>(hT + h_off(b, 8 * j));
    }
  }
  cluster_sync();   // no CTA leaves while another may still read its partial logits
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, Cfg::kTmemCols);
  }
}

// halves per CTA: two when one half per CTA would need a cluster of more than 4
int head_tc_halves(int H) { return H / kHT > 4 ? 2 : 1; }

}  // namespace

bool head_tc_supported(int H, int B, int C) {
  if (C != kHTC || B % 32 != 0 || B < 32 || B > kHTRows || H % kHT != 0) return false;
  const int F = kHT * head_tc_halves(H);
  return H % F == 0 && H / F <= kHTMaxCluster;
}

template <int NH>
cudaError_t launch_head_tc_nh(const CUtensorMap& mH, const CUtensorMap& mW2, const HeadArgs& a, int n_active,
                              cudaStream_t s) {
  using Cfg = HTCfg<NH>;
  cudaError_t e = cudaFuncSetAttribute(head_tc_kernel<NH>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmem);
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_active, a.H / Cfg::F, 1);
  cfg.blockDim = dim3(kHTThreads, 1, 1);
  cfg.dynamicSmemBytes = Cfg::kSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = a.H / Cfg::F;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.pdl ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, head_tc_kernel<NH>, mH, mW2, a);
}

cudaError_t launch_head_tc(const CUtensorMap& mH, const CUtensorMap& mW2, const HeadArgs& a, int n_active,
                           cudaStream_t s) {
  if (!head_tc_supported(a.H, a.B, a.C)) return cudaErrorInvalidValue;
  return head_tc_halves(a.H) == 2 ? launch_head_tc_nh<2>(mH, mW2, a, n_active, s)
                                  : launch_head_tc_nh<1>(mH, mW2, a, n_active, s);
}

}  // namespace oscars
