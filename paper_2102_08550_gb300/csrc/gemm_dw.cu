// Weight gradient + SGD of one dense layer for every active worker in one
// persistent launch (Eq. 4, "otherwise" branch: x <- x - lr g(x)):
//
//   dW[m][n] = sum_b G[b][m] X[b][n]        bf16 operands, fp32 sums in TMEM
//   W'[m][n] = fmaf(-lr, dW[m][n], W[m][n])  fp32 master and its bf16 copy
//   b'[m]    = fmaf(-lr, gb[m], b[m])        (with column tile 0)
//
// G^T [lane][M][B] and X^T [lane][N][B] are the K-major operands (K = the
// batch).  The work is the stream of the fp32 master (read once, written
// once) and its bf16 copy, so the kernel is built around moving those bytes
// asynchronously:
//  * tiles of 128 x 128 outputs, tile t = (lane, m-tile, n-tile) with n
//    fastest, CTAs striding over the tiles (one CTA per SM);
//  * warp 0 lane 0 (TMA producer) loads each tile's fp32 master block into
//    one of two buffers (four 32-column boxes, 128-byte swizzle) as soon as
//    that buffer is free, and the operand k-blocks through a 2-slot ring;
//  * warp 1 lane 0 issues tcgen05.mma into one of two TMEM accumulators of
//    128 columns, so tile i + 1's products run under tile i's epilogue;
//  * warp 2 owns the TMEM allocation;
//  * warps 4-11 (two per TMEM lane quarter, 32 rows x 64 columns each)
//    update their part of the master block in place in shared memory, write
//    the bf16 copy into a staging tile, and store both parts to the worker's
//    slot with their own TMA stores (32-row boxes): no epilogue warp waits
//    for another, and no thread waits for the writes to reach memory.  A
//    warp waits for its stores to have read shared memory only when it
//    starts the next tile; then it releases the previous master buffer.
// All mbarrier waits are bounded and there is no named barrier: a warp that
// gives up leaves its loop, and the waits of the others run out in turn.
#include "common.cuh"
#include "internal.h"

namespace oscars {

namespace {

constexpr int kDwTile = 128;                          // outputs per tile side
constexpr int kDwBK = 64;                             // K per operand k-block
constexpr int kDwThreads = 384;                       // 12 warps
constexpr int kDwEpiThreads = 256;                    // warps 4-11
constexpr int kDwMasterBytes = kDwTile * kDwTile * 4; // one fp32 block (four 32-column boxes)
constexpr int kDwBoxF32 = kDwTile * 32 * 4;           // 16 KB
constexpr int kDwOpBytes = 2 * kDwTile * kDwBK * 2;   // A + B of one k-block: 32 KB
constexpr int kDwShadowBytes = kDwTile * kDwTile * 2; // bf16 staging (two 64-column boxes)
constexpr int kDwBoxBf16 = kDwTile * 64 * 2;          // 16 KB
constexpr int kDwOffOps = 2 * kDwMasterBytes;
constexpr int kDwOffShadow = kDwOffOps + 2 * kDwOpBytes;
constexpr int kDwOffBar = kDwOffShadow + kDwShadowBytes;
constexpr int kDwSmem = kDwOffBar + 256 + 1024;       // barriers, TMEM slot, 1 KB alignment slack

struct DwBars {
  uint64_t full[2], empty[2];     // operand ring
  uint64_t mfull[2], mempty[2];   // master buffers
  uint64_t afull[2], aempty[2];   // TMEM accumulators
  uint64_t mma_done;              // the MMA issuer's last products, before TMEM is released
  uint32_t tmem;
};

__device__ __forceinline__ void dw_tile_coords(const DwArgs& a, int t, int mt, int nt, int& lane, int& m0, int& n0) {
  lane = t / (mt * nt);
  const int r = t - lane * mt * nt;
  m0 = (r / nt) * kDwTile;
  n0 = (r % nt) * kDwTile;
}

__global__ void __launch_bounds__(kDwThreads, 1) gemm_dw_kernel(const __grid_constant__ CUtensorMap mapA,
                                                                 const __grid_constant__ CUtensorMap mapB,
                                                                 const __grid_constant__ CUtensorMap mapMaster,
                                                                 const __grid_constant__ CUtensorMap mapMasterSt,
                                                                 const __grid_constant__ CUtensorMap mapShadowSt,
                                                                 const __grid_constant__ DwArgs a) {
  extern __shared__ uint8_t dw_smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(dw_smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sMaster = smem;                     // [2][4 boxes][128 rows][128 B]
  uint8_t* sOps = smem + kDwOffOps;            // [2][A 16 KB | B 16 KB]
  uint8_t* sShadow = smem + kDwOffShadow;      // [2 boxes][128 rows][128 B]
  DwBars* bars = reinterpret_cast<DwBars*>(smem + kDwOffBar);

  const int warp = threadIdx.x >> 5, lane_id = threadIdx.x & 31;
  const int mt = a.M / kDwTile, nt = (a.N + kDwTile - 1) / kDwTile;
  const int tiles = a.n_active * mt * nt;
  const int nk = (a.K + kDwBK - 1) / kDwBK;

  if (threadIdx.x == 0) {
    prefetch_tmap(&mapA);
    prefetch_tmap(&mapB);
    prefetch_tmap(&mapMaster);
    prefetch_tmap(&mapMasterSt);
    prefetch_tmap(&mapShadowSt);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->full[i], 1);
      mbar_init(&bars->empty[i], 1);
      mbar_init(&bars->mfull[i], 1);
      mbar_init(&bars->mempty[i], kDwEpiThreads / 32);
      mbar_init(&bars->afull[i], 1);
      mbar_init(&bars->aempty[i], kDwEpiThreads / 32);
    }
    mbar_init(&bars->mma_done, 1);
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  if (warp == 2) {
    tmem_alloc(&bars->tmem, 2 * kDwTile);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = bars->tmem;
  pdl_wait();      // the previous kernel's outputs (gradients, bias gradients) are complete
  pdl_trigger();

  if (warp == 0 && lane_id == 0) {
    // ---- TMA producer
    int kc = 0, it = 0;
    int armed_ops[2] = {0, 0}, armed_master[2] = {0, 0};
    bool ok = true;
    for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x, ++it) {
      int li, m0, n0;
      dw_tile_coords(a, t, mt, nt, li, m0, n0);
      const int wid = a.wid ? a.wid[li] : li, src = a.src ? a.src[li] : li;
      const int b = it & 1;
      if (it >= 2 && !(ok = mbar_wait(&bars->mempty[b], ((it >> 1) + 1) & 1, a.err, kDevTimeoutEmpty))) break;
      mbar_arrive_expect_tx(&bars->mfull[b], kDwMasterBytes);
      ++armed_master[b];
#pragma unroll
      for (int q = 0; q < 4; ++q)
        tma_load_3d(sMaster + b * kDwMasterBytes + q * kDwBoxF32, &mapMaster, n0 + 32 * q, m0, src, &bars->mfull[b]);
      for (int kb = 0; kb < nk; ++kb, ++kc) {
        const int s = kc & 1;
        if (kc >= 2 && !(ok = mbar_wait(&bars->empty[s], ((kc >> 1) + 1) & 1, a.err, kDevTimeoutEmpty))) break;
        mbar_arrive_expect_tx(&bars->full[s], kDwOpBytes);
        ++armed_ops[s];
        tma_load_3d(sOps + s * kDwOpBytes, &mapA, kb * kDwBK, m0, wid, &bars->full[s]);
        tma_load_3d(sOps + s * kDwOpBytes + kDwOpBytes / 2, &mapB, kb * kDwBK, n0, wid, &bars->full[s]);
      }
    }
    // no copy may still be landing in shared memory when the CTA ends (all
    // complete at once in a normal run; after a timeout the waits are bounded)
    for (int i = 0; i < 2; ++i) {
      if (armed_ops[i]) mbar_wait(&bars->full[i], (armed_ops[i] - 1) & 1, a.err, kDevTimeoutFull);
      if (armed_master[i]) mbar_wait(&bars->mfull[i], (armed_master[i] - 1) & 1, a.err, kDevTimeoutFull);
    }
  } else if (warp == 1 && lane_id == 0) {
    // ---- MMA issuer
    constexpr uint32_t idesc = idesc_bf16_f32(kDwTile, kDwTile);
    int kc = 0, it = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < tiles; t += gridDim.x, ++it) {
      const int b = it & 1;
      if (it >= 2 && !(ok = mbar_wait(&bars->aempty[b], ((it >> 1) + 1) & 1, a.err, kDevTimeoutAccum))) break;
      tc_fence_after();
      const uint32_t acc = tmem + static_cast<uint32_t>(b * kDwTile);
      for (int kb = 0; kb < nk; ++kb, ++kc) {
        const int s = kc & 1;
        if (!(ok = mbar_wait(&bars->full[s], (kc >> 1) & 1, a.err, kDevTimeoutFull))) break;
        tc_fence_after();
        const uint32_t a_base = smem_u32(sOps + s * kDwOpBytes);
        const uint32_t b_base = a_base + kDwOpBytes / 2;
#pragma unroll
        for (int j = 0; j < kDwBK / 16; ++j)
          umma_bf16(acc, smem_desc_k128(a_base + j * 32), smem_desc_k128(b_base + j * 32), idesc, (kb | j) != 0 ? 1u : 0u);
        umma_commit(&bars->empty[s]);
      }
      if (ok) umma_commit(&bars->afull[b]);
    }
    umma_commit(&bars->mma_done);      // every product issued above has landed before TMEM is released
    mbar_wait(&bars->mma_done, 0, a.err, kDevTimeoutAccum);
  } else if (warp >= 4) {
    // ---- epilogue: warp quarter q owns TMEM lanes [32 q, 32 q + 32) (tile rows),
    // half h owns columns [64 h, 64 h + 64)
    const int q = warp & 3, h = (warp - 4) >> 2;
    const int r = 32 * q + lane_id;
    const uint32_t rsw = static_cast<uint32_t>(r & 7);      // 128-byte swizzle phase of this row
    int it = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++it) {
      int li, m0, n0;
      dw_tile_coords(a, t, mt, nt, li, m0, n0);
      const int wid = a.wid ? a.wid[li] : li, src = a.src ? a.src[li] : li;
      const int b = it & 1;
      const bool ok = mbar_wait(&bars->afull[b], (it >> 1) & 1, a.err, kDevTimeoutAccum) &&
                      mbar_wait(&bars->mfull[b], (it >> 1) & 1, a.err, kDevTimeoutFull);
      if (!__all_sync(0xffffffffu, ok)) break;
      tc_fence_after();
      // this warp's stores of the previous tile have read the staging tile and
      // their part of the other master buffer: release that buffer
      if (lane_id == 0) {
        bulk_wait_read_all();
        if (it >= 1) mbar_arrive(&bars->mempty[b ^ 1]);
      }
      __syncwarp();
      uint8_t* mblk = sMaster + b * kDwMasterBytes;
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int col0 = 64 * h + 32 * c;                     // this chunk's 32 columns
        float v[32];
        tmem_ld_32x32b_x32(tmem + static_cast<uint32_t>(b * kDwTile + col0) + (static_cast<uint32_t>(32 * q) << 16), v);
        float4* row = reinterpret_cast<float4*>(mblk + (col0 / 32) * kDwBoxF32 + r * 128);
        uint4* srow = reinterpret_cast<uint4*>(sShadow + h * kDwBoxBf16 + r * 128);
        uint32_t pk[16];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float4* p = row + (static_cast<uint32_t>(j) ^ rsw);
          const float4 o = *p;
          float4 nw;
          nw.x = fmaf(-a.lr, v[4 * j + 0], o.x);
          nw.y = fmaf(-a.lr, v[4 * j + 1], o.y);
          nw.z = fmaf(-a.lr, v[4 * j + 2], o.z);
          nw.w = fmaf(-a.lr, v[4 * j + 3], o.w);
          *p = nw;
          pk[2 * j] = pack_bf16x2(nw.x, nw.y);
          pk[2 * j + 1] = pack_bf16x2(nw.z, nw.w);
        }
#pragma unroll
        for (int k = 0; k < 4; ++k)   // bf16 columns 32 c + 8 k .. + 8 of box h
          srow[static_cast<uint32_t>(4 * c + k) ^ rsw] = make_uint4(pk[4 * k], pk[4 * k + 1], pk[4 * k + 2], pk[4 * k + 3]);
      }
      // the accumulator is free for tile it + 2
      tc_fence_before();
      __syncwarp();
      if (lane_id == 0) mbar_arrive(&bars->aempty[b]);
      fence_proxy_async_smem();         // this thread's shared-memory writes, visible to the TMA store
      __syncwarp();
      if (lane_id == 0) {
        // the warp's 32 rows: two 32-column fp32 boxes and one 64-column bf16
        // box; boxes that start past N are skipped, a box that straddles N is
        // clipped by the TMA unit
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const int col0 = 64 * h + 32 * c;
          if (n0 + col0 < a.N)
            tma_store_3d(&mapMasterSt, mblk + (col0 / 32) * kDwBoxF32 + 32 * q * 128, n0 + col0, m0 + 32 * q, wid);
        }
        if (n0 + 64 * h < a.N)
          tma_store_3d(&mapShadowSt, sShadow + h * kDwBoxBf16 + 32 * q * 128, n0 + 64 * h, m0 + 32 * q, wid);
        bulk_commit_group();
      }
      // bias with the first column tile
      if (h == 0 && n0 == 0) {
        const int m = m0 + r;
        a.master_w[static_cast<int64_t>(wid) * a.slot_stride + a.offB + m] =
            fmaf(-a.lr, a.gb[static_cast<int64_t>(wid) * a.M + m],
                 a.master[static_cast<int64_t>(src) * a.slot_stride + a.offB + m]);
      }
    }
    if (lane_id == 0) bulk_wait_all();
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc(tmem, 2 * kDwTile);
  }
}

}  // namespace

bool gemm_dw_supported(int M, int N, int K) { return M % kDwTile == 0 && N % 8 == 0 && K >= 1; }

cudaError_t launch_gemm_dw(const CUtensorMap& mA, const CUtensorMap& mB, const CUtensorMap& mMaster,
                           const CUtensorMap& mMasterSt, const CUtensorMap& mShadowSt, const DwArgs& a, int sms,
                           cudaStream_t s) {
  if (!gemm_dw_supported(a.M, a.N, a.K) || a.n_active < 1 || sms < 1) return cudaErrorInvalidValue;
  cudaError_t e = cudaFuncSetAttribute(gemm_dw_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kDwSmem);
  if (e != cudaSuccess) return e;
  const int tiles = a.n_active * (a.M / kDwTile) * ((a.N + kDwTile - 1) / kDwTile);
  const int grid = tiles < sms ? tiles : sms;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid, 1, 1);
  cfg.blockDim = dim3(kDwThreads, 1, 1);
  cfg.dynamicSmemBytes = kDwSmem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = a.pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, gemm_dw_kernel, mA, mB, mMaster, mMasterSt, mShadowSt, a);
}

}  // namespace oscars
