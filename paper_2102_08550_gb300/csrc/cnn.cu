// The convolutional worker: local SGD steps of a CIFAR-shaped residual
// network (Eq. 4, "otherwise" branch, for the paper's kind of workload:
// ResNet on CIFAR-10, Section "Dataset and DL Models").
//
//   s = relu(conv(x) + b0);  per block u = relu(conv(h) + b_a),
//   v = relu(conv(u) + b_b + h);  g = mean_{y,x} v;  logits = g W_f^T + b_f
//
// Every convolution is 3x3, stride 1, zero padding 1, on 32 x 32 images with
// 64 channels (the input's channels are zero-padded to 64).  Activations are
// bf16 NHWC [lane][image][32][32][64]; a lane is one worker's batch.
//
// Kernels (all workers of a local step in one launch, grid y = active worker):
//  * conv_igemm_kernel: implicit GEMM on tcgen05.  An output tile is 128
//    pixels (4 image rows) x 64 channels, the sum over the 9 taps of
//    [128 pixels x 64 in-channels] x [64 x 64] products; the input boxes are
//    loaded by TMA shifted by the tap offsets (the zero padding is TMA's
//    out-of-bounds fill), one 6-row box per x-offset serving the three
//    y-offsets, and a CTA keeps its worker's weights resident across its
//    tiles.  Forward epilogue: bias, optional residual, ReLU, bf16.
//    Input-gradient mode: the boxes are shifted the other way and the weights
//    are the transposed copy; epilogue: optional skip-path gradient, the ReLU
//    mask of the layer input, bf16, and per-CTA channel sums for the bias
//    gradient.
//  * conv_wgrad_kernel: dW[o][tap][i] = sum_p dz[p][o] x[p + off(tap)][i] on
//    tcgen05 with both operands MN-major straight from the NHWC tensors: the
//    K dimension is the pixels, taps are stacked in pairs to make M = 128
//    (in-channels of two taps), N = 64 out-channels; one 4-row input box per
//    x-offset serves the three y-offsets.  Split over chunks of images (one
//    wave of CTAs); partial sums go to global memory.
//  * conv_sgd_kernel: sums the chunks in order, SGD of the fp32 master and
//    its bf16 copies (the forward layout and the transposed one), bias from
//    the per-tile sums.
//  * pool, head, and output-gradient kernels on CUDA cores; input staging.
#include "common.cuh"
#include "internal.h"

namespace oscars {
namespace {

constexpr int kCC = 64;                     // channels
constexpr int kImg = 32;                    // image height and width
constexpr int kPix = kImg * kImg;
constexpr int kTileRows = 4;                // image rows per 128-pixel tile
constexpr int kTilePix = kTileRows * kImg;  // 128
constexpr int kTilesPerImg = kImg / kTileRows;
constexpr int kTaps = 9;
constexpr int kCT = 128;                    // threads of the implicit-GEMM and pixel kernels
constexpr int kCB = kCC * kCC * 2;          // 8 KB: one tap of the weights
// weight gradient
constexpr int kWT = 128;
constexpr int kWTile = 2 * kImg * kCC * 2;  // 8 KB: 64 pixels (2 rows) x 64 channels
constexpr int kWPairs = 5;                  // accumulators of stacked tap pairs

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// ------------------------------------------------------------------ implicit GEMM (forward / input gradient)
// A CTA works through tiles c, c + cpw, c + 2 cpw, ... of one worker (grid x
// = c < cpw, grid y = active worker) with that worker's 9 weight taps resident
// in shared memory.  Per tile and x-offset dx one TMA box of 6 image rows
// (rows y0 - 1 .. y0 + 4, shifted by the x-offset) is loaded; the three
// y-offsets are its 4-row sub-tiles at row offsets 0, 1, 2 (multiples of 8
// pixel rows of 128 bytes, so the 128-byte swizzle phase is unchanged).  Two
// TMEM accumulators: the epilogue of one tile overlaps the MMAs of the next.
constexpr int kGT = 192;                    // warp 0 TMA, warp 1 MMA, warps 2-5 epilogue
constexpr int kGSlots = 6;                  // input boxes in flight (two tiles)
constexpr int kGBox = 6 * kImg * kCC * 2;   // 24 KB: 6 rows x 32 pixels x 64 channels
constexpr int kGW = kTaps * kCB;            // 72 KB of resident weights
constexpr int kGSmem = kGW + kGSlots * kGBox + 512 + 1024;   // + barriers, TMEM slot, bias
static_assert(kTilePix * (kCC + 1) * 4 <= kGSlots * kGBox, "the bias reduction reuses the input slots");

template <int MODE>   // 0 forward, 1 input gradient
__global__ void __launch_bounds__(kGT, 1) conv_igemm_kernel(const __grid_constant__ CUtensorMap mIn,
                                                            const __grid_constant__ CUtensorMap mW,
                                                            const __grid_constant__ ConvArgs a) {
  extern __shared__ uint8_t cs_raw[];
  uint8_t* sm = align1024(cs_raw);
  uint8_t* wts = sm;                 // [9][64][64] bf16, 128-byte swizzled K-major
  uint8_t* slots = sm + kGW;         // [kGSlots][6 rows][32][64]
  uint64_t* wfull = reinterpret_cast<uint64_t*>(slots + kGSlots * kGBox);
  uint64_t* full = wfull + 1;
  uint64_t* empty = full + kGSlots;
  uint64_t* accf = empty + kGSlots;  // [2]
  uint64_t* acce = accf + 2;         // [2] 128 arrivals
  uint32_t* tslot = reinterpret_cast<uint32_t*>(acce + 2);
  float* bias_s = reinterpret_cast<float*>(tslot + 4);   // [64] this worker's bias (forward)
  const int t = threadIdx.x, warp = t >> 5, lane_id = t & 31;
  const int c0 = blockIdx.x, cpw = gridDim.x, e = blockIdx.y;
  const int lane = a.wid[e], slot = a.src[e];
  const int ntiles = a.B * kTilesPerImg;
  const int my_tiles = (ntiles - c0 + cpw - 1) / cpw;
  if (t == 0) {
    prefetch_tmap(&mIn);
    prefetch_tmap(&mW);
    mbar_init(wfull, 1);
    for (int i = 0; i < kGSlots; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&accf[i], 1);
      mbar_init(&acce[i], 128);
    }
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 128);
    tmem_relinquish();
  }
  if (MODE == 0 && t >= 64 && t < 64 + kCC)
    bias_s[t - 64] = a.bias[static_cast<int64_t>(slot) * a.slot_stride + a.off_bias + (t - 64)];
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  constexpr int sgn = MODE == 0 ? 1 : -1;   // the input gradient reads the output gradient at p - off(tap)
  // im2col stem (forward): one tap of weights, one 4-row box per tile (mIn's
  // box is {64, 32, 4, 1}), four MMAs
  const bool one_tap = MODE == 0 && a.im2col;
  const int nbox = one_tap ? 1 : 3;
  if (t == 0) {
    mbar_arrive_expect_tx(wfull, one_tap ? kCB : kGW);
    for (int tap = 0; tap < (one_tap ? 1 : kTaps); ++tap) {
      if (MODE == 0) tma_load_4d(wts + tap * kCB, &mW, 0, tap, 0, slot, wfull);   // {in, tap, out, slot}
      else tma_load_4d(wts + tap * kCB, &mW, 0, 0, tap, slot, wfull);             // {out, in, tap, slot}
    }
    int it = 0;
    for (int k = 0; k < my_tiles; ++k) {
      const int tile = c0 + k * cpw;
      const int img = lane * a.B + tile / kTilesPerImg, y0 = (tile % kTilesPerImg) * kTileRows;
      for (int dx = 0; dx < nbox; ++dx, ++it) {
        const int sl = it % kGSlots;
        if (it >= kGSlots && !mbar_wait(&empty[sl], ((it / kGSlots) + 1) & 1, a.err, kDevTimeoutEmpty)) {
          k = my_tiles;
          break;
        }
        if (one_tap) {
          mbar_arrive_expect_tx(&full[sl], kTilePix * kCC * 2);
          tma_load_4d(slots + sl * kGBox, &mIn, 0, 0, y0, img, &full[sl]);
        } else {
          mbar_arrive_expect_tx(&full[sl], kGBox);
          tma_load_4d(slots + sl * kGBox, &mIn, 0, sgn * (dx - 1), y0 - 1, img, &full[sl]);
        }
      }
    }
  } else if (t == 32) {
    constexpr uint32_t idesc = idesc_bf16_f32(128, kCC);
    bool ok = mbar_wait(wfull, 0, a.err, kDevTimeoutFull);
    tc_fence_after();
    int it = 0;
    for (int k = 0; ok && k < my_tiles; ++k) {
      const int buf = k & 1, use = k >> 1;
      if (use >= 1 && !mbar_wait(&acce[buf], (use - 1) & 1, a.err, kDevTimeoutAccum)) break;
      tc_fence_after();
      for (int dx = 0; dx < nbox; ++dx, ++it) {
        const int sl = it % kGSlots;
        if (!mbar_wait(&full[sl], (it / kGSlots) & 1, a.err, kDevTimeoutFull)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t sa = smem_u32(slots + sl * kGBox);
        if (one_tap) {
#pragma unroll
          for (int j = 0; j < kCC / 16; ++j)
            umma_bf16(tmem + buf * kCC, smem_desc_k128(sa + j * 32), smem_desc_k128(smem_u32(wts) + j * 32), idesc,
                      j != 0 ? 1u : 0u);
          umma_commit(&empty[sl]);
          continue;
        }
#pragma unroll
        for (int dy = 0; dy < 3; ++dy) {
          const int rowoff = MODE == 0 ? dy : 2 - dy;   // sub-tile of the 6-row box
          const uint32_t aa = sa + rowoff * kImg * kCC * 2;
          const uint32_t bb = smem_u32(wts + (dy * 3 + dx) * kCB);
#pragma unroll
          for (int j = 0; j < kCC / 16; ++j)
            umma_bf16(tmem + buf * kCC, smem_desc_k128(aa + j * 32), smem_desc_k128(bb + j * 32), idesc,
                      (dx | dy | j) != 0 ? 1u : 0u);
        }
        umma_commit(&empty[sl]);
      }
      if (ok) umma_commit(&accf[buf]);
    }
  } else if (warp >= 2) {
    // epilogue: thread = output pixel (TMEM lane of its warp's quarter), 64 channels
    const int quarter = warp & 3;
    const int p = quarter * 32 + lane_id;
    const uint32_t trow = tmem + (static_cast<uint32_t>(quarter * 32) << 16);
    float bsum[kCC];
#pragma unroll
    for (int c = 0; c < kCC; ++c) bsum[c] = 0.f;
    for (int k = 0; k < my_tiles; ++k) {
      const int tile = c0 + k * cpw;
      const int img = lane * a.B + tile / kTilesPerImg, y0 = (tile % kTilesPerImg) * kTileRows;
      const int buf = k & 1, use = k >> 1;
      int ok = mbar_wait(&accf[buf], use & 1, a.err, kDevTimeoutAccum) ? 1 : 0;
      ok = __all_sync(0xffffffffu, ok);
      tc_fence_after();
      float v[kCC];
      {
        float lo[32], hi[32];
        tmem_ld_32x32b_x32_pair(trow + buf * kCC, lo, trow + buf * kCC + 32, hi);
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          v[c] = ok ? lo[c] : 0.f;
          v[32 + c] = ok ? hi[c] : 0.f;
        }
      }
      tc_fence_before();
      mbar_arrive(&acce[buf]);   // the accumulator has been read: the next tile may use it
      const int64_t base = (static_cast<int64_t>(img) * kPix + y0 * kImg + p) * kCC;
      if (MODE == 0) {
#pragma unroll
        for (int c = 0; c < kCC; ++c) v[c] += bias_s[c];
      }
      if (a.add) {
#pragma unroll
        for (int q = 0; q < kCC / 8; ++q) {
          const uint4 r = *reinterpret_cast<const uint4*>(a.add + base + 8 * q);
          const __nv_bfloat162* r2 = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float2 f = __bfloat1622float2(r2[j]);
            v[8 * q + 2 * j] += f.x;
            v[8 * q + 2 * j + 1] += f.y;
          }
        }
      }
      if (MODE == 0) {
#pragma unroll
        for (int c = 0; c < kCC; ++c) v[c] = fmaxf(v[c], 0.f);
      } else {
#pragma unroll
        for (int q = 0; q < kCC / 8; ++q) {
          const uint4 r = *reinterpret_cast<const uint4*>(a.mask + base + 8 * q);
          const __nv_bfloat162* r2 = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const float2 f = __bfloat1622float2(r2[j]);
            if (!(f.x > 0.f)) v[8 * q + 2 * j] = 0.f;
            if (!(f.y > 0.f)) v[8 * q + 2 * j + 1] = 0.f;
          }
        }
#pragma unroll
        for (int c = 0; c < kCC; ++c) bsum[c] += v[c];
      }
#pragma unroll
      for (int q = 0; q < kCC / 8; ++q)
        *reinterpret_cast<uint4*>(a.out + base + 8 * q) =
            make_uint4(pack_bf16x2(v[8 * q], v[8 * q + 1]), pack_bf16x2(v[8 * q + 2], v[8 * q + 3]),
                       pack_bf16x2(v[8 * q + 4], v[8 * q + 5]), pack_bf16x2(v[8 * q + 6], v[8 * q + 7]));
    }
    if (MODE == 1 && a.bias_part) {
      // this CTA's channel sums: per thread over its tiles in order, then over
      // the 128 pixels of the tile in pixel order (the input slots are idle now)
      float* T = reinterpret_cast<float*>(slots);
#pragma unroll
      for (int c = 0; c < kCC; ++c) T[p * (kCC + 1) + c] = bsum[c];
    }
  }
  if (MODE == 1 && a.bias_part) {
    __syncthreads();
    if (t < kCC) {
      const float* T = reinterpret_cast<const float*>(slots);
      float s = 0.f;
      for (int q = 0; q < kTilePix; ++q) s += T[q * (kCC + 1) + t];
      a.bias_part[(static_cast<int64_t>(lane) * cpw + c0) * kCC + t] = s;
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 128);
  }
}

// ------------------------------------------------------------------ weight gradient
// K-block = 64 pixels (2 image rows yr, yr + 1).  Per K-block TMA loads the
// output-gradient tile (2 rows) and, per x-offset dx, one 4-row box of the
// input (rows yr - 1 .. yr + 2, shifted by dx - 1); tap (dy, dx)'s operand is
// the box's 2-row sub-tile at row offset dy.  The A operand (M = 128) stacks
// two taps as two 64-channel atoms `lbo` bytes apart:
//   pair 0..2: (dy 0, dy 1) of box dx = pair      (atoms 4 KB apart)
//   pair 3:    dy 2 of box 0 and of box 1         (atoms one box apart)
//   pair 4:    dy 2 of box 2                      (upper half unused)
constexpr int kWRow = kImg * kCC * 2;           // 4 KB: one image row, 64 channels
constexpr int kWBox = 4 * kWRow;                // 16 KB
constexpr int kWStage2 = 3 * kWBox + kWTile;    // 56 KB: three input boxes + the output-gradient tile
constexpr int kWStages2 = 3;
constexpr int kWSmem2 = kWStages2 * kWStage2 + 256 + 1024;

__device__ __forceinline__ void wgrad_pair(int pr, int& start, int& lbo, int& tap0, int& tap1) {
  if (pr < 3) {
    start = pr * kWBox;
    lbo = kWRow;
    tap0 = pr;            // (dy 0, dx pr)
    tap1 = 3 + pr;        // (dy 1, dx pr)
  } else if (pr == 3) {
    start = 2 * kWRow;
    lbo = kWBox;
    tap0 = 6;             // (dy 2, dx 0)
    tap1 = 7;             // (dy 2, dx 1)
  } else {
    start = 2 * kWBox + 2 * kWRow;
    lbo = kWRow;
    tap0 = 8;             // (dy 2, dx 2)
    tap1 = -1;
  }
}

__global__ void __launch_bounds__(kWT, 1) conv_wgrad_kernel(const __grid_constant__ CUtensorMap mIn,
                                                            const __grid_constant__ CUtensorMap mDz,
                                                            const __grid_constant__ WgradArgs a) {
  extern __shared__ uint8_t ws_raw[];
  uint8_t* sm = align1024(ws_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(sm + kWStages2 * kWStage2);
  uint64_t* empty = full + kWStages2;
  uint64_t* accb = empty + kWStages2;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int t = threadIdx.x, warp = t >> 5;
  const int chunk = blockIdx.x, e = blockIdx.y;
  const int lane = a.wid[e];
  const int i0 = chunk * a.img_per_chunk;
  const int n_img = min(a.img_per_chunk, a.B - i0);
  const int nk = n_img * (kImg / 2);             // K-blocks: 64 pixels = 2 image rows
  if (t == 0) {
    prefetch_tmap(&mIn);
    prefetch_tmap(&mDz);
    for (int i = 0; i < kWStages2; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    mbar_init(accb, 1);
    fence_barrier_init();
  }
  if (warp == 0) {
    tmem_alloc(tslot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tslot;
  // im2col stem: one 2-row input box per K-block (mIn's box is {64, 32, 2, 1})
  // and one accumulator, tap 0 in its lower half
  const int npairs = a.im2col ? 1 : kWPairs;
  if (t == 0) {
    for (int kb = 0; kb < nk; ++kb) {
      const int st = kb % kWStages2;
      if (kb >= kWStages2 && !mbar_wait(&empty[st], ((kb / kWStages2) + 1) & 1, a.err, kDevTimeoutEmpty)) break;
      uint8_t* sa = sm + st * kWStage2;
      const int img = lane * a.B + i0 + kb / (kImg / 2), yr = (kb % (kImg / 2)) * 2;
      if (a.im2col) {
        mbar_arrive_expect_tx(&full[st], 2 * kWRow + kWTile);
        tma_load_4d(sa, &mIn, 0, 0, yr, img, &full[st]);
      } else {
        mbar_arrive_expect_tx(&full[st], kWStage2);
        for (int dx = 0; dx < 3; ++dx) tma_load_4d(sa + dx * kWBox, &mIn, 0, dx - 1, yr - 1, img, &full[st]);
      }
      tma_load_4d(sa + 3 * kWBox, &mDz, 0, 0, yr, img, &full[st]);
    }
  } else if (t == 32) {
    constexpr uint32_t idesc = idesc_bf16_f32_mn(128, kCC);
    for (int kb = 0; kb < nk; ++kb) {
      const int st = kb % kWStages2;
      if (!mbar_wait(&full[st], (kb / kWStages2) & 1, a.err, kDevTimeoutFull)) break;
      tc_fence_after();
      const uint32_t sa = smem_u32(sm + st * kWStage2);
      const uint32_t sb = sa + 3 * kWBox;
      if (a.im2col) {
        // A = the 2-row box (in-channels k); its upper atom (the next row) is not read back
#pragma unroll
        for (int j = 0; j < 4; ++j)
          umma_bf16(tmem, smem_desc_mn128(sa + j * 2048, kWRow), smem_desc_mn128(sb + j * 2048, kWTile), idesc,
                    (kb | j) != 0 ? 1u : 0u);
        umma_commit(&empty[st]);
        continue;
      }
#pragma unroll
      for (int pr = 0; pr < kWPairs; ++pr) {
        int start, lbo, tap0, tap1;
        wgrad_pair(pr, start, lbo, tap0, tap1);
#pragma unroll
        for (int j = 0; j < 4; ++j)   // K = 16 pixels per MMA: two 8-row groups
          umma_bf16(tmem + pr * kCC, smem_desc_mn128(sa + start + j * 2048, lbo), smem_desc_mn128(sb + j * 2048, kWTile),
                    idesc, (kb | j) != 0 ? 1u : 0u);
      }
      umma_commit(&empty[st]);
    }
    umma_commit(accb);
  }
  int ok = mbar_wait(accb, 0, a.err, kDevTimeoutAccum) ? 1 : 0;
  ok = __all_sync(0xffffffffu, ok);
  tc_fence_after();
  // TMEM lane r: row r of each pair's accumulator = (tap of atom r / 64, in-channel r % 64)
  const int r = t;
  const int ci = r & (kCC - 1);
  for (int pr = 0; pr < npairs; ++pr) {
    int start, lbo, tap0, tap1;
    wgrad_pair(pr, start, lbo, tap0, tap1);
    if (a.im2col) tap1 = -1;
    const int tap = r < 64 ? tap0 : tap1;
    float lo[32], hi[32];
    tmem_ld_32x32b_x32_pair(tmem + (static_cast<uint32_t>(warp * 32) << 16) + pr * kCC, lo,
                            tmem + (static_cast<uint32_t>(warp * 32) << 16) + pr * kCC + 32, hi);
    if (tap >= 0 && ok) {
      float* dst = a.part + ((static_cast<int64_t>(lane) * a.n_chunks + chunk) * kTaps + tap) * kCC * kCC + ci * kCC;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        reinterpret_cast<float4*>(dst)[q] = make_float4(lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
        reinterpret_cast<float4*>(dst + 32)[q] = make_float4(hi[4 * q], hi[4 * q + 1], hi[4 * q + 2], hi[4 * q + 3]);
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
}

// ------------------------------------------------------------------ reduce + SGD of the convolution layers
// grid (taps * 4, active workers, layers), 256 threads: one tap's 16 in-channel
// rows x 64 out-channels of one layer; the chunks are summed in chunk order.
// The im2col stem has one tap (its blocks of taps 1..8 return at once).
constexpr int kSgdRows = 16;
__global__ void __launch_bounds__(256) conv_sgd_kernel(const __grid_constant__ ConvSgdArgs a) {
  __shared__ float T[kSgdRows][kCC + 1];   // [in][out]
  const int tap = blockIdx.x / (kCC / kSgdRows), r0 = (blockIdx.x % (kCC / kSgdRows)) * kSgdRows;
  const int e = blockIdx.y, layer = blockIdx.z;
  const int lane = a.wid[e], src = a.src[e];
  const int t = threadIdx.x;
  const int ntap = a.im2col[layer] ? 1 : kTaps;   // the im2col stem: [out][k], one tap
  if (tap >= ntap) return;
  const float* part = a.part[layer] + (static_cast<int64_t>(lane) * a.n_chunks * kTaps + tap) * kCC * kCC + r0 * kCC;
  const int64_t chunk_stride = static_cast<int64_t>(kTaps) * kCC * kCC;
  for (int q = t; q < kSgdRows * kCC; q += 256) {
    float s = 0.f;
#pragma unroll 4
    for (int c = 0; c < a.n_chunks; ++c) s += part[c * chunk_stride + q];
    T[q / kCC][q % kCC] = s;
  }
  __syncthreads();
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride, dof = static_cast<int64_t>(lane) * a.slot_stride;
  const int64_t offW = a.offW[layer];
  // master / forward copy: [out][tap][in], in fastest
  for (int q = t; q < kSgdRows * kCC; q += 256) {
    const int co = q / kSgdRows, ci = q % kSgdRows;
    const int64_t off = offW + (static_cast<int64_t>(co) * ntap + tap) * kCC + r0 + ci;
    const float nw = fmaf(-a.lr, T[ci][co], a.master[so + off]);
    a.master_w[dof + off] = nw;
    a.shadow[dof + off] = __float2bfloat16_rn(nw);
    T[ci][co] = nw;   // in this loop every element is read and rewritten by one thread
  }
  if (a.wt[layer]) {
    __syncthreads();
    // transposed copy [tap][in][out], out fastest
    __nv_bfloat16* wt = a.wt[layer] + static_cast<int64_t>(lane) * a.wt_slot_stride +
                        (static_cast<int64_t>(tap) * kCC + r0) * kCC;
    for (int q = t; q < kSgdRows * kCC; q += 256) wt[q] = __float2bfloat16_rn(T[q / kCC][q % kCC]);
  }
  if (blockIdx.x == 0 && t < kCC) {   // bias: per-tile sums in tile order
    const float* bp = a.bias_part[layer] + static_cast<int64_t>(lane) * a.n_tiles[layer] * kCC;
    float s = 0.f;
    for (int i = 0; i < a.n_tiles[layer]; ++i) s += bp[static_cast<int64_t>(i) * kCC + t];
    a.master_w[dof + a.offB[layer] + t] = fmaf(-a.lr, s, a.master[so + a.offB[layer] + t]);
  }
}

// bf16 transposed weight copies of one slot from its fp32 master (after a merge)
__global__ void conv_refresh_wt_kernel(const float* master, __nv_bfloat16* wt, int64_t offW) {
  const int tap = blockIdx.x;
  for (int q = threadIdx.x; q < kCC * kCC; q += blockDim.x) {
    const int ci = q / kCC, co = q % kCC;
    wt[static_cast<int64_t>(tap) * kCC * kCC + q] =
        __float2bfloat16_rn(master[offW + (static_cast<int64_t>(co) * kTaps + tap) * kCC + ci]);
  }
}

// ------------------------------------------------------------------ input staging
// grid (B * 8 tiles, active), 128 threads: the image row of sample b is
// (start[lane] + s * B + b) mod n[lane] of the lane's shard (fp32 NHWC, Cin
// channels).  Channels >= Cin stay zero: the buffer is cleared once when the
// context is built, so only the 16-byte chunks that hold input channels are
// written (one chunk for Cin <= 8), item = (pixel, chunk) with consecutive
// threads on consecutive chunks.  With im2col (9 Cin <= 64) channel
// k = tap * Cin + i of pixel (y, x) is x[y + dy - 1][x + dx - 1][i] for
// tap = 3 dy + dx (zero outside the image): the stem becomes one 64 x 64
// product per pixel.
// im2col: the tile's 6 source rows (y0 - 1 .. y0 + 4, zero outside the
// image) are first copied to shared memory with coalesced loads; a table
// gives each channel k its offset from the centre pixel and its x-offset.
constexpr int kStageMaxCin = kCC / kTaps;   // 7: the largest input with an im2col stem
constexpr int kNoTap = 1 << 20;
__global__ void __launch_bounds__(kCT) cnn_stage_kernel(const __grid_constant__ CnnStageArgs a) {
  __shared__ float rows[(kTileRows + 2) * kImg * kStageMaxCin];
  __shared__ int koff[kCC], kdx[kCC];
  const int tile = blockIdx.x, e = blockIdx.y;
  const int lane = a.wid[e];
  const int b = tile / kTilesPerImg, pix0 = (tile % kTilesPerImg) * kTilePix;
  const int64_t n = a.n[lane];
  const int64_t row = (a.start[lane] + static_cast<int64_t>(a.step) * a.B + b) % n;
  const float* src = a.x[lane] + row * static_cast<int64_t>(kPix) * a.Cin;
  __nv_bfloat16* dst = a.out + ((static_cast<int64_t>(lane) * a.B + b) * kPix + pix0) * kCC;
  const int K = a.im2col ? kTaps * a.Cin : a.Cin;
  const int chunks = (K + 7) / 8;
  if (a.labels && tile % kTilesPerImg == 0 && threadIdx.x == 0)
    a.labels[static_cast<int64_t>(lane) * a.B + b] = a.y[lane][row];
  if (a.im2col) {
    const int Cin = a.Cin, rowel = kImg * Cin, y0 = pix0 / kImg;
    if (threadIdx.x < kCC) {
      const int k = threadIdx.x;
      if (k < K) {
        const int tap = k / Cin, i = k - tap * Cin, dy = tap / 3, dx = tap % 3;
        koff[k] = (dy - 1) * rowel + (dx - 1) * Cin + i;
        kdx[k] = dx - 1;
      } else {
        koff[k] = 0;
        kdx[k] = kNoTap;
      }
    }
    for (int i = threadIdx.x; i < (kTileRows + 2) * rowel; i += kCT) {
      const int yy = y0 - 1 + i / rowel;
      rows[i] = yy >= 0 && yy < kImg ? src[static_cast<int64_t>(y0 - 1) * rowel + i] : 0.f;
    }
    __syncthreads();
    for (int it = threadIdx.x; it < kTilePix * chunks; it += kCT) {
      const int px = it / chunks, q = it - px * chunks;
      const int x = px % kImg;
      const int centre = (px / kImg + 1) * rowel + x * Cin;
      float v[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int k = 8 * q + j, xx = x + kdx[k];
        v[j] = xx >= 0 && xx < kImg ? rows[centre + koff[k]] : 0.f;
      }
      *reinterpret_cast<uint4*>(dst + static_cast<int64_t>(px) * kCC + 8 * q) =
          make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
    }
    return;
  }
  for (int it = threadIdx.x; it < kTilePix * chunks; it += kCT) {
    const int px = it / chunks, q = it - px * chunks;
    float v[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int c = 8 * q + j;
      v[j] = c < K ? src[static_cast<int64_t>(pix0 + px) * a.Cin + c] : 0.f;
    }
    *reinterpret_cast<uint4*>(dst + static_cast<int64_t>(px) * kCC + 8 * q) =
        make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
  }
}

// ------------------------------------------------------------------ pooling
// grid (B, active), 256 threads: g[lane][b][c] = sum over the 1024 pixels / 1024.
// Thread t sums channels 8 (t % 8) .. + 8 over pixels t / 8 + 32 i (16-byte
// loads, a warp reading 512 contiguous bytes), then the 32 partials of each
// channel group are summed in order.
__global__ void __launch_bounds__(256) cnn_pool_kernel(const __nv_bfloat16* v, const int* wid, int B, float* g) {
  __shared__ float part[32][kCC + 1];
  const int b = blockIdx.x, lane = wid[blockIdx.y];
  const int q = threadIdx.x & 7, p0 = threadIdx.x >> 3;
  const __nv_bfloat16* src = v + (static_cast<int64_t>(lane) * B + b) * kPix * kCC + 8 * q;
  float s[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) s[j] = 0.f;
#pragma unroll 4
  for (int p = p0; p < kPix; p += 32) {
    const uint4 r = *reinterpret_cast<const uint4*>(src + static_cast<int64_t>(p) * kCC);
    const __nv_bfloat162* r2 = reinterpret_cast<const __nv_bfloat162*>(&r);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(r2[j]);
      s[2 * j] += f.x;
      s[2 * j + 1] += f.y;
    }
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) part[p0][8 * q + j] = s[j];
  __syncthreads();
  if (threadIdx.x < kCC) {
    float t = 0.f;
    for (int r = 0; r < 32; ++r) t += part[r][threadIdx.x];
    g[(static_cast<int64_t>(lane) * B + b) * kCC + threadIdx.x] = t / static_cast<float>(kPix);
  }
}

// ------------------------------------------------------------------ head: FC, softmax CE, backward, SGD of the FC
// grid (active), 256 threads; B <= 256, K <= 32
__global__ void __launch_bounds__(256) cnn_head_kernel(const __grid_constant__ CnnHeadArgs a) {
  extern __shared__ float hsm[];
  const int K = a.K, B = a.B;
  float* gb = hsm;                    // [B][64] bf16-rounded pooled features
  float* wf = gb + B * kCC;           // [K][64] bf16-rounded head weights
  float* wm = wf + K * kCC;           // [K][64] fp32 master
  float* dl = wm + K * kCC;           // [B][K] fp32 logit gradient
  float* dlb = dl + B * K;            // [B][K] bf16-rounded
  float* rl = dlb + B * K;            // [B] per-sample loss
  float* bfm = rl + B;                // [32]
  const int e = blockIdx.x, lane = a.wid[e], src = a.src[e];
  const int t = threadIdx.x;
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride, dof = static_cast<int64_t>(lane) * a.slot_stride;
  for (int q = t; q < B * kCC; q += 256) gb[q] = bf16_round(a.g[static_cast<int64_t>(lane) * B * kCC + q]);
  for (int q = t; q < K * kCC; q += 256) {
    const float m = a.master[so + a.offWf + q];
    wm[q] = m;
    wf[q] = bf16_round(m);
  }
  if (t < K) bfm[t] = a.master[so + a.offBf + t];
  __syncthreads();
  for (int b = t; b < B; b += 256) {
    const int y = a.labels[static_cast<int64_t>(lane) * B + b];
    float z[32];
    float mx = -INFINITY, zy = 0.f;
    for (int k = 0; k < K; ++k) {
      float acc = 0.f;
      for (int c = 0; c < kCC; ++c) acc = fmaf(gb[b * kCC + c], wf[k * kCC + c], acc);
      z[k] = acc + bfm[k];
      if (k == y) zy = z[k];
      mx = fmaxf(mx, z[k]);
    }
    float se = 0.f, so_ = 0.f;
    for (int k = 0; k < K; ++k) {
      const float ev = expf(z[k] - mx);
      z[k] = ev;
      se += ev;
      if (k != y) so_ += ev;
    }
    rl[b] = mx + logf(se) - zy;
    const float inv = 1.0f / static_cast<float>(B);
    for (int k = 0; k < K; ++k) {
      const float gk = (k == y ? -(so_ / se) : z[k] / se) * inv;
      dl[b * K + k] = gk;
      dlb[b * K + k] = bf16_round(gk);
    }
  }
  __syncthreads();
  if (a.loss_part && t < (B + kRowsPerLossChunk - 1) / kRowsPerLossChunk) {
    float l = 0.f;
    for (int r = t * kRowsPerLossChunk; r < min(B, (t + 1) * kRowsPerLossChunk); ++r) l += rl[r];
    a.loss_part[(static_cast<int64_t>(lane) * a.max_tau + a.step) * a.n_loss_chunks + t] = l;
  }
  // dg[b][c] = sum_k dlb[b][k] wf[k][c] (old weights)
  for (int q = t; q < B * kCC; q += 256) {
    const int b = q / kCC, c = q % kCC;
    float acc = 0.f;
    for (int k = 0; k < K; ++k) acc = fmaf(dlb[b * K + k], wf[k * kCC + c], acc);
    a.dg[static_cast<int64_t>(lane) * B * kCC + q] = acc;
  }
  // head weights and bias
  for (int q = t; q < K * kCC; q += 256) {
    const int k = q / kCC, c = q % kCC;
    float acc = 0.f;
    for (int b = 0; b < B; ++b) acc = fmaf(dlb[b * K + k], gb[b * kCC + c], acc);
    const float nw = fmaf(-a.lr, acc, wm[q]);
    a.master_w[dof + a.offWf + q] = nw;
    a.shadow[dof + a.offWf + q] = __float2bfloat16_rn(nw);
  }
  if (t < K) {
    float acc = 0.f;
    for (int b = 0; b < B; ++b) acc += dl[b * K + t];
    const float nb = fmaf(-a.lr, acc, bfm[t]);
    a.master_w[dof + a.offBf + t] = nb;
    a.shadow[dof + a.offBf + t] = __float2bfloat16_rn(nb);
  }
}

// loss of the global model on labelled pooled features (evaluation): grid 1, 256 threads
__global__ void __launch_bounds__(256) cnn_head_loss_kernel(const float* g, const int32_t* labels, int B, int K,
                                                            const float* master, int64_t offWf, int64_t offBf,
                                                            float* out) {
  __shared__ float wf[32 * kCC];
  __shared__ float bfm[32];
  __shared__ float rl[256];
  const int t = threadIdx.x;
  for (int q = t; q < K * kCC; q += 256) wf[q] = bf16_round(master[offWf + q]);
  if (t < K) bfm[t] = master[offBf + t];
  __syncthreads();
  float l = 0.f;
  for (int b = t; b < B; b += 256) {
    float z[32], mx = -INFINITY;
    for (int k = 0; k < K; ++k) {
      float acc = 0.f;
      for (int c = 0; c < kCC; ++c) acc = fmaf(bf16_round(g[static_cast<int64_t>(b) * kCC + c]), wf[k * kCC + c], acc);
      z[k] = acc + bfm[k];
      mx = fmaxf(mx, z[k]);
    }
    float se = 0.f;
    for (int k = 0; k < K; ++k) se += expf(z[k] - mx);
    l += mx + logf(se) - z[labels[b]];
  }
  rl[t] = l;
  __syncthreads();
  if (t == 0) {
    float s = 0.f;
    for (int i = 0; i < 256; ++i) s += rl[i];
    out[0] = s;
  }
}

// ------------------------------------------------------------------ output gradient of the last block
// grid (B * 8 tiles, active), 128 threads: dz = v > 0 ? dg / 1024 : 0, bf16,
// and per-tile channel sums of the fp32 values.  Item = (pixel, 16-byte
// chunk of 8 channels): thread t always has chunk t % 8 (pixels t / 8 + 16 i),
// so its 8 channel sums stay in registers; the 16 threads of a chunk add
// theirs in order through shared memory.  dg / 1024 is exact as dg * 2^-10.
__global__ void __launch_bounds__(kCT) cnn_dzb_kernel(const __nv_bfloat16* v, const float* dg, const int* wid, int B,
                                                      __nv_bfloat16* dz, float* bias_part) {
  __shared__ float dgs[kCC];
  __shared__ float T[kCT / 8][kCC + 1];
  const int tile = blockIdx.x, lane = wid[blockIdx.y];
  const int b = tile / kTilesPerImg, pix0 = (tile % kTilesPerImg) * kTilePix;
  const int64_t base = ((static_cast<int64_t>(lane) * B + b) * kPix + pix0) * kCC;
  if (threadIdx.x < kCC) dgs[threadIdx.x] = dg[(static_cast<int64_t>(lane) * B + b) * kCC + threadIdx.x] / static_cast<float>(kPix);
  __syncthreads();
  const int q = threadIdx.x & 7, p0 = threadIdx.x >> 3;
  float d[8], sum[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    d[j] = dgs[8 * q + j];
    sum[j] = 0.f;
  }
#pragma unroll 4
  for (int p = p0; p < kTilePix; p += kCT / 8) {
    const int64_t off = base + static_cast<int64_t>(p) * kCC + 8 * q;
    const uint4 r = *reinterpret_cast<const uint4*>(v + off);
    const __nv_bfloat162* r2 = reinterpret_cast<const __nv_bfloat162*>(&r);
    float o[8];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(r2[j]);
      o[2 * j] = f.x > 0.f ? d[2 * j] : 0.f;
      o[2 * j + 1] = f.y > 0.f ? d[2 * j + 1] : 0.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) sum[j] += o[j];
    *reinterpret_cast<uint4*>(dz + off) = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]),
                                                     pack_bf16x2(o[4], o[5]), pack_bf16x2(o[6], o[7]));
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) T[p0][8 * q + j] = sum[j];
  __syncthreads();
  if (threadIdx.x < kCC) {
    float s = 0.f;
    for (int r = 0; r < kCT / 8; ++r) s += T[r][threadIdx.x];
    bias_part[(static_cast<int64_t>(lane) * B * kTilesPerImg + tile) * kCC + threadIdx.x] = s;
  }
}

}  // namespace

// ------------------------------------------------------------------ launchers
int cnn_tiles_per_image() { return kTilesPerImg; }

int conv_ctas_per_worker(int B, int n_active, int sms) {
  const int tiles = B * kTilesPerImg;
  int cpw = sms / (n_active > 0 ? n_active : 1);
  if (cpw < 1) cpw = 1;
  if (cpw > tiles) cpw = tiles;
  return cpw;
}

cudaError_t launch_conv_igemm(int mode, const CUtensorMap& mIn, const CUtensorMap& mW, const ConvArgs& a, int n_active,
                              int cpw, cudaStream_t s) {
  const dim3 grid(cpw, n_active);
  if (mode == 0) {
    cudaError_t e = cudaFuncSetAttribute(conv_igemm_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem);
    if (e != cudaSuccess) return e;
    conv_igemm_kernel<0><<<grid, kGT, kGSmem, s>>>(mIn, mW, a);
  } else {
    cudaError_t e = cudaFuncSetAttribute(conv_igemm_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem);
    if (e != cudaSuccess) return e;
    conv_igemm_kernel<1><<<grid, kGT, kGSmem, s>>>(mIn, mW, a);
  }
  return cudaGetLastError();
}

int conv_wgrad_images_per_chunk(int B, int n_active, int sms) {
  int per_worker = sms / (n_active > 0 ? n_active : 1);   // CTAs per worker in one wave
  if (per_worker < 1) per_worker = 1;
  return (B + per_worker - 1) / per_worker;
}

cudaError_t launch_conv_wgrad(const CUtensorMap& mIn, const CUtensorMap& mDz, const WgradArgs& a, int n_active,
                              cudaStream_t s) {
  cudaError_t e = cudaFuncSetAttribute(conv_wgrad_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kWSmem2);
  if (e != cudaSuccess) return e;
  conv_wgrad_kernel<<<dim3(a.n_chunks, n_active), kWT, kWSmem2, s>>>(mIn, mDz, a);
  return cudaGetLastError();
}

cudaError_t launch_conv_sgd(const ConvSgdArgs& a, int n_active, cudaStream_t s) {
  if (a.layers < 1 || a.layers > kMaxConvLayers) return cudaErrorInvalidValue;
  conv_sgd_kernel<<<dim3(kTaps * (kCC / kSgdRows), n_active, a.layers), 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_conv_refresh_wt(const float* master, __nv_bfloat16* wt, int64_t offW, cudaStream_t s) {
  conv_refresh_wt_kernel<<<kTaps, 256, 0, s>>>(master, wt, offW);
  return cudaGetLastError();
}

cudaError_t launch_cnn_stage(const CnnStageArgs& a, int n_active, cudaStream_t s) {
  cnn_stage_kernel<<<dim3(a.B * kTilesPerImg, n_active), kCT, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_cnn_pool(const __nv_bfloat16* v, const int* wid, int B, float* g, int n_active, cudaStream_t s) {
  cnn_pool_kernel<<<dim3(B, n_active), 256, 0, s>>>(v, wid, B, g);
  return cudaGetLastError();
}

size_t cnn_head_smem(int B, int K) { return sizeof(float) * (static_cast<size_t>(B) * kCC + 2 * K * kCC + 2 * B * K + B + 32); }

cudaError_t launch_cnn_head(const CnnHeadArgs& a, int n_active, cudaStream_t s) {
  const size_t smem = cnn_head_smem(a.B, a.K);
  cudaError_t e = cudaFuncSetAttribute(cnn_head_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cnn_head_kernel<<<n_active, 256, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_cnn_head_loss(const float* g, const int32_t* labels, int B, int K, const float* master,
                                 int64_t offWf, int64_t offBf, float* out, cudaStream_t s) {
  cnn_head_loss_kernel<<<1, 256, 0, s>>>(g, labels, B, K, master, offWf, offBf, out);
  return cudaGetLastError();
}

cudaError_t launch_cnn_dzb(const __nv_bfloat16* v, const float* dg, const int* wid, int B, __nv_bfloat16* dz,
                           float* bias_part, int n_active, cudaStream_t s) {
  cnn_dzb_kernel<<<dim3(B * kTilesPerImg, n_active), kCT, 0, s>>>(v, dg, wid, B, dz, bias_part);
  return cudaGetLastError();
}

}  // namespace oscars
