// CUDA-core kernels of the MLP worker step (Eq. 4, "otherwise" branch) that
// are not dense contractions worth a tensor core: staging of the mini-batch,
// the classifier head (last layer: C <= 32 classes) with the softmax
// cross-entropy and its gradient, and small bookkeeping kernels.
//
// Operand precision (reading; the paper fixes none): every GEMM operand is
// rounded to bf16 (RNE) and products accumulate in fp32; bias, ReLU, softmax
// and the SGD update are fp32.
#include "common.cuh"
#include "internal.h"

namespace oscars {

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

// ---------------------------------------------------------------- stage
// Mini-batch of lane w: rows (start[w] + row_add + b) mod n[w] of its sample
// matrix, rounded to bf16 as A0 [B][D] and transposed A0T [D][B] (the
// K-major operand of the first layer's weight-gradient GEMM).  32 x 32
// tiles through shared memory so both writes are coalesced.
__device__ __forceinline__ void stage_tile(const StageArgs& a, int w, int64_t base, __nv_bfloat16* A0,
                                           __nv_bfloat16* A0T, int32_t* labels) {
  __shared__ __nv_bfloat16 tile[32][34];
  const int k0 = blockIdx.x * 32, b0 = blockIdx.y * 32;
  const float* X = a.x[w];
  const int64_t n = a.n[w];
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8
  for (int r = ty; r < 32; r += 8) {
    const int b = b0 + r, k = k0 + tx;
    __nv_bfloat16 v = __float2bfloat16_rn(0.f);
    if (b < a.B && k < a.D) {
      const int64_t row = (base + b) % n;
      v = __float2bfloat16_rn(X[row * a.D + k]);
      A0[static_cast<int64_t>(b) * a.D + k] = v;
    }
    tile[r][tx] = v;
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    const int k = k0 + r, b = b0 + tx;
    if (k < a.D && b < a.B) A0T[static_cast<int64_t>(k) * a.B + b] = tile[tx][r];
  }
  if (blockIdx.x == 0 && threadIdx.x < 32) {
    const int b = b0 + threadIdx.x;
    if (b < a.B) labels[b] = a.y[w][(base + b) % n];
  }
}

__global__ void __launch_bounds__(256) stage_kernel(const __grid_constant__ StageArgs a) {
  const int w = a.wid[blockIdx.z];
  const int64_t off = static_cast<int64_t>(w) * a.B * a.D;
  stage_tile(a, w, a.start[w] + a.row_add, a.A0 + off, a.A0T + off, a.labels + static_cast<int64_t>(w) * a.B);
}

// Every mini-batch of a round at once: grid z = step * W + worker (or the
// table of active slots); a CTA whose worker has fewer local steps returns at
// once.  Step s of worker w lands at offset (s * W + w) of the per-step
// buffers.  A CTA converts 32 rows x 128 features: the row offsets (cursor
// arithmetic modulo the shard) once per row, 16-byte loads of fp32 (D % 4 ==
// 0), all issued before any store, 8-byte bf16 stores of the row-major copy,
// and the transposed copy through a [row][feature] shared tile whose row
// stride (65 words) keeps both its writes and its column reads apart in the
// banks, written as 32-byte pieces of 16 samples.
constexpr int kStageRows = 32, kStageCols = 128;
constexpr int kStageLd = kStageCols + 2;   // bf16 row stride of the tile

// One tile of one (step, worker) slot: rows [by * kStageRows, +kStageRows)
// and features [bx * kStageCols, +kStageCols) of the slot's mini-batch.
__device__ __forceinline__ void stage_round_tile(const StageArgs& a, const int32_t* tau, int W, int bx, int by,
                                                 int bz, __nv_bfloat16 (&tile)[kStageRows][kStageLd],
                                                 int64_t (&rowoff)[kStageRows]) {
  const int z = a.slots ? a.slots[bz] : bz;
  const int s = z / W, w = z - s * W;
  if (s >= tau[w]) return;
  const int64_t slot = static_cast<int64_t>(s) * W + w;
  const int64_t off = slot * a.B * a.D;
  __nv_bfloat16* A0 = a.A0 + off;
  __nv_bfloat16* A0T = a.A0T + off;
  const float* X = a.x[w];
  const int64_t n = a.n[w];
  const int64_t base = a.start[w] + (static_cast<int64_t>(s) + (a.ahead ? a.ahead[w] : 0)) * a.B;
  const int k0 = bx * kStageCols, b0 = by * kStageRows;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;   // 32 x 8
  if (threadIdx.x < kStageRows) {
    const int b = b0 + threadIdx.x;
    const int64_t row = (base + b) % n;
    rowoff[threadIdx.x] = row * a.D;
    if (bx == 0 && b < a.B) a.labels[slot * a.B + b] = a.y[w][row];
  }
  __syncthreads();
  const int k = k0 + tx * 4;
  const bool kok = k < a.D;
  // all of this thread's rows are loaded before any is stored: the shards may
  // sit in host memory, where every load waits a round trip over the link
  float4 xv[kStageRows / 8];
#pragma unroll
  for (int i = 0; i < kStageRows / 8; ++i) {
    const int r = ty + 8 * i;
    xv[i] = make_float4(0.f, 0.f, 0.f, 0.f);
    if (b0 + r < a.B && kok) xv[i] = *reinterpret_cast<const float4*>(X + rowoff[r] + k);
  }
#pragma unroll
  for (int i = 0; i < kStageRows / 8; ++i) {
    const int r = ty + 8 * i, b = b0 + r;
    const float4 v = xv[i];
    const uint32_t lo = pack_bf16x2(v.x, v.y), hi = pack_bf16x2(v.z, v.w);
    if (b < a.B && kok) *reinterpret_cast<uint2*>(A0 + static_cast<int64_t>(b) * a.D + k) = make_uint2(lo, hi);
    uint32_t* t = reinterpret_cast<uint32_t*>(&tile[r][tx * 4]);
    t[0] = lo;
    t[1] = hi;
  }
  __syncthreads();
  {   // 128 feature rows x 32 samples: two 16-sample pieces per row
    const int kr = threadIdx.x >> 1, piece = threadIdx.x & 1;
    const int kk = k0 + kr;
    const int bb = b0 + piece * 16;
    if (kk < a.D && bb < a.B) {
      uint32_t p[8];
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const uint32_t e0 = __bfloat16_as_ushort(tile[piece * 16 + 2 * j][kr]);
        const uint32_t e1 = __bfloat16_as_ushort(tile[piece * 16 + 2 * j + 1][kr]);
        p[j] = e0 | (e1 << 16);
      }
      uint4* dst = reinterpret_cast<uint4*>(A0T + static_cast<int64_t>(kk) * a.B + bb);
      dst[0] = make_uint4(p[0], p[1], p[2], p[3]);
      dst[1] = make_uint4(p[4], p[5], p[6], p[7]);
    }
  }
}

__global__ void __launch_bounds__(256) stage_round_kernel(const __grid_constant__ StageArgs a, const int32_t* tau,
                                                          int W) {
  __shared__ __align__(16) __nv_bfloat16 tile[kStageRows][kStageLd];
  __shared__ int64_t rowoff[kStageRows];
  stage_round_tile(a, tau, W, blockIdx.x, blockIdx.y, blockIdx.z, tile, rowoff);
}

// The same tiles from a fixed number of blocks striding over them: a staging
// that runs beside other kernels keeps a bounded footprint (each block fits
// beside the GEMM blocks of an SM) while its loads stay in flight.
__global__ void __launch_bounds__(256) stage_round_strided_kernel(const __grid_constant__ StageArgs a,
                                                                  const int32_t* tau, int W, int nx, int ny,
                                                                  int nz) {
  __shared__ __align__(16) __nv_bfloat16 tile[kStageRows][kStageLd];
  __shared__ int64_t rowoff[kStageRows];
  const int64_t total = static_cast<int64_t>(nx) * ny * nz;
  for (int64_t lin = blockIdx.x; lin < total; lin += gridDim.x) {
    const int bx = static_cast<int>(lin % nx), by = static_cast<int>((lin / nx) % ny);
    const int bz = static_cast<int>(lin / (static_cast<int64_t>(nx) * ny));
    stage_round_tile(a, tau, W, bx, by, bz, tile, rowoff);
    __syncthreads();   // the tile and the row offsets are rewritten by the next one
  }
}

// ---------------------------------------------------------------- head forward
// Logits of the last layer z[b][c] = sum_k bf16(h[b][k]) bf16(W[c][k]) + bias[c]
// (fp32 accumulate), softmax cross-entropy, dlogits = (p - onehot)/B.
// Grid (active lanes, B/16); 16 rows per CTA, one warp per two rows; each
// lane keeps its slice of the row in registers (16-byte loads issued up
// front), the class weights sit in shared memory.
//
// Softmax without cancellation: e_c = exp(z_c - max z), s = sum_c e_c,
// p_c = e_c / s, and for the label 1 - p_y = (sum_{c != y} e_c) / s, so the
// gradient of a confidently classified sample keeps its relative accuracy.
constexpr int kHeadFwdThreads = 256;
constexpr int kHeadMaxH8 = 8;   // up to 8 x 16-byte slices per lane: H <= 2048

__global__ void __launch_bounds__(kHeadFwdThreads) head_fwd_kernel(const __grid_constant__ HeadArgs a) {
  extern __shared__ __align__(16) float hsm[];
  const int H = a.H, C = a.C, B = a.B;
  float* Wsm = hsm;            // [C][H] bf16 values as float
  __shared__ float rowloss[kRowsPerLossChunk];
  const int i = blockIdx.x;
  const int w = a.wid[i], src = a.src[i];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const __nv_bfloat16* Wg = a.shadow + static_cast<int64_t>(src) * a.slot_stride + a.offW;
  const float* bias = a.master + static_cast<int64_t>(src) * a.slot_stride + a.offB;
  for (int q = threadIdx.x; q < C * H / 8; q += kHeadFwdThreads) {
    const uint4 v = reinterpret_cast<const uint4*>(Wg)[q];
    const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(p2[j]);
      Wsm[q * 8 + 2 * j] = f.x;
      Wsm[q * 8 + 2 * j + 1] = f.y;
    }
  }
  __syncthreads();
  const int nslice = H / 256;   // 16-byte slices per lane (H is a multiple of 128; remainder below)
  for (int rr = warp; rr < kRowsPerLossChunk; rr += kHeadFwdThreads / 32) {
    const int b = blockIdx.y * kRowsPerLossChunk + rr;
    const __nv_bfloat16* h = a.Ain + (static_cast<int64_t>(w) * B + b) * H;
    // this lane's 8-element slices: k = (j * 32 + lane) * 8
    float hv[kHeadMaxH8][8];
#pragma unroll
    for (int j = 0; j < kHeadMaxH8; ++j) {
      const int k = (j * 32 + lane) * 8;
      if (k < H) {
        const uint4 v = *reinterpret_cast<const uint4*>(h + k);
        const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
        for (int t = 0; t < 4; ++t) {
          const float2 f = __bfloat1622float2(p2[t]);
          hv[j][2 * t] = f.x;
          hv[j][2 * t + 1] = f.y;
        }
      } else {
#pragma unroll
        for (int t = 0; t < 8; ++t) hv[j][t] = 0.f;
      }
    }
    (void)nslice;
    float zc = -INFINITY;  // lane c holds z_c
    for (int c = 0; c < C; ++c) {
      const float* wr = Wsm + c * H;
      float acc = 0.f;
#pragma unroll
      for (int j = 0; j < kHeadMaxH8; ++j) {
        const int k = (j * 32 + lane) * 8;
        if (k < H) {
          const float4 w0 = *reinterpret_cast<const float4*>(wr + k);
          const float4 w1 = *reinterpret_cast<const float4*>(wr + k + 4);
          acc = fmaf(hv[j][0], w0.x, acc);
          acc = fmaf(hv[j][1], w0.y, acc);
          acc = fmaf(hv[j][2], w0.z, acc);
          acc = fmaf(hv[j][3], w0.w, acc);
          acc = fmaf(hv[j][4], w1.x, acc);
          acc = fmaf(hv[j][5], w1.y, acc);
          acc = fmaf(hv[j][6], w1.z, acc);
          acc = fmaf(hv[j][7], w1.w, acc);
        }
      }
      acc = warp_sum(acc) + bias[c];
      if (lane == c) zc = acc;
    }
    const int y = a.labels[static_cast<int64_t>(w) * B + b];
    const float m = warp_max(zc);
    const float e = lane < C ? expf(zc - m) : 0.f;
    const float s = warp_sum(e);
    const float s_other = warp_sum(lane < C && lane != y ? e : 0.f);
    const float zy = __shfl_sync(0xffffffffu, zc, y);
    if (lane < C) {
      const float g = lane == y ? -(s_other / s) : e / s;
      a.dlog[(static_cast<int64_t>(w) * B + b) * C + lane] = g / static_cast<float>(B);
    }
    if (lane == 0) rowloss[rr] = m + logf(s) - zy;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float l = 0.f;
    for (int r = 0; r < kRowsPerLossChunk; ++r) l += rowloss[r];
    const int64_t row = static_cast<int64_t>(w) * a.part_mul + a.part_add;
    a.loss_part[row * (B / kRowsPerLossChunk) + blockIdx.y] = l;
  }
}

// ---------------------------------------------------------------- head backward
// CTA = (active lane, 64 hidden features k); 256 threads.
//  dh[b][k] = sum_c bf16(dz[b][c]) bf16(W_old[c][k]);  g = dh * (h[b][k] > 0)
//    -> bf16 G [B][H] and G^T [H][B] (operands of the next GEMMs) and
//       gb[k] = sum_b g (fp32, the bias gradient of the layer below);
//  dW[c][k] = sum_b bf16(dz[b][c]) bf16(h[b][k]);  W <- W - lr dW (fmaf);
//  CTA column 0 also updates the head bias with db[c] = sum_b dz[b][c].
// The h tile, dz and the old weight columns are staged in shared memory
// with 16-byte loads; G^T is assembled in shared memory and written row by
// row.
constexpr int kHeadBwdThreads = 256;
constexpr int kHB = 64;        // hidden features per CTA
constexpr int kHBGroups = kHeadBwdThreads / kHB;

size_t head_bwd_smem(int B, int C) {
  return sizeof(float) * (2 * static_cast<size_t>(B) * C + static_cast<size_t>(B) * kHB + static_cast<size_t>(C) * kHB +
                          kHBGroups * kHB) +
         sizeof(__nv_bfloat16) * static_cast<size_t>(kHB) * (B + 8);
}

__global__ void __launch_bounds__(kHeadBwdThreads) head_bwd_kernel(const __grid_constant__ HeadArgs a) {
  extern __shared__ __align__(16) float dsm[];
  const int H = a.H, C = a.C, B = a.B;
  float* dz = dsm;                       // [B][C] fp32
  float* dzb = dz + B * C;               // [B][C] bf16-rounded
  float* hs = dzb + B * C;               // [B][kHB] bf16 h as float
  float* wcs = hs + B * kHB;             // [C][kHB] old bf16 weights as float
  float* gbp = wcs + C * kHB;            // [kHBGroups][kHB]
  __nv_bfloat16* gts = reinterpret_cast<__nv_bfloat16*>(gbp + kHBGroups * kHB);  // [kHB][B + 8]
  const int gts_ld = B + 8;
  const int i = blockIdx.x;
  const int w = a.wid[i], src = a.src[i];
  const int k0 = blockIdx.y * kHB;
  const int t = threadIdx.x;
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride;
  const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;
  const float* dl = a.dlog + static_cast<int64_t>(w) * B * C;
  for (int q = t; q < B * C; q += kHeadBwdThreads) {
    const float v = dl[q];
    dz[q] = v;
    dzb[q] = bf16_round(v);
  }
  // h tile: B rows x 64 bf16 = 8 x 16-byte chunks per row
  const __nv_bfloat16* h = a.Ain + static_cast<int64_t>(w) * B * H;
  for (int q = t; q < B * (kHB / 8); q += kHeadBwdThreads) {
    const int b = q >> 3, c8 = (q & 7) * 8;
    float f8[8];
    if (k0 + c8 < H) {
      const uint4 v = *reinterpret_cast<const uint4*>(h + static_cast<int64_t>(b) * H + k0 + c8);
      const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const float2 f = __bfloat1622float2(p2[j]);
        f8[2 * j] = f.x;
        f8[2 * j + 1] = f.y;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 8; ++j) f8[j] = 0.f;
    }
#pragma unroll
    for (int j = 0; j < 8; ++j) hs[b * kHB + c8 + j] = f8[j];
  }
  for (int q = t; q < C * kHB; q += kHeadBwdThreads) {
    const int c = q / kHB, k = q - c * kHB;
    wcs[q] = k0 + k < H ? __bfloat162float(a.shadow[so + a.offW + static_cast<int64_t>(c) * H + k0 + k]) : 0.f;
  }
  __syncthreads();

  // input gradient of the layer below, masked by its ReLU
  {
    const int k = t % kHB, grp = t / kHB;
    const int rows = B / kHBGroups;
    float gsum = 0.f;
    __nv_bfloat16* G = a.G + static_cast<int64_t>(w) * B * H;
    for (int r = 0; r < rows; ++r) {
      const int b = grp * rows + r;
      const float hv = hs[b * kHB + k];
      float dh = 0.f;
      for (int c = 0; c < C; ++c) dh = fmaf(dzb[b * C + c], wcs[c * kHB + k], dh);
      const float g = hv > 0.f ? dh : 0.f;
      gsum += g;
      const __nv_bfloat16 gb16 = __float2bfloat16_rn(g);
      if (k0 + k < H) G[static_cast<int64_t>(b) * H + k0 + k] = gb16;
      gts[k * gts_ld + b] = gb16;
    }
    gbp[grp * kHB + k] = gsum;
  }
  __syncthreads();
  if (t < kHB && k0 + t < H) {
    float g = 0.f;
    for (int grp = 0; grp < kHBGroups; ++grp) g += gbp[grp * kHB + t];
    a.gb[static_cast<int64_t>(w) * H + k0 + t] = g;
  }
  // G^T rows: B bf16 per hidden feature, 16-byte stores
  {
    uint4* GT = reinterpret_cast<uint4*>(a.GT + (static_cast<int64_t>(w) * H + k0) * B);
    const int per_row = B / 8;
    for (int q = t; q < kHB * per_row; q += kHeadBwdThreads) {
      const int k = q / per_row, j = q - k * per_row;
      if (k0 + k < H) GT[static_cast<int64_t>(k) * per_row + j] = *reinterpret_cast<const uint4*>(gts + k * gts_ld + j * 8);
    }
  }
  // weight gradient and SGD of the head
  for (int q = t; q < C * kHB; q += kHeadBwdThreads) {
    const int c = q / kHB, k = q - c * kHB;
    if (k0 + k >= H) continue;
    float dw = 0.f;
    for (int b = 0; b < B; ++b) dw = fmaf(dzb[b * C + c], hs[b * kHB + k], dw);
    const int64_t e = a.offW + static_cast<int64_t>(c) * H + k0 + k;
    const float nw = fmaf(-a.lr, dw, a.master[so + e]);
    a.master_w[dof + e] = nw;
    a.shadow_w[dof + e] = __float2bfloat16_rn(nw);
  }
  if (blockIdx.y == 0 && t < C) {
    float g = 0.f;
    for (int b = 0; b < B; ++b) g += dz[b * C + t];
    a.master_w[dof + a.offB + t] = fmaf(-a.lr, g, a.master[so + a.offB + t]);
  }
}

// ---------------------------------------------------------------- fused head
// Forward and backward of the last layer in one launch, specialised for a
// compile-time class count C.  A cluster of H/128 CTAs serves one active
// lane; CTA r owns hidden features [128 r, 128 r + 128):
//  1. partial logits over its features (tpr threads per row, each over an
//     interleaved set of 4-feature chunks, all C classes in registers);
//  2. cluster barrier; the logits are the partials of ranks 0..n-1 summed in
//     that order from distributed shared memory (so every CTA holds the same
//     values), then the softmax cross-entropy without cancellation;
//  3. a second cluster barrier (no CTA leaves while others read its partials);
//  4. masked input gradient of the layer below for its features: item =
//     (2 features, 8 rows), the 2 x C old weights in registers -> bf16 G
//     (4 bytes per row), G^T (16 bytes per feature) and the fp32 bias
//     gradient;
//  5. head weight gradient + SGD: item = (class, 4 features).
// Rank 0 also writes the loss partials and updates the head bias.
// The h tile stays bf16 in shared memory (about 60 KB per CTA at B = 128),
// so several clusters share an SM and all active lanes run in one wave.
constexpr int kHF = 128;                 // hidden features per CTA
constexpr int kHFThreads = 256;
constexpr int kHFWarps = kHFThreads / 32;
constexpr int kHFMaxCluster = 8;
constexpr int kHFClasses = 10;           // the fused path's class count
constexpr int kHFPairs = kHF / 2;        // phase 4: feature pairs ...
constexpr int kHFRowGroups = kHFThreads / kHFPairs;   // ... x interleaved groups of 8-row blocks

// threads per row in phase 1 and the row stride of the bf16 h tile in
// elements (stride / 2 = 4 (mod 32) words: the 8-byte reads of rows r and
// r + 1 land 4 banks apart, so 8 rows x 2 threads cover the 32 banks once)
__host__ __device__ constexpr int hf_tpr(int B) { return B >= 256 ? 1 : kHFThreads / B; }
constexpr int kHFStride = kHF + 8;

size_t head_fused_smem(int B, int C) {
  return sizeof(__nv_bfloat16) * static_cast<size_t>(B) * kHFStride +
         sizeof(float) * (static_cast<size_t>(C) * kHF + 3 * static_cast<size_t>(B) * C + kHFRowGroups * kHF + B);
}

// 4 bf16 of the h tile as floats
__device__ __forceinline__ float4 hf_ld4(const __nv_bfloat16* p) {
  const uint2 v = *reinterpret_cast<const uint2*>(p);
  const float2 lo = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.x));
  const float2 hi = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&v.y));
  return make_float4(lo.x, lo.y, hi.x, hi.y);
}

template <int C>
__global__ void __launch_bounds__(kHFThreads) head_fused_kernel(const __grid_constant__ HeadArgs a) {
  extern __shared__ __align__(16) float hfsm[];
  const int H = a.H, B = a.B;
  __nv_bfloat16* hs = reinterpret_cast<__nv_bfloat16*>(hfsm);  // [B][kHFStride] bf16 h
  float* wcs = reinterpret_cast<float*>(hs + B * kHFStride);   // [C][kHF] old bf16 head weights as float
  float* pl = wcs + C * kHF;               // [B][C] partial logits (read by the cluster)
  float* dz = pl + B * C;                  // [B][C] logits, then dlogits fp32
  float* dzb = dz + B * C;                 // [B][C] bf16-rounded dlogits
  float* gbp = dzb + B * C;                // [kHFRowGroups][kHF] bias-gradient partials
  float* rowloss = gbp + kHFRowGroups * kHF;   // [B]
  const int i = blockIdx.x;
  const int w = a.wid[i], src = a.src[i];
  const uint32_t rank = cluster_ctarank();
  const int ncl = static_cast<int>(gridDim.y);
  const int k0 = blockIdx.y * kHF;
  const int t = threadIdx.x;
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride;
  const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;
  const __nv_bfloat16* h = a.Ain + static_cast<int64_t>(w) * B * H;

  for (int q = t; q < B * (kHF / 8); q += kHFThreads) {
    const int b = q / (kHF / 8), c8 = (q % (kHF / 8)) * 8;
    *reinterpret_cast<uint4*>(hs + b * kHFStride + c8) =
        *reinterpret_cast<const uint4*>(h + static_cast<int64_t>(b) * H + k0 + c8);
  }
  for (int q = t; q < C * (kHF / 8); q += kHFThreads) {
    const int c = q / (kHF / 8), c8 = (q % (kHF / 8)) * 8;
    const uint4 v = *reinterpret_cast<const uint4*>(a.shadow + so + a.offW + static_cast<int64_t>(c) * H + k0 + c8);
    const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const float2 f = __bfloat1622float2(p2[j]);
      wcs[c * kHF + c8 + 2 * j] = f.x;
      wcs[c * kHF + c8 + 2 * j + 1] = f.y;
    }
  }
  __syncthreads();

  // 1. partial logits
  {
    const int tpr = hf_tpr(B);
    const int rb = t / tpr, q = t % tpr;
    if (rb < B) {
      float acc[C];
#pragma unroll
      for (int c = 0; c < C; ++c) acc[c] = 0.f;
      for (int k = 4 * q; k < kHF; k += 4 * tpr) {
        const float4 hv = hf_ld4(hs + rb * kHFStride + k);
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const float4 wv = *reinterpret_cast<const float4*>(wcs + c * kHF + k);
          acc[c] = fmaf(hv.x, wv.x, acc[c]);
          acc[c] = fmaf(hv.y, wv.y, acc[c]);
          acc[c] = fmaf(hv.z, wv.z, acc[c]);
          acc[c] = fmaf(hv.w, wv.w, acc[c]);
        }
      }
#pragma unroll
      for (int c = 0; c < C; ++c) {
        for (int o = tpr / 2; o > 0; o >>= 1) acc[c] += __shfl_xor_sync(0xffffffffu, acc[c], o);
        if (q == 0) pl[rb * C + c] = acc[c];
      }
    }
  }
  cluster_sync();
  // 2. logits (cluster sum in rank order), softmax cross-entropy
  const float* bias = a.master + so + a.offB;
  for (int q = t; q < B * C; q += kHFThreads) {
    float part[kHFMaxCluster];
#pragma unroll
    for (int r = 0; r < kHFMaxCluster; ++r) part[r] = r < ncl ? ld_dsmem_f32(pl + q, r) : 0.f;
    float acc = 0.f;
#pragma unroll
    for (int r = 0; r < kHFMaxCluster; ++r)
      if (r < ncl) acc += part[r];
    dz[q] = acc + bias[q % C];
  }
  cluster_sync();   // every remote read of pl is done
  for (int b = t; b < B; b += kHFThreads) {
    float z[C];
#pragma unroll
    for (int c = 0; c < C; ++c) z[c] = dz[b * C + c];
    float m = z[0];
#pragma unroll
    for (int c = 1; c < C; ++c) m = fmaxf(m, z[c]);
    const int y = a.labels[static_cast<int64_t>(w) * B + b];
    float e[C], s = 0.f, so_ = 0.f, zy = 0.f;
#pragma unroll
    for (int c = 0; c < C; ++c) {
      e[c] = expf(z[c] - m);
      s += e[c];
      if (c != y) so_ += e[c];
      else zy = z[c];
    }
    rowloss[b] = m + logf(s) - zy;
    const float inv = 1.0f / static_cast<float>(B);
#pragma unroll
    for (int c = 0; c < C; ++c) {
      const float g = (c == y ? -(so_ / s) : e[c] / s) * inv;
      dz[b * C + c] = g;
      dzb[b * C + c] = bf16_round(g);
    }
  }
  __syncthreads();
  if (rank == 0) {
    if (t < B / kRowsPerLossChunk) {
      float l = 0.f;
      for (int r = 0; r < kRowsPerLossChunk; ++r) l += rowloss[t * kRowsPerLossChunk + r];
      const int64_t row = static_cast<int64_t>(w) * a.part_mul + a.part_add;
      a.loss_part[row * (B / kRowsPerLossChunk) + t] = l;
    }
    // head bias: db[c] = sum_b dz[b][c]; 16 threads per class, then shuffles
    if (t < C * 16) {
      const int c = t >> 4, j = t & 15;
      float g = 0.f;
      for (int b = j; b < B; b += 16) g += dz[b * C + c];
#pragma unroll
      for (int o = 8; o > 0; o >>= 1) g += __shfl_xor_sync(0xffffffffu, g, o, 16);
      if (j == 0) a.master_w[dof + a.offB + c] = fmaf(-a.lr, g, a.master[so + a.offB + c]);
    }
  }
  // 4. masked input gradient of the layer below: item = (2 features, 8 rows)
  {
    const int kk = (t % kHFPairs) * 2;     // this thread's 2 features
    const int rg = t / kHFPairs;
    float2 wc[C];
#pragma unroll
    for (int c = 0; c < C; ++c) wc[c] = *reinterpret_cast<const float2*>(wcs + c * kHF + kk);
    float2 gs = make_float2(0.f, 0.f);
    __nv_bfloat16* G = a.G + static_cast<int64_t>(w) * B * H + k0 + kk;
    __nv_bfloat16* GT = a.GT + (static_cast<int64_t>(w) * H + k0 + kk) * B;
    for (int b8 = rg * 8; b8 < B; b8 += kHFRowGroups * 8) {
      uint32_t p0[4], p1[4];               // G^T rows kk and kk + 1 over these 8 rows
#pragma unroll
      for (int r = 0; r < 8; ++r) {
        const int b = b8 + r;
        const float2 hv = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(hs + b * kHFStride + kk));
        float2 dh = make_float2(0.f, 0.f);
#pragma unroll
        for (int c = 0; c < C; ++c) {
          const float g = dzb[b * C + c];
          dh.x = fmaf(g, wc[c].x, dh.x);
          dh.y = fmaf(g, wc[c].y, dh.y);
        }
        dh.x = hv.x > 0.f ? dh.x : 0.f;
        dh.y = hv.y > 0.f ? dh.y : 0.f;
        gs.x += dh.x;
        gs.y += dh.y;
        const __nv_bfloat162 pr = __floats2bfloat162_rn(dh.x, dh.y);
        *reinterpret_cast<__nv_bfloat162*>(G + static_cast<int64_t>(b) * H) = pr;
        const uint32_t lo = __bfloat16_as_ushort(pr.x), hi = __bfloat16_as_ushort(pr.y);
        if (r & 1) {
          p0[r >> 1] |= lo << 16;
          p1[r >> 1] |= hi << 16;
        } else {
          p0[r >> 1] = lo;
          p1[r >> 1] = hi;
        }
      }
      *reinterpret_cast<uint4*>(GT + b8) = make_uint4(p0[0], p0[1], p0[2], p0[3]);
      *reinterpret_cast<uint4*>(GT + B + b8) = make_uint4(p1[0], p1[1], p1[2], p1[3]);
    }
    *reinterpret_cast<float2*>(gbp + rg * kHF + kk) = gs;
  }
  __syncthreads();
  if (t < kHF) {
    float g = 0.f;
#pragma unroll
    for (int r = 0; r < kHFRowGroups; ++r) g += gbp[r * kHF + t];
    a.gb[static_cast<int64_t>(w) * H + k0 + t] = g;
  }
  // 5. head weight gradient + SGD: item = (class, 4 features)
  for (int q = t; q < C * (kHF / 4); q += kHFThreads) {
    const int c = q / (kHF / 4), k4 = (q % (kHF / 4)) * 4;
    float4 dw = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int b = 0; b < B; ++b) {
      const float g = dzb[b * C + c];
      const float4 hv = hf_ld4(hs + b * kHFStride + k4);
      dw.x = fmaf(g, hv.x, dw.x);
      dw.y = fmaf(g, hv.y, dw.y);
      dw.z = fmaf(g, hv.z, dw.z);
      dw.w = fmaf(g, hv.w, dw.w);
    }
    const int64_t e = a.offW + static_cast<int64_t>(c) * H + k0 + k4;
    const float4 o = *reinterpret_cast<const float4*>(a.master + so + e);
    float4 nw;
    nw.x = fmaf(-a.lr, dw.x, o.x);
    nw.y = fmaf(-a.lr, dw.y, o.y);
    nw.z = fmaf(-a.lr, dw.z, o.z);
    nw.w = fmaf(-a.lr, dw.w, o.w);
    *reinterpret_cast<float4*>(a.master_w + dof + e) = nw;
    *reinterpret_cast<uint2*>(a.shadow_w + dof + e) = make_uint2(pack_bf16x2(nw.x, nw.y), pack_bf16x2(nw.z, nw.w));
  }
}

// ---------------------------------------------------------------- bookkeeping
__global__ void loss_finalize_kernel(const float* part, const int32_t* tau, int W, int max_tau,
                                     int nc, int B, float* loss) {
  const int w = blockIdx.x * blockDim.x + threadIdx.x;
  if (w >= W) return;
  double s = 0.0;
  const int t = tau[w];
  for (int st = 0; st < t; ++st)
    for (int c = 0; c < nc; ++c) s += part[(static_cast<int64_t>(w) * max_tau + st) * nc + c];
  loss[w] = static_cast<float>(s / (static_cast<double>(B) * t));
}

__global__ void sum_scaled_kernel(const float* part, int64_t count, double scale, float* out) {
  __shared__ double red[256];
  double s = 0.0;
  for (int64_t i = threadIdx.x; i < count; i += blockDim.x) s += part[i];
  red[threadIdx.x] = s;
  __syncthreads();
  for (int o = 128; o > 0; o >>= 1) {
    if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
    __syncthreads();
  }
  if (threadIdx.x == 0) out[0] = static_cast<float>(red[0] * scale);
}

__global__ void cursor_advance_kernel(int64_t* cursor, const int32_t* tau, const int64_t* n, int B, int W) {
  const int w = blockIdx.x * blockDim.x + threadIdx.x;
  if (w < W) cursor[w] = (cursor[w] + static_cast<int64_t>(tau[w]) * B) % n[w];
}

__global__ void shadow_refresh_kernel(const float* __restrict__ m, __nv_bfloat16* __restrict__ s, int64_t count) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count; i += stride)
    s[i] = __float2bfloat16_rn(m[i]);
}

// dst[c][r] = src[r][c] for a rows x cols bf16 matrix
__global__ void transpose_bf16_kernel(const __nv_bfloat16* __restrict__ src, __nv_bfloat16* __restrict__ dst,
                                      int rows, int cols) {
  __shared__ __nv_bfloat16 t[32][34];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int r = ty; r < 32; r += 8)
    if (r0 + r < rows && c0 + tx < cols) t[r][tx] = src[static_cast<int64_t>(r0 + r) * cols + c0 + tx];
  __syncthreads();
  for (int c = ty; c < 32; c += 8)
    if (c0 + c < cols && r0 + tx < rows) dst[static_cast<int64_t>(c0 + c) * rows + r0 + tx] = t[tx][c];
}

__global__ void broadcast_kernel(const float* __restrict__ xg, float* __restrict__ slab, int64_t stride, int W,
                                 int64_t count) {
  const int64_t gs = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count; i += gs) {
    const float v = xg[i];
    for (int k = 0; k < W; ++k) slab[static_cast<int64_t>(k) * stride + i] = v;
  }
}

}  // namespace

cudaError_t launch_stage(const StageArgs& a, int n_active, cudaStream_t s) {
  dim3 grid((a.D + 31) / 32, (a.B + 31) / 32, n_active);
  stage_kernel<<<grid, 256, 0, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_stage_round_priority(const StageArgs& a, const int32_t* tau, int W, int max_tau, int priority,
                                        cudaStream_t s) {
  if (a.D % 4 != 0 || a.B % 16 != 0) return cudaErrorInvalidValue;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((a.D + kStageCols - 1) / kStageCols, (a.B + kStageRows - 1) / kStageRows,
                     a.slots ? a.n_slots : W * max_tau);
  cfg.blockDim = dim3(256, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributePriority;
  attr[0].val.priority = priority;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, stage_round_kernel, a, tau, W);
}

cudaError_t launch_stage_round_strided(const StageArgs& a, const int32_t* tau, int W, int max_tau, int blocks,
                                       int priority, cudaStream_t s) {
  if (a.D % 4 != 0 || a.B % 16 != 0 || blocks < 1) return cudaErrorInvalidValue;
  const int nx = (a.D + kStageCols - 1) / kStageCols, ny = (a.B + kStageRows - 1) / kStageRows;
  const int nz = a.slots ? a.n_slots : W * max_tau;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(blocks), 1, 1);
  cfg.blockDim = dim3(256, 1, 1);
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributePriority;
  attr[0].val.priority = priority;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, stage_round_strided_kernel, a, tau, W, nx, ny, nz);
}

cudaError_t launch_stage_round(const StageArgs& a, const int32_t* tau, int W, int max_tau, cudaStream_t s) {
  if (a.D % 4 != 0 || a.B % 16 != 0) return cudaErrorInvalidValue;
  dim3 grid((a.D + kStageCols - 1) / kStageCols, (a.B + kStageRows - 1) / kStageRows, a.slots ? a.n_slots : W * max_tau);
  stage_round_kernel<<<grid, 256, 0, s>>>(a, tau, W);
  return cudaGetLastError();
}

cudaError_t launch_head_fwd(const HeadArgs& a, int n_active, cudaStream_t s) {
  if (a.H % 8 != 0 || a.H > 32 * 8 * kHeadMaxH8) return cudaErrorInvalidValue;
  const size_t smem = sizeof(float) * static_cast<size_t>(a.C) * a.H;
  cudaError_t e = cudaFuncSetAttribute(head_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(n_active, a.B / kRowsPerLossChunk);
  head_fwd_kernel<<<grid, kHeadFwdThreads, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_head_bwd(const HeadArgs& a, int n_active, cudaStream_t s) {
  if (a.B % (8 * kHBGroups) != 0 || a.H % 8 != 0) return cudaErrorInvalidValue;
  const size_t smem = head_bwd_smem(a.B, a.C);
  cudaError_t e = cudaFuncSetAttribute(head_bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(n_active, (a.H + kHB - 1) / kHB);
  head_bwd_kernel<<<grid, kHeadBwdThreads, smem, s>>>(a);
  return cudaGetLastError();
}

bool head_fused_supported(int H, int B, int C) {
  return C == kHFClasses && H % kHF == 0 && H / kHF <= kHFMaxCluster && B % 32 == 0 && B <= 256 &&
         head_fused_smem(B, C) <= 220 * 1024;
}

cudaError_t launch_head_fused(const HeadArgs& a, int n_active, cudaStream_t s) {
  if (!head_fused_supported(a.H, a.B, a.C)) return cudaErrorInvalidValue;
  const size_t smem = head_fused_smem(a.B, a.C);
  cudaError_t e = cudaFuncSetAttribute(head_fused_kernel<kHFClasses>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_active, a.H / kHF, 1);
  cfg.blockDim = dim3(kHFThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = 1;
  attr[0].val.clusterDim.y = a.H / kHF;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, head_fused_kernel<kHFClasses>, a);
}

cudaError_t launch_loss_finalize(const float* part, const int32_t* tau, int W, int max_tau, int nc, int B,
                                 float* loss, cudaStream_t s) {
  loss_finalize_kernel<<<(W + 63) / 64, 64, 0, s>>>(part, tau, W, max_tau, nc, B, loss);
  return cudaGetLastError();
}

cudaError_t launch_sum_scaled(const float* part, int64_t count, double scale, float* out, cudaStream_t s) {
  sum_scaled_kernel<<<1, 256, 0, s>>>(part, count, scale, out);
  return cudaGetLastError();
}

cudaError_t launch_cursor_advance(int64_t* cursor, const int32_t* tau, const int64_t* n, int B, int W,
                                  cudaStream_t s) {
  cursor_advance_kernel<<<(W + 63) / 64, 64, 0, s>>>(cursor, tau, n, B, W);
  return cudaGetLastError();
}

cudaError_t launch_shadow_refresh(const float* master, __nv_bfloat16* shadow, int64_t count, cudaStream_t s) {
  int64_t blocks = (count + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) return cudaSuccess;
  shadow_refresh_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(master, shadow, count);
  return cudaGetLastError();
}

cudaError_t launch_transpose_bf16(const __nv_bfloat16* src, __nv_bfloat16* dst, int rows, int cols,
                                  cudaStream_t s) {
  dim3 grid((cols + 31) / 32, (rows + 31) / 32);
  transpose_bf16_kernel<<<grid, 256, 0, s>>>(src, dst, rows, cols);
  return cudaGetLastError();
}

cudaError_t launch_broadcast(const float* xg, float* slab, int64_t stride, int W, int64_t count,
                             cudaStream_t s) {
  int64_t blocks = (count + 255) / 256;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) return cudaSuccess;
  broadcast_kernel<<<static_cast<unsigned>(blocks), 256, 0, s>>>(xg, slab, stride, W, count);
  return cudaGetLastError();
}

}  // namespace oscars
