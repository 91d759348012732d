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
__global__ void __launch_bounds__(256) stage_kernel(const __grid_constant__ StageArgs a) {
  __shared__ __nv_bfloat16 tile[32][34];
  const int w = a.wid[blockIdx.z];
  const int k0 = blockIdx.x * 32, b0 = blockIdx.y * 32;
  const float* X = a.x[w];
  const int64_t n = a.n[w];
  const int64_t base = a.start[w] + a.row_add;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;  // 32 x 8
  __nv_bfloat16* A0 = a.A0 + static_cast<int64_t>(w) * a.B * a.D;
  __nv_bfloat16* A0T = a.A0T + static_cast<int64_t>(w) * a.B * a.D;
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
    if (b < a.B) a.labels[static_cast<int64_t>(w) * a.B + b] = a.y[w][(base + b) % n];
  }
}

// ---------------------------------------------------------------- head forward
// Logits of the last layer z[b][c] = sum_k bf16(h[b][k]) bf16(W[c][k]) + bias[c]
// (fp32 accumulate), softmax cross-entropy, dlogits = (p - onehot)/B.
// Grid (active lanes, B/16); 16 rows per CTA, one warp per two rows.
constexpr int kHeadFwdThreads = 256;

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
  for (int q = threadIdx.x; q < C * H; q += kHeadFwdThreads) Wsm[q] = __bfloat162float(Wg[q]);
  __syncthreads();
  for (int rr = warp; rr < kRowsPerLossChunk; rr += kHeadFwdThreads / 32) {
    const int b = blockIdx.y * kRowsPerLossChunk + rr;
    const __nv_bfloat16* h = a.Ain + (static_cast<int64_t>(w) * B + b) * H;
    float zc = -INFINITY;  // lane c holds z_c
    for (int c = 0; c < C; ++c) {
      const float* wr = Wsm + c * H;
      float acc = 0.f;
      for (int k = lane; k < H; k += 32) acc = fmaf(__bfloat162float(h[k]), wr[k], acc);
      acc = warp_sum(acc) + bias[c];
      if (lane == c) zc = acc;
    }
    const float m = warp_max(zc);
    const float e = lane < C ? expf(zc - m) : 0.f;
    const float lse = m + logf(warp_sum(e));
    const int y = a.labels[static_cast<int64_t>(w) * B + b];
    const float zy = __shfl_sync(0xffffffffu, zc, y);
    if (lane < C) {
      const float p = expf(zc - lse);
      a.dlog[(static_cast<int64_t>(w) * B + b) * C + lane] = (p - (lane == y ? 1.f : 0.f)) / static_cast<float>(B);
    }
    if (lane == 0) rowloss[rr] = lse - zy;
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
// One thread per hidden feature k (grid: active lanes, H/128):
//  dW[c][k] = sum_b bf16(dz[b][c]) bf16(h[b][k]);  W <- W - lr dW (fmaf);
//  dh[b][k] = sum_c bf16(dz[b][c]) bf16(W_old[c][k]);  g = dh * (h > 0)
//  -> G [B][H] and GT [H][B] in bf16 (operands of the next GEMMs) and
//  gb[k] = sum_b g (fp32, the bias gradient of the layer below).
// CTA column 0 also updates the head bias with db[c] = sum_b dz[b][c].
constexpr int kHeadBwdThreads = 128;

__global__ void __launch_bounds__(kHeadBwdThreads) head_bwd_kernel(const __grid_constant__ HeadArgs a) {
  extern __shared__ __align__(16) float dsm[];
  const int H = a.H, C = a.C, B = a.B;
  float* dz = dsm;             // [B][C] fp32
  float* dzb = dz + B * C;     // [B][C] bf16-rounded
  const int i = blockIdx.x;
  const int w = a.wid[i], src = a.src[i];
  const float* dl = a.dlog + static_cast<int64_t>(w) * B * C;
  for (int q = threadIdx.x; q < B * C; q += kHeadBwdThreads) {
    const float v = dl[q];
    dz[q] = v;
    dzb[q] = bf16_round(v);
  }
  __syncthreads();
  const int64_t so = static_cast<int64_t>(src) * a.slot_stride;
  const int64_t dof = static_cast<int64_t>(w) * a.slot_stride;
  if (blockIdx.y == 0 && threadIdx.x < C) {
    const int c = threadIdx.x;
    float g = 0.f;
    for (int b = 0; b < B; ++b) g += dz[b * C + c];
    a.master_w[dof + a.offB + c] = fmaf(-a.lr, g, a.master[so + a.offB + c]);
  }
  const int k = blockIdx.y * kHeadBwdThreads + threadIdx.x;
  if (k >= H) return;
  // fully unrolled over kMaxClasses so both arrays stay in registers
  float wc[kMaxClasses], dw[kMaxClasses];
#pragma unroll
  for (int c = 0; c < kMaxClasses; ++c) {
    wc[c] = c < C ? __bfloat162float(a.shadow[so + a.offW + static_cast<int64_t>(c) * H + k]) : 0.f;
    dw[c] = 0.f;
  }
  const __nv_bfloat16* h = a.Ain + static_cast<int64_t>(w) * B * H;
  __nv_bfloat16* G = a.G + static_cast<int64_t>(w) * B * H;
  uint4* GT = reinterpret_cast<uint4*>(a.GT + (static_cast<int64_t>(w) * H + k) * B);
  float gb = 0.f;
  uint32_t pk[4];
  for (int b = 0; b < B; ++b) {
    const float hv = __bfloat162float(h[static_cast<int64_t>(b) * H + k]);
    float dh = 0.f;
#pragma unroll
    for (int c = 0; c < kMaxClasses; ++c) {
      if (c < C) {
        const float g = dzb[b * C + c];
        dw[c] = fmaf(g, hv, dw[c]);
        dh = fmaf(g, wc[c], dh);
      }
    }
    const float gv = hv > 0.f ? dh : 0.f;
    gb += gv;
    const __nv_bfloat16 gbv = __float2bfloat16_rn(gv);
    G[static_cast<int64_t>(b) * H + k] = gbv;
    const uint32_t bits = static_cast<uint32_t>(*reinterpret_cast<const uint16_t*>(&gbv));
    const int slot = (b & 7) >> 1;
    if ((b & 1) == 0) pk[slot] = bits; else pk[slot] |= bits << 16;
    if ((b & 7) == 7) GT[b >> 3] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
  }
  a.gb[static_cast<int64_t>(w) * H + k] = gb;
#pragma unroll
  for (int c = 0; c < kMaxClasses; ++c) {
    if (c < C) {
      const int64_t e = a.offW + static_cast<int64_t>(c) * H + k;
      const float nw = fmaf(-a.lr, dw[c], a.master[so + e]);
      a.master_w[dof + e] = nw;
      a.shadow_w[dof + e] = __float2bfloat16_rn(nw);
    }
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

cudaError_t launch_head_fwd(const HeadArgs& a, int n_active, cudaStream_t s) {
  const size_t smem = sizeof(float) * static_cast<size_t>(a.C) * a.H;
  cudaError_t e = cudaFuncSetAttribute(head_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(n_active, a.B / kRowsPerLossChunk);
  head_fwd_kernel<<<grid, kHeadFwdThreads, smem, s>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_head_bwd(const HeadArgs& a, int n_active, cudaStream_t s) {
  const size_t smem = sizeof(float) * 2 * static_cast<size_t>(a.B) * a.C;
  cudaError_t e = cudaFuncSetAttribute(head_bwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  dim3 grid(n_active, (a.H + kHeadBwdThreads - 1) / kHeadBwdThreads);
  head_bwd_kernel<<<grid, kHeadBwdThreads, smem, s>>>(a);
  return cudaGetLastError();
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
