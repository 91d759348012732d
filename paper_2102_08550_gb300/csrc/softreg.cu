// Local steps of softmax regression in fp32 (one linear layer + softmax
// cross-entropy): Eq. 4, "otherwise" branch, x <- x - lr * g(x) with g the
// mean mini-batch gradient.
//
// Each worker's whole round runs in one launch: the worker pulls the global
// model into shared memory (the pull of the parameter-server description,
// fused: nothing is copied through HBM), runs tau_i SGD steps on successive
// mini-batches of its shard with the weights resident in shared memory, and
// writes the result to the worker's replica (the push).  Workers never
// exchange data inside a round.  Two kernels: softreg_cluster_round_kernel
// puts each worker on a cluster of 8 CTAs that split the input columns (the
// round kernel of a context, batch <= 256); softreg_round_kernel puts each
// worker on one CTA (larger batches, and the allocation-free entry point).
//
// Per step: logits z[b][c] = sum_k x[b][k] W[c][k] + bias[c] (warp-level dot
// products), p = softmax(z), loss_b = logsumexp(z_b) - z_b[y_b],
// dz = (p - onehot(y)) / B, dW[c][k] = sum_b dz[b][c] x[b][k],
// db[c] = sum_b dz[b][c], W <- W - lr dW (fmaf), all fp32.
#include "common.cuh"
#include "internal.h"

namespace oscars {

namespace {

constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
static_assert(kSoftregMaxBatch <= kThreads, "one thread per mini-batch row");

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// float4 items of one mini-batch a thread holds in registers while the
// previous step computes (the next step's rows are loaded ahead)
constexpr int kPrefetch = 16;

// Round bookkeeping of worker w at the end of its round: the mean loss over
// its tau steps (the step partials summed in step order in double, divided
// by B tau) and the data cursor advanced by tau mini-batches.
__device__ __forceinline__ void finish_worker(const SoftregArgs& a, int w, int tau, int64_t cur, int64_t n) {
  if (a.loss_out) {
    double sum = 0.0;
    for (int st = 0; st < tau; ++st) sum += a.loss_part[static_cast<int64_t>(w) * a.max_tau + st];
    a.loss_out[w] = static_cast<float>(sum / (static_cast<double>(a.B) * tau));
  }
  if (a.cursor_next) a.cursor_next[w] = (cur + static_cast<int64_t>(tau) * a.B) % n;
}

__global__ void __launch_bounds__(kThreads) softreg_round_kernel(const __grid_constant__ SoftregArgs a) {
  extern __shared__ __align__(16) float sm[];
  const int D = a.D, C = a.C, B = a.B;
  float* Wsm = sm;                 // [C][D]
  float* bsm = Wsm + C * D;        // [C] (padded to 32)
  float* Xsm = bsm + 32;           // [B][D]
  float* Zsm = Xsm + B * D;        // [B][C] logits, then dz
  float* Lsm = Zsm + B * C;        // [B] per-sample loss
  int* Ysm = reinterpret_cast<int*>(Lsm + B);  // [B]
  int64_t* Rsm = reinterpret_cast<int64_t*>((reinterpret_cast<uintptr_t>(Ysm + B) + 7) & ~uintptr_t(7));   // [B] row offsets

  const int w = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int tau = a.tau[w];
  const float* gsrc = a.master + static_cast<int64_t>(a.global_slot) * a.slot_stride;
  float* dst = a.master_out + static_cast<int64_t>(w) * a.slot_stride;

  // pull: global model -> shared memory
  for (int i = tid; i < C * D; i += kThreads) Wsm[i] = gsrc[a.offW + i];
  for (int i = tid; i < C; i += kThreads) bsm[i] = gsrc[a.offB + i];

  const float* X = a.shard_x[w];
  const int32_t* Y = a.shard_y[w];
  const int64_t n = a.shard_n[w];
  const int64_t cur = a.cursor[w];
  const float invB = 1.0f / static_cast<float>(B);
  // with D % 4 == 0, a 16-byte aligned shard and a mini-batch of at most
  // kPrefetch float4 per thread, step s + 1's rows are loaded into registers
  // while step s computes (otherwise rows are read one float at a time)
  const int D4 = D / 4;
  const bool vec = (D & 3) == 0 && (reinterpret_cast<uintptr_t>(X) & 15) == 0 && B * D4 <= kPrefetch * kThreads;
  float4 pf[kPrefetch];
  auto fetch = [&](int s) {   // rows of step s into registers (row offsets already in Rsm)
#pragma unroll
    for (int j = 0; j < kPrefetch; ++j) {
      const int i = tid + j * kThreads;
      if (i < B * D4) {
        const int b = i / D4, k4 = i - b * D4;
        pf[j] = *reinterpret_cast<const float4*>(X + Rsm[b] + 4 * k4);
      }
    }
  };
  auto row_offsets = [&](int s) {
    if (tid < B) {
      const int64_t r = (cur + static_cast<int64_t>(s) * B + tid) % n;
      Rsm[tid] = r * D;
      Ysm[tid] = Y[r];
    }
  };
  if (vec && tau > 0) {
    row_offsets(0);
    __syncthreads();
    fetch(0);
  }

  for (int s = 0; s < tau; ++s) {
    __syncthreads();   // the previous step is done with Xsm and Zsm
    int yl = 0;        // the label of row tid (tid < B) of this step
    if (vec) {
      // this step's rows, fetched during the previous step; then the next
      // step's row offsets and labels (thread tid rewrites only entry tid,
      // which it alone has read) and its rows, in flight during this step
      if (tid < B) yl = Ysm[tid];
#pragma unroll
      for (int j = 0; j < kPrefetch; ++j) {
        const int i = tid + j * kThreads;
        if (i < B * D4) reinterpret_cast<float4*>(Xsm)[i] = pf[j];
      }
      if (s + 1 < tau) row_offsets(s + 1);
      __syncthreads();
      if (s + 1 < tau) fetch(s + 1);
    } else {
      // mini-batch rows (cursor + s*B + b) mod n
      row_offsets(s);
      __syncthreads();
      for (int i = tid; i < B * D; i += kThreads) {
        const int b = i / D, k = i - b * D;
        Xsm[i] = X[Rsm[b] + k];
      }
      if (tid < B) yl = Ysm[tid];
      __syncthreads();
    }
    // logits: one warp per (b, c) dot product
    for (int q = warp; q < B * C; q += kWarps) {
      const int b = q / C, c = q - b * C;
      const float* xr = Xsm + b * D;
      const float* wr = Wsm + c * D;
      float acc = 0.f;
      if ((D & 3) == 0) {
        for (int k4 = lane; k4 < D4; k4 += 32) {
          const float4 xv = reinterpret_cast<const float4*>(xr)[k4];
          const float4 wv = reinterpret_cast<const float4*>(wr)[k4];
          acc = fmaf(xv.x, wv.x, acc);
          acc = fmaf(xv.y, wv.y, acc);
          acc = fmaf(xv.z, wv.z, acc);
          acc = fmaf(xv.w, wv.w, acc);
        }
      } else {
        for (int k = lane; k < D; k += 32) acc = fmaf(xr[k], wr[k], acc);
      }
      acc = warp_sum(acc);
      if (lane == 0) Zsm[q] = acc + bsm[c];
    }
    __syncthreads();
    // softmax cross-entropy, one thread per row
    if (tid < B) {
      const int b = tid;
      float* z = Zsm + b * C;
      float m = z[0];
      for (int c = 1; c < C; ++c) m = fmaxf(m, z[c]);
      // p_c = e_c / s; 1 - p_y = (sum_{c != y} e_c) / s (no cancellation)
      const int y = yl;
      float se = 0.f, so = 0.f;
      for (int c = 0; c < C; ++c) {
        const float e = expf(z[c] - m);
        se += e;
        if (c != y) so += e;
      }
      Lsm[b] = m + logf(se) - z[y];
      for (int c = 0; c < C; ++c) z[c] = (c == y ? -(so / se) : expf(z[c] - m) / se) * invB;
    }
    __syncthreads();
    if (tid == 0) {
      float l = 0.f;
      for (int b = 0; b < B; ++b) l += Lsm[b];
      a.loss_part[static_cast<int64_t>(w) * a.max_tau + s] = l;
    }
    // weight gradient and update: item = (class, 4 input features) (or one
    // feature when D % 4 != 0)
    if ((D & 3) == 0) {
      for (int q = tid; q < C * D4; q += kThreads) {
        const int c = q / D4, k4 = q - c * D4;
        float4 g = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int b = 0; b < B; ++b) {
          const float d = Zsm[b * C + c];
          const float4 xv = reinterpret_cast<const float4*>(Xsm + b * D)[k4];
          g.x = fmaf(d, xv.x, g.x);
          g.y = fmaf(d, xv.y, g.y);
          g.z = fmaf(d, xv.z, g.z);
          g.w = fmaf(d, xv.w, g.w);
        }
        float4* wp = reinterpret_cast<float4*>(Wsm + c * D) + k4;
        float4 wv = *wp;
        wv.x = fmaf(-a.lr, g.x, wv.x);
        wv.y = fmaf(-a.lr, g.y, wv.y);
        wv.z = fmaf(-a.lr, g.z, wv.z);
        wv.w = fmaf(-a.lr, g.w, wv.w);
        *wp = wv;
      }
    } else {
      for (int k = tid; k < D; k += kThreads) {
        for (int c = 0; c < C; ++c) {
          float g = 0.f;
          for (int b = 0; b < B; ++b) g = fmaf(Zsm[b * C + c], Xsm[b * D + k], g);
          Wsm[c * D + k] = fmaf(-a.lr, g, Wsm[c * D + k]);
        }
      }
    }
    for (int c = tid; c < C; c += kThreads) {
      float g = 0.f;
      for (int b = 0; b < B; ++b) g += Zsm[b * C + c];
      bsm[c] = fmaf(-a.lr, g, bsm[c]);
    }
  }
  __syncthreads();
  // push: replica <- shared memory
  for (int i = tid; i < C * D; i += kThreads) dst[a.offW + i] = Wsm[i];
  for (int i = tid; i < C; i += kThreads) dst[a.offB + i] = bsm[i];
  if (tid == 0) finish_worker(a, w, tau, cur, n);   // the thread that wrote the loss partials
}

// The same round with each worker on a cluster of kCl CTAs that split the
// input columns: CTA r owns columns [r * Dc, min(D, (r + 1) * Dc)) (Dc a
// multiple of 4) of W and of every mini-batch row, so a step's work and the
// shared memory it needs are divided by kCl.  Per step each CTA computes the
// partial logits of the whole mini-batch over its columns; after one cluster
// barrier every CTA sums the kCl partials in rank order (distributed shared
// memory loads) and adds the bias, and runs the softmax cross-entropy of every
// row itself (identical arithmetic in every CTA); then it updates its own
// columns of W, and its private copy of the bias (the same update in every
// CTA; rank 0 writes it back).  The partial logits are double-buffered by
// step parity: a CTA rewrites a buffer two steps later, after a barrier that
// every reader of the buffer has passed.
constexpr int kCl = 8;
constexpr int kClThreads = 256;
// columns per CTA: D / kCl rounded up to a multiple of 4
__host__ __device__ inline int cluster_cols(int D) { return ((D + kCl - 1) / kCl + 3) / 4 * 4; }
constexpr int kClPrefetch = 8;   // float4 items of the next step's rows held per thread

__global__ void __launch_bounds__(kClThreads) softreg_cluster_round_kernel(const __grid_constant__ SoftregArgs a) {
  extern __shared__ __align__(16) float sm[];
  const int D = a.D, C = a.C, B = a.B;
  const int Dc = cluster_cols(D);
  const int rank = static_cast<int>(cluster_ctarank());
  const int c0 = rank * Dc;
  const int nc = D - c0 < Dc ? (D - c0 > 0 ? D - c0 : 0) : Dc;   // this CTA's columns (may be 0)
  float* Wsm = sm;                       // [C][Dc]
  float* bsm = Wsm + C * Dc;             // [32]
  float* Xsm = bsm + 32;                 // [B][Dc]
  float* Psm = Xsm + B * Dc;             // [2][B][C] partial logits, by step parity
  float* Zsm = Psm + 2 * B * C;          // [B][C] logits, then dz
  float* Lsm = Zsm + B * C;              // [B]
  int* Ysm = reinterpret_cast<int*>(Lsm + B);   // [B]
  int64_t* Rsm = reinterpret_cast<int64_t*>((reinterpret_cast<uintptr_t>(Ysm + B) + 7) & ~uintptr_t(7));  // [B]

  const int w = blockIdx.y;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int tau = a.tau[w];
  const float* gsrc = a.master + static_cast<int64_t>(a.global_slot) * a.slot_stride;
  float* dst = a.master_out + static_cast<int64_t>(w) * a.slot_stride;
  const float* X = a.shard_x[w];
  const int32_t* Y = a.shard_y[w];
  const int64_t n = a.shard_n[w];
  const int64_t cur = a.cursor[w];
  const float invB = 1.0f / static_cast<float>(B);
  const int nc4 = nc / 4;

  // pull: this CTA's columns of the global model, and the whole bias
  for (int i = tid; i < C * Dc; i += kClThreads) {
    const int c = i / Dc, k = i - c * Dc;
    Wsm[i] = k < nc ? gsrc[a.offW + static_cast<int64_t>(c) * D + c0 + k] : 0.f;
  }
  for (int i = tid; i < C; i += kClThreads) bsm[i] = gsrc[a.offB + i];

  // rows of step s: (cursor + s*B + b) mod n; this CTA's columns of each,
  // as 16-byte loads when every row's slice is 16-byte aligned
  const bool vec = (D & 3) == 0 && (reinterpret_cast<uintptr_t>(X) & 15) == 0 && B * nc4 <= kClPrefetch * kClThreads;
  float4 pf[kClPrefetch];
  auto row_offsets = [&](int s) {
    if (tid < B) {
      const int64_t r = (cur + static_cast<int64_t>(s) * B + tid) % n;
      Rsm[tid] = r * D + c0;
      Ysm[tid] = Y[r];
    }
  };
  auto fetch = [&]() {
#pragma unroll
    for (int j = 0; j < kClPrefetch; ++j) {
      const int i = tid + j * kClThreads;
      if (i < B * nc4) {
        const int b = i / nc4, k4 = i - b * nc4;
        pf[j] = *reinterpret_cast<const float4*>(X + Rsm[b] + 4 * k4);
      }
    }
  };
  if (vec && tau > 0) {
    row_offsets(0);
    __syncthreads();
    fetch();
  }

  for (int s = 0; s < tau; ++s) {
    float* Pp = Psm + (s & 1) * B * C;
    __syncthreads();   // the previous step is done with Xsm and Zsm
    int yl = 0;
    if (vec) {
      if (tid < B) yl = Ysm[tid];
#pragma unroll
      for (int j = 0; j < kClPrefetch; ++j) {
        const int i = tid + j * kClThreads;
        if (i < B * nc4) {
          const int b = i / nc4, k4 = i - b * nc4;
          reinterpret_cast<float4*>(Xsm + b * Dc)[k4] = pf[j];
        }
      }
      if (s + 1 < tau) row_offsets(s + 1);
      __syncthreads();
      if (s + 1 < tau) fetch();
    } else {
      row_offsets(s);
      __syncthreads();
      for (int i = tid; i < B * nc; i += kClThreads) {
        const int b = i / nc, k = i - b * nc;
        Xsm[b * Dc + k] = X[Rsm[b] + k];
      }
      if (tid < B) yl = Ysm[tid];
      __syncthreads();
    }
    // partial logits over this CTA's columns: one thread per (row, class)
    for (int q = tid; q < B * C; q += kClThreads) {
      const int b = q / C, c = q - b * C;
      const float* xr = Xsm + b * Dc;
      const float* wr = Wsm + c * Dc;
      float acc = 0.f;
      if ((nc & 3) == 0) {
        for (int k4 = 0; k4 < nc4; ++k4) {
          const float4 xv = reinterpret_cast<const float4*>(xr)[k4];
          const float4 wv = reinterpret_cast<const float4*>(wr)[k4];
          acc = fmaf(xv.x, wv.x, acc);
          acc = fmaf(xv.y, wv.y, acc);
          acc = fmaf(xv.z, wv.z, acc);
          acc = fmaf(xv.w, wv.w, acc);
        }
      } else {
        for (int k = 0; k < nc; ++k) acc = fmaf(xr[k], wr[k], acc);
      }
      Pp[q] = acc;
    }
    cluster_sync();
    // logits: the partials of every CTA in rank order, then the bias
    for (int q = tid; q < B * C; q += kClThreads) {
      float part[kCl];
#pragma unroll
      for (int r = 0; r < kCl; ++r) part[r] = ld_dsmem_f32(Pp + q, r);
      float acc = 0.f;
#pragma unroll
      for (int r = 0; r < kCl; ++r) acc += part[r];
      Zsm[q] = acc + bsm[q % C];
    }
    __syncthreads();
    // softmax cross-entropy, one thread per row
    if (tid < B) {
      float* z = Zsm + tid * C;
      float m = z[0];
      for (int c = 1; c < C; ++c) m = fmaxf(m, z[c]);
      const int y = yl;
      float se = 0.f, so = 0.f;
      for (int c = 0; c < C; ++c) {
        const float e = expf(z[c] - m);
        se += e;
        if (c != y) so += e;
      }
      Lsm[tid] = m + logf(se) - z[y];
      for (int c = 0; c < C; ++c) z[c] = (c == y ? -(so / se) : expf(z[c] - m) / se) * invB;
    }
    __syncthreads();
    if (rank == 0 && warp == 0) {   // the step's loss: rows summed in order
      if (lane == 0) {
        float l = 0.f;
        for (int b = 0; b < B; ++b) l += Lsm[b];
        a.loss_part[static_cast<int64_t>(w) * a.max_tau + s] = l;
      }
    }
    // weight gradient and update of this CTA's columns: item = (class, 4 columns)
    if ((nc & 3) == 0) {
      for (int q = tid; q < C * nc4; q += kClThreads) {
        const int c = q / nc4, k4 = q - c * nc4;
        float4 g = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int b = 0; b < B; ++b) {
          const float d = Zsm[b * C + c];
          const float4 xv = reinterpret_cast<const float4*>(Xsm + b * Dc)[k4];
          g.x = fmaf(d, xv.x, g.x);
          g.y = fmaf(d, xv.y, g.y);
          g.z = fmaf(d, xv.z, g.z);
          g.w = fmaf(d, xv.w, g.w);
        }
        float4* wp = reinterpret_cast<float4*>(Wsm + c * Dc) + k4;
        float4 wv = *wp;
        wv.x = fmaf(-a.lr, g.x, wv.x);
        wv.y = fmaf(-a.lr, g.y, wv.y);
        wv.z = fmaf(-a.lr, g.z, wv.z);
        wv.w = fmaf(-a.lr, g.w, wv.w);
        *wp = wv;
      }
    } else {
      for (int q = tid; q < C * nc; q += kClThreads) {
        const int c = q / nc, k = q - c * nc;
        float g = 0.f;
        for (int b = 0; b < B; ++b) g = fmaf(Zsm[b * C + c], Xsm[b * Dc + k], g);
        Wsm[c * Dc + k] = fmaf(-a.lr, g, Wsm[c * Dc + k]);
      }
    }
    for (int c = tid; c < C; c += kClThreads) {   // the bias, the same update in every CTA
      float g = 0.f;
      for (int b = 0; b < B; ++b) g += Zsm[b * C + c];
      bsm[c] = fmaf(-a.lr, g, bsm[c]);
    }
  }
  __syncthreads();
  // push: this CTA's columns into the replica (rank 0 also the bias)
  for (int i = tid; i < C * nc; i += kClThreads) {
    const int c = i / nc, k = i - c * nc;
    dst[a.offW + static_cast<int64_t>(c) * D + c0 + k] = Wsm[c * Dc + k];
  }
  if (rank == 0)
    for (int i = tid; i < C; i += kClThreads) dst[a.offB + i] = bsm[i];
  cluster_sync();   // no CTA leaves while a peer may still read its partial logits
  // every CTA has read the cursor; rank 0's thread 0 wrote the loss partials
  if (rank == 0 && tid == 0) finish_worker(a, w, tau, cur, n);
}

// Mean cross-entropy of the global model: one warp per sample, partial sums
// per block (summed afterwards in a fixed order).
__global__ void __launch_bounds__(256) softreg_eval_kernel(const __grid_constant__ SoftregEvalArgs a) {
  __shared__ float part[8];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float mine = 0.f;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * 8 + warp; i < a.n; i += static_cast<int64_t>(gridDim.x) * 8) {
    const float* xr = a.x + i * a.D;
    float z[kMaxClasses];
    for (int c = 0; c < a.C; ++c) {
      const float* wr = a.master + a.offW + static_cast<int64_t>(c) * a.D;
      float acc = 0.f;
      for (int k = lane; k < a.D; k += 32) acc = fmaf(xr[k], wr[k], acc);
      z[c] = warp_sum(acc) + a.master[a.offB + c];
    }
    float m = z[0];
    for (int c = 1; c < a.C; ++c) m = fmaxf(m, z[c]);
    float se = 0.f;
    for (int c = 0; c < a.C; ++c) se += expf(z[c] - m);
    mine += m + logf(se) - z[a.y[i]];
  }
  if (lane == 0) part[warp] = mine;
  __syncthreads();
  if (threadIdx.x == 0) {
    float s = 0.f;
    for (int i = 0; i < 8; ++i) s += part[i];
    a.loss_sum[blockIdx.x] = s;
  }
}

}  // namespace

size_t softreg_smem_bytes(int D, int C, int B) {
  return sizeof(float) * (static_cast<size_t>(C) * D + 32 + static_cast<size_t>(B) * D +
                          static_cast<size_t>(B) * C + B) +
         sizeof(int) * B + 8 + sizeof(int64_t) * B;
}

cudaError_t launch_softreg_round(const SoftregArgs& a, int W, cudaStream_t s) {
  const size_t smem = softreg_smem_bytes(a.D, a.C, a.B);
  cudaError_t e = cudaFuncSetAttribute(softreg_round_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  softreg_round_kernel<<<W, kThreads, smem, s>>>(a);
  return cudaGetLastError();
}

int softreg_cluster_cols(int D) { return cluster_cols(D); }

size_t softreg_cluster_smem_bytes(int D, int C, int B) {
  const size_t Dc = static_cast<size_t>(softreg_cluster_cols(D));
  return sizeof(float) * (C * Dc + 32 + static_cast<size_t>(B) * Dc + 3 * static_cast<size_t>(B) * C + B) +
         sizeof(int) * B + 8 + sizeof(int64_t) * B;
}

bool softreg_cluster_supported(int D, int C, int B) {
  return B <= kClThreads && softreg_cluster_smem_bytes(D, C, B) <= 200 * 1024;
}

cudaError_t launch_softreg_cluster_round(const SoftregArgs& a, int W, cudaStream_t s) {
  const size_t smem = softreg_cluster_smem_bytes(a.D, a.C, a.B);
  cudaError_t e = cudaFuncSetAttribute(softreg_cluster_round_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(smem));
  if (e != cudaSuccess) return e;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kCl, W, 1);
  cfg.blockDim = dim3(kClThreads, 1, 1);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr;
  attr.id = cudaLaunchAttributeClusterDimension;
  attr.val.clusterDim.x = kCl;
  attr.val.clusterDim.y = 1;
  attr.val.clusterDim.z = 1;
  cfg.attrs = &attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, softreg_cluster_round_kernel, a);
}

cudaError_t launch_softreg_eval(const SoftregEvalArgs& a, int blocks, cudaStream_t s) {
  softreg_eval_kernel<<<blocks, 256, 0, s>>>(a);
  return cudaGetLastError();
}

}  // namespace oscars
