// Server merge and global update (Eq. 4, first branch; the parameter-server
// push / combine / pull of the Introduction), delta form:
//
//   x_g[p] <- x_g[p] + eta_s * sum_k w_k * delta_k[p],
//   delta_k = pushed delta, or x^k[p] - x_g[p] for pushed replicas.
//
// HBM-bound streaming kernel: every byte of the W pushed buffers is read
// once with 16-byte streaming loads (ld.global.cs: evict-first, they are
// never reused), the sum is kept in fp32 registers in worker order
// k = 0..W-1, and x_g is read and written once.  Algorithmic traffic:
// (W + 2) * P * 4 bytes.  The pointer table and weights travel in a
// __grid_constant__ parameter block, so each thread only loads data.
//
// In MLP mode the same pass also writes the bf16 operand copy of x_g.
//
// Grid: persistent, (SM count) x 3 blocks of 224 threads striding over
// 16-byte chunks; each thread keeps 16 independent 16-byte loads in flight
// per group of 16 workers (the rest in groups of 8, 4, 2 and 1), still
// summing in worker order.
//
// Alignment: the vector kernel needs every buffer at the same offset modulo
// 16 bytes.  When they share one offset that is not 0, the first (up to 3)
// elements are peeled off to the scalar kernel and the vector kernel starts
// at the first 16-byte boundary; only buffers with different offsets fall
// back to the scalar kernel for the whole vector.
#include <atomic>

#include "common.cuh"
#include "internal.h"

namespace oscars {

namespace {

// 7 warps and 3 resident blocks per SM: the launch bounds cap a thread at 96
// registers, enough for 16 float4 loads in flight (without the cap the
// compiler picks 32 registers for full occupancy and the loads of a thread
// run one after the other); 672 threads per SM cover the 407 K-parameter
// model of the 784-512-10 MLP in one wave
constexpr int kThreads = 224;
constexpr int kMinBlocks = 3;
constexpr int kGroup = 16;   // replica loads in flight per thread before the first is used

__device__ __forceinline__ float4 ld_stream4(const float4* p) { return __ldcs(p); }

// Workers [k, k + G) of 16-byte chunk i added to acc in worker order: all G
// loads are issued before the first is used, so a thread keeps G of them in
// flight (the kernel's launch bounds leave it the registers for 16).
template <int G, bool kReplica>
__device__ __forceinline__ void merge_group(const MergeArgs& a, int k, int64_t i, const float4& x, float4& acc) {
  float4 v[G];
#pragma unroll
  for (int j = 0; j < G; ++j) v[j] = ld_stream4(reinterpret_cast<const float4*>(a.src[k + j]) + i);
#pragma unroll
  for (int j = 0; j < G; ++j) {
    const float w = a.w[k + j];
    if (kReplica) {
      acc.x = fmaf(w, v[j].x - x.x, acc.x);
      acc.y = fmaf(w, v[j].y - x.y, acc.y);
      acc.z = fmaf(w, v[j].z - x.z, acc.z);
      acc.w = fmaf(w, v[j].w - x.w, acc.w);
    } else {
      acc.x = fmaf(w, v[j].x, acc.x);
      acc.y = fmaf(w, v[j].y, acc.y);
      acc.z = fmaf(w, v[j].z, acc.z);
      acc.w = fmaf(w, v[j].w, acc.w);
    }
  }
}

template <bool kReplica, bool kShadow>
__global__ void __launch_bounds__(kThreads, kMinBlocks) merge_vec4_kernel(const __grid_constant__ MergeArgs a,
                                                                          float* __restrict__ x_g, int64_t n4,
                                                                          float eta, __nv_bfloat16* __restrict__ shadow) {
  float4* xg4 = reinterpret_cast<float4*>(x_g);
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
    const float4 x = __ldcs(xg4 + i);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    int k = 0;
    for (; k + kGroup <= a.W; k += kGroup) merge_group<kGroup, kReplica>(a, k, i, x, acc);
    // the rest in groups of 8, 4, 2 and 1, still in worker order
    if (k + 8 <= a.W) {
      merge_group<8, kReplica>(a, k, i, x, acc);
      k += 8;
    }
    if (k + 4 <= a.W) {
      merge_group<4, kReplica>(a, k, i, x, acc);
      k += 4;
    }
    if (k + 2 <= a.W) {
      merge_group<2, kReplica>(a, k, i, x, acc);
      k += 2;
    }
    if (k < a.W) merge_group<1, kReplica>(a, k, i, x, acc);
    float4 out;
    out.x = fmaf(eta, acc.x, x.x);
    out.y = fmaf(eta, acc.y, x.y);
    out.z = fmaf(eta, acc.z, x.z);
    out.w = fmaf(eta, acc.w, x.w);
    __stcs(xg4 + i, out);
    if (kShadow)   // the bf16 operand copy of the new global model, same pass
      reinterpret_cast<uint2*>(shadow)[i] = make_uint2(pack_bf16x2(out.x, out.y), pack_bf16x2(out.z, out.w));
  }
}

// Any alignment: one element per thread and iteration, over the elements
// [0, head) and [tail, P) (the peeled head and the tail of the vector
// kernel, or head = tail = 0 for the whole vector).
template <bool kReplica>
__global__ void __launch_bounds__(kThreads) merge_scalar_kernel(const __grid_constant__ MergeArgs a,
                                                                float* __restrict__ x_g,
                                                                int64_t head, int64_t tail, int64_t P, float eta,
                                                                __nv_bfloat16* __restrict__ shadow) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  const int64_t count = head + (P - tail);
  for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < count; q += stride) {
    const int64_t p = q < head ? q : tail + (q - head);
    const float x = x_g[p];
    float acc = 0.f;
    for (int k = 0; k < a.W; ++k) {
      const float v = __ldcs(a.src[k] + p);
      acc = fmaf(a.w[k], kReplica ? v - x : v, acc);
    }
    const float out = fmaf(eta, acc, x);
    x_g[p] = out;
    if (shadow) shadow[p] = __float2bfloat16_rn(out);
  }
}

constexpr int kMaxDevices = 64;
std::atomic<int> g_sm_count[kMaxDevices];

// SM count of the current device (queried once per device)
int sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
  if (dev >= kMaxDevices) {
    int n = 0;
    return cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess && n > 0 ? n : 1;
  }
  int n = g_sm_count[dev].load(std::memory_order_relaxed);
  if (n == 0) {
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 1;
    g_sm_count[dev].store(n, std::memory_order_relaxed);
  }
  return n;
}

}  // namespace

cudaError_t launch_merge(const MergeArgs& a, float* x_g, int64_t P, float eta, bool replica,
                         cudaStream_t s, __nv_bfloat16* shadow) {
  if (P <= 0) return cudaSuccess;
  // elements before the first 16-byte boundary of x_g; the vector kernel
  // runs from there when every buffer has the same offset modulo 16 bytes
  // (and the bf16 copy, two bytes per element, is then 8-byte aligned)
  const uintptr_t off = reinterpret_cast<uintptr_t>(x_g) & 15;
  bool vec = (off & 3) == 0;
  int64_t head = vec ? static_cast<int64_t>((16 - off) & 15) / 4 : 0;
  if (head > P) head = P;
  for (int k = 0; k < a.W && vec; ++k) vec = (reinterpret_cast<uintptr_t>(a.src[k]) & 15) == off;
  if (vec && shadow) vec = (reinterpret_cast<uintptr_t>(shadow + head) & 7) == 0;
  const int ctas_per_sm = kMinBlocks;
  const int64_t n4 = vec ? (P - head) / 4 : 0;
  if (n4 == 0) head = 0;
  if (n4 > 0) {
    MergeArgs av = a;   // the same buffers from the first 16-byte boundary on
    for (int k = 0; k < a.W; ++k) av.src[k] = a.src[k] + head;
    float* xv = x_g + head;
    __nv_bfloat16* sv = shadow ? shadow + head : nullptr;
    int64_t blocks = static_cast<int64_t>(sm_count()) * ctas_per_sm;
    const int64_t need = (n4 + kThreads - 1) / kThreads;
    if (need < blocks) blocks = need;
    const unsigned nb = static_cast<unsigned>(blocks);
    if (replica && shadow)
      merge_vec4_kernel<true, true><<<nb, kThreads, 0, s>>>(av, xv, n4, eta, sv);
    else if (replica)
      merge_vec4_kernel<true, false><<<nb, kThreads, 0, s>>>(av, xv, n4, eta, nullptr);
    else if (shadow)
      merge_vec4_kernel<false, true><<<nb, kThreads, 0, s>>>(av, xv, n4, eta, sv);
    else
      merge_vec4_kernel<false, false><<<nb, kThreads, 0, s>>>(av, xv, n4, eta, nullptr);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  const int64_t tail = head + n4 * 4;
  if (head > 0 || tail < P) {
    int64_t blocks = static_cast<int64_t>(sm_count()) * ctas_per_sm;
    const int64_t need = (head + (P - tail) + kThreads - 1) / kThreads;
    if (need < blocks) blocks = need;
    const unsigned nb = static_cast<unsigned>(blocks);
    if (replica)
      merge_scalar_kernel<true><<<nb, kThreads, 0, s>>>(a, x_g, head, tail, P, eta, shadow);
    else
      merge_scalar_kernel<false><<<nb, kThreads, 0, s>>>(a, x_g, head, tail, P, eta, shadow);
    return cudaGetLastError();
  }
  return cudaSuccess;
}

}  // namespace oscars
