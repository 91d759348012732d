// One worker's fp32 softmax-regression local steps without any device
// allocation: the same round kernel as oscars_local_steps runs with its
// global scratch (the one-worker argument tables and the per-step loss
// partials) placed in a fixed array that the library reserves when it is
// loaded.
//
// Who needs this: a caller that must not allocate device memory at the point
// of the call.  Examples: code running while a CUDA graph is being captured
// (cudaMalloc is not allowed in a global-mode capture), a host framework
// whose own pool owns all device memory and forbids side allocations, and a
// latency-critical loop that cannot afford cudaMalloc/cudaFree, which may
// synchronise the device.
//
// The scratch array is a file-scope __device__ variable, so every GPU that
// loads the library holds kScratchBytes of it until the process exits.  In
// host code its name is only a host-side stand-in: the device address is
// looked up once per device with cudaGetSymbolAddress and cached.
#include <mutex>

#include "../../include/oscars.h"
#include "common.cuh"
#include "internal.h"

namespace oscars {
namespace {

constexpr size_t kScratchBytes = 64 * 1024;   // 64 KB per device
constexpr size_t kTableBytes = 256;           // argument tables at the front
constexpr int kMaxSteps = static_cast<int>((kScratchBytes - kTableBytes) / sizeof(float));
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// one-worker argument tables, written by noalloc_setup_kernel
struct Tables {
  const float* x;
  const int32_t* y;
  int64_t n;
  int64_t cursor;
  int32_t tau;
};
static_assert(sizeof(Tables) <= kTableBytes, "tables must fit the reserved front of the scratch");

__global__ void noalloc_setup_kernel(const float* x, const int32_t* y, int64_t n, int64_t cursor, int32_t tau) {
  Tables* t = reinterpret_cast<Tables*>(g_noalloc_scratch);
  t->x = x;
  t->y = y;
  t->n = n;
  t->cursor = cursor;
  t->tau = tau;
}

std::mutex g_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch on the current device (set-up on first use).
cudaError_t scratch_address(void** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace oscars

using namespace oscars;

extern "C" oscars_status oscars_softreg_steps_noalloc(const float* params_in, float* params_out, const float* x,
                                                      const int32_t* y, int64_t n, int64_t cursor, int32_t tau,
                                                      int32_t dim, int32_t classes, int32_t batch, float lr,
                                                      float* loss_out, void* stream) {
  if (!params_in || !params_out || !x || !y || !loss_out) return OSCARS_EINVAL;
  if (n < 1 || cursor < 0 || dim < 1 || batch < 1 || classes < 2 || classes > kMaxClasses) return OSCARS_EINVAL;
  if (tau < 1 || tau > kMaxSteps) return OSCARS_EINVAL;   // beyond the fixed scratch
  if (batch > kSoftregMaxBatch) return OSCARS_ENOTSUP;
  if (softreg_smem_bytes(dim, classes, batch) > 220 * 1024) return OSCARS_ENOTSUP;
  void* base = nullptr;
  if (scratch_address(&base) != cudaSuccess) return OSCARS_ECUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  unsigned char* sc = static_cast<unsigned char*>(base);
  Tables* t = reinterpret_cast<Tables*>(sc);
  float* loss_part = reinterpret_cast<float*>(sc + kTableBytes);

  noalloc_setup_kernel<<<1, 1, 0, s>>>(x, y, n, cursor, tau);
  if (cudaGetLastError() != cudaSuccess) return OSCARS_ECUDA;
  SoftregArgs a;
  a.master = params_in;        // source model: slot 0 with stride 0
  a.master_out = params_out;   // the one CTA (worker 0) writes here
  a.slot_stride = 0;
  a.global_slot = 0;
  a.offW = 0;
  a.offB = static_cast<int64_t>(classes) * dim;
  a.D = dim;
  a.C = classes;
  a.B = batch;
  a.lr = lr;
  a.tau = &t->tau;
  a.shard_x = &t->x;
  a.shard_y = &t->y;
  a.shard_n = &t->n;
  a.cursor = &t->cursor;
  a.loss_part = loss_part;     // every entry s < tau is written before it is read
  a.max_tau = tau;
  if (launch_softreg_round(a, 1, s) != cudaSuccess) return OSCARS_ECUDA;
  if (launch_loss_finalize(loss_part, &t->tau, 1, tau, 1, batch, loss_out, s) != cudaSuccess) return OSCARS_ECUDA;
  return OSCARS_OK;
}
