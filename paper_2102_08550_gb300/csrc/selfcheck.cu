// A wait that runs out on purpose, through the same bounded mbarrier wait and
// device error word as the round kernels: one thread waits on an mbarrier
// that nothing completes, for a given number of polls, records its code in
// the error word and returns.  The host then reads the error word as after a
// round.  This exercises the failure path of every kernel wait (the error is
// reported, the kernel ends, the context stays usable) without a fault.
#include "common.cuh"
#include "internal.h"

namespace oscars {
namespace {

__global__ void wait_selfcheck_kernel(int* err, uint32_t polls) {
  __shared__ __align__(8) uint64_t bar;
  mbar_init(&bar, 1);   // one arrival expected, none will come
  fence_barrier_init();
  mbar_wait(&bar, 0, err, kDevTimeoutCheck, polls);
}

}  // namespace

cudaError_t launch_wait_selfcheck(int* err, uint32_t polls, cudaStream_t s) {
  wait_selfcheck_kernel<<<1, 1, 0, s>>>(err, polls);
  return cudaGetLastError();
}

}  // namespace oscars
