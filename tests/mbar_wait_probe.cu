// Test probe (not part of libedp): the bounded mbarrier wait that the staged
// frame-stack delivery uses, run on its own.  One thread initialises an
// mbarrier expecting one arrival and waits for phase 0 with a time limit:
// first with nothing arriving (the wait must give up after about the limit
// and report false), then after its own arrival (true at once).  Times are
// read from %globaltimer.
#include <cuda_runtime.h>
#include <stdint.h>

#include "edp_internal.cuh"

__global__ void k_mbar_wait_probe(uint64_t limit_ns, unsigned long long *out) {
  __shared__ unsigned long long bar;
  if (threadIdx.x != 0) return;
  edp::mbar_init(&bar, 1);
  edp::mbar_init_fence();
  const uint64_t t0 = edp::global_ns();
  const bool got = edp::mbar_wait(&bar, 0, limit_ns);  // nothing arrives
  const uint64_t t1 = edp::global_ns();
  edp::mbar_arrive(&bar);                              // completes phase 0
  const bool got2 = edp::mbar_wait(&bar, 0, limit_ns);
  const uint64_t t2 = edp::global_ns();
  out[0] = got;
  out[1] = t1 - t0;
  out[2] = got2;
  out[3] = t2 - t1;
}

// out: device unsigned long long [4] = (first wait succeeded, its ns,
// second wait succeeded, its ns).  Returns a cudaError_t.
extern "C" int mbar_wait_probe(uint64_t limit_ns, unsigned long long *out) {
  k_mbar_wait_probe<<<1, 32>>>(limit_ns, out);
  cudaError_t e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  return (int)e;
}
