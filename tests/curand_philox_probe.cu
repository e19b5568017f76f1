// Test infrastructure: cuRAND's device Philox4_32_10 through its public API,
// for cross-checking the oracle's Philox4x32-10.  curand_init(seed,
// subsequence, offset) positions the generator `offset` values into
// subsequence `subsequence`; with offset = 4 * j, curand4 returns the
// block of counter (j lo, j hi, subsequence lo, subsequence hi) under key
// (seed lo, seed hi).
#include <cuda_runtime.h>
#include <curand_kernel.h>
#include <stdint.h>

__global__ void k_probe(const unsigned long long *seed, const unsigned long long *subseq,
                        const unsigned long long *offset, unsigned n, uint4 *out) {
  const unsigned i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  curandStatePhilox4_32_10_t st;
  curand_init(seed[i], subseq[i], offset[i], &st);
  out[i] = curand4(&st);
}

extern "C" int curand_philox_probe(const unsigned long long *seed,
                                   const unsigned long long *subseq,
                                   const unsigned long long *offset, unsigned n,
                                   uint4 *out) {
  k_probe<<<(n + 127) / 128, 128>>>(seed, subseq, offset, n, out);
  if (cudaGetLastError() != cudaSuccess) return 1;
  return cudaDeviceSynchronize() == cudaSuccess ? 0 : 2;
}
