// Test-only kernel for the library's bounded in-kernel wait (mbar_wait in
// dmc_internal.cuh). The test builds it with a shortened DMC_WAIT_LIMIT_NS:
// waiting on an mbarrier that nobody arrives at must give up after the limit,
// set DMC_FAULT_WAIT_TIMEOUT and return false; with the one expected arrival
// made first, the same wait must succeed at once. No tensor-core work runs.
#include "dmc_internal.cuh"

__global__ void wait_probe_kernel(int arrive_first, unsigned int* err, int* ok,
                                  unsigned long long* ns) {
  __shared__ __align__(8) uint64_t bar;
  const uint32_t b = dmc::smem_u32(&bar);
  if (threadIdx.x == 0) {
    dmc::mbar_init(b, 1);
    dmc::fence_mbar_init();
  }
  __syncthreads();
  if (arrive_first && threadIdx.x == 0) dmc::mbar_arrive(b);
  __syncthreads();
  const uint64_t t0 = dmc::globaltimer_ns();
  const bool done = dmc::mbar_wait(b, 0, err);  // phase 0 completes only with the arrival
  const uint64_t t1 = dmc::globaltimer_ns();
  ok[threadIdx.x] = done ? 1 : 0;
  if (threadIdx.x == 0) *ns = t1 - t0;
}

extern "C" int dmc_wait_probe(int arrive_first, int threads, unsigned int* err_dev, int* ok_dev,
                              unsigned long long* ns_dev, cudaStream_t stream) {
  if (threads < 1 || threads > 1024) return (int)cudaErrorInvalidValue;
  wait_probe_kernel<<<1, threads, 0, stream>>>(arrive_first, err_dev, ok_dev, ns_dev);
  return (int)cudaGetLastError();
}
