// Self-test of the library's failure detection: every wait a kernel here makes
// (on an mbarrier, or on a flag another CTA sets in global memory) is bounded,
// and a wait that runs out records SP_DEVERR_TIMEOUT in the caller's error word
// and returns instead of spinning.  This kernel runs the same two wait helpers
// the path's kernels use, with a caller-given short limit, on an mbarrier and a
// flag that nothing completes (unless the caller asks the kernel to complete
// them itself first), so that the timeout path can be exercised on a GPU
// without a hang.
#include "common.cuh"
#include "internal.h"

namespace sp {

namespace {

__global__ void wait_probe_kernel(const int* __restrict__ flag, uint64_t limit_ns, int complete, int* out,
                                  int* err) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  fence_mbar_init();
  if (complete) mbar_arrive(&bar);
  out[0] = mbar_wait(&bar, 0, err, limit_ns) ? 1 : 0;
  out[1] = wait_flag(flag, err, limit_ns) ? 1 : 0;
}

}  // namespace

}  // namespace sp

using namespace sp;

extern "C" {

sp_status sp_wait_probe(const int* flag, unsigned int limit_us, int complete, int* out, int* err, sp_stream stream) {
  if (!flag || !out) return report(SP_ERR_INVALID_ARG, "sp_wait_probe: flag and out are required");
  if (limit_us < 1 || limit_us > 2000000u) return report(SP_ERR_SHAPE, "sp_wait_probe: limit_us in 1..2,000,000");
  wait_probe_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(flag, (uint64_t)limit_us * 1000ull, complete ? 1 : 0, out,
                                                          err);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return report(SP_ERR_CUDA, "sp_wait_probe: %s", cudaGetErrorString(e));
  return SP_OK;
}

}  // extern "C"
