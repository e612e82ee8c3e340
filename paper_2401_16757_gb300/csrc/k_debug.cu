// Failure-detection probe (a test hook, not part of the inference path):
// one kernel whose bounded device wait runs out, so that tests can check on
// the GPU that a wait which never completes is reported as a timeout and
// leaves the context usable, without faulting or hanging the device.
#include <cuda_runtime.h>

#include <string>

#include "device.cuh"
#include "internal.h"
#include "kernels.h"

namespace swapnet {

namespace {
// Failure-detection probe: one thread waits, with the kernels' bounded wait,
// on an mbarrier that nothing ever completes; the wait gives up after the
// limit, records the timeout in the error word and the kernel returns.
__global__ void wait_timeout_probe_kernel(int* err) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  abort_flag = 0;
  mbar_init(smem_u32(&bar), 1);
  fence_barrier_init();
  mbar_wait_bounded(smem_u32(&bar), 0, &abort_flag, err);
}
}  // namespace

}  // namespace swapnet

extern "C" int swapnet_debug_wait_timeout(swapnet_stream stream) {
  return swapnet::guard_abi([&]() -> int {
    using namespace swapnet;
    int* err = nullptr;
    int rc = tc_error_word(&err);
    if (rc) return rc;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    wait_timeout_probe_kernel<<<1, 32, 0, s>>>(err);
    int w = 0;
    const int zero = 0;
    cudaError_t ce = cudaGetLastError();
    if (ce == cudaSuccess) ce = cudaStreamSynchronize(s);
    if (ce == cudaSuccess) ce = cudaMemcpy(&w, err, sizeof(int), cudaMemcpyDeviceToHost);
    if (ce == cudaSuccess) ce = cudaMemcpy(err, &zero, sizeof(int), cudaMemcpyHostToDevice);
    if (ce != cudaSuccess) SN_FAIL(SWAPNET_ERR_CUDA, std::string("timeout probe: ") + cudaGetErrorString(ce));
    if (w == kDevErrTimeout) SN_FAIL(SWAPNET_ERR_TIMEOUT, "a device-side wait gave up (probe)");
    if (w) SN_FAIL(SWAPNET_ERR_CUDA, "unexpected error word from the probe");
    return SWAPNET_OK;
  });
}
