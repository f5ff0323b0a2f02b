// evisel_selftest_wait: runs the kernels' bounded mbarrier wait on a barrier
// that is (arrive = 0) or is not (arrive = 1) left incomplete, so that a test
// can check that a stuck wait ends as an EVISEL_ETIMEOUT status the host reads,
// with the device still usable. Nothing here faults or traps.
#include <cstdint>
#include <string>

#include <cuda_runtime.h>

#include "../../include/evisel.h"
#include "evisel_internal.h"
#include "sm103_ptx.cuh"

namespace evisel {
int set_last_error(int code, const char* msg);
void clear_last_error();
}

using namespace evisel;

static __device__ int g_selftest_status;

namespace {

__global__ void selftest_wait_kernel(uint64_t timeout_ns, int arrive) {
  __shared__ uint64_t bar_word;
  __shared__ int abort_flag;
  const uint32_t bar = ptx::smem_addr(&bar_word);
  if (threadIdx.x == 0) {
    ptx::mbar_init(bar, 1);
    abort_flag = 0;
    ptx::fence_mbar_init();
  }
  __syncwarp();
  if (arrive && threadIdx.x == 0) ptx::mbar_arrive(bar);
  __syncwarp();
  const bool ok = ptx::mbar_wait(bar, 0, &abort_flag, timeout_ns);
  if (__all_sync(0xffffffffu, ok)) {
    if (threadIdx.x == 0) g_selftest_status = EVISEL_OK;
  } else if (threadIdx.x == 0) {
    g_selftest_status = kStatusTimeout;
  }
}

}  // namespace

extern "C" int evisel_selftest_wait(int timeout_us, int arrive, void* stream_ptr, int* device_status) {
  clear_last_error();
  if (timeout_us < 1 || timeout_us > 1000000) return set_last_error(EVISEL_EINVAL, "timeout_us must be in [1, 1e6]");
  if (!device_status) return set_last_error(EVISEL_EINVAL, "device_status is NULL");
  cudaStream_t stream = static_cast<cudaStream_t>(stream_ptr);
  const int unset = 1;   // neither EVISEL_OK nor an error code: the kernel must overwrite it
  cudaError_t e = cudaMemcpyToSymbolAsync(g_selftest_status, &unset, sizeof(int), 0, cudaMemcpyHostToDevice, stream);
  if (e == cudaSuccess) {
    selftest_wait_kernel<<<1, 32, 0, stream>>>(static_cast<uint64_t>(timeout_us) * 1000u, arrive != 0);
    e = cudaGetLastError();
  }
  if (e == cudaSuccess) e = cudaStreamSynchronize(stream);
  if (e == cudaSuccess) e = cudaMemcpyFromSymbol(device_status, g_selftest_status, sizeof(int));
  if (e != cudaSuccess) {
    cudaGetLastError();
    return set_last_error(EVISEL_ECUDA, (std::string("selftest: ") + cudaGetErrorString(e)).c_str());
  }
  return EVISEL_OK;
}
