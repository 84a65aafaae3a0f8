// Self-test of the bounded device waits: one thread waits on an mbarrier
// that nothing arrives on, through the same mbar_wait every tensor-core
// kernel uses, with a caller-chosen limit. When the limit passes, the wait
// records MLA_ERR_TIMEOUT in the device status word and the kernel returns,
// so the host sees the timeout and the context stays usable.
#include "internal.h"
#include "ptx_sm103.cuh"

namespace vmla {
namespace {

__global__ void bounded_wait_selftest_kernel(unsigned long long limit_ns, int* status) {
  __shared__ __align__(8) uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x != 0) return;
  mbar_init(&bar, 1);
  abort_flag = 0;
  fence_mbar_init();
  const WaitCtx wc{&abort_flag, status};
  mbar_wait(&bar, 0, wc, limit_ns);  // nothing arrives: returns after limit_ns
}

}  // namespace

int launch_wait_selftest(unsigned long long limit_ns, int* status, cudaStream_t stream) {
  bounded_wait_selftest_kernel<<<1, 32, 0, stream>>>(limit_ns, status);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) {
    set_last_cuda_error(e);
    return MLA_ERR_CUDA;
  }
  return MLA_OK;
}

}  // namespace vmla
