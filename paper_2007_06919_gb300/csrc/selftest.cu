// selftest.cu -- exercises the device-side failure path of the library's kernels without
// faulting anything: the bounded mbarrier wait (tc_ptx.cuh) that every tensor-core kernel
// uses, on a barrier that nobody arrives at, so that it expires, latches kStatusTimeout in
// the device status word through fail(), and lets a second role unwind through the shared
// abort flag, as the roles of conv_tc_kernel do. Every wait is bounded; the kernel returns.
#include <cuda_runtime.h>

#include <string>

#include "common.cuh"
#include "kernels.h"
#include "tc_ptx.cuh"

namespace aqd {
namespace tc {

constexpr uint64_t kSelfTestLimitNs = 2000000ull;  // 2 ms: the short wait that must expire

// out[0]: 1 if role 0's short wait expired (returned false); out[1]: its wait in ns.
// out[2]: 1 if role 1's 1 s wait returned false; out[3]: its wait in ns (well under 1 s when
// it left through the abort flag). out[4]: 1 if the control barrier that did complete was
// seen as complete.
__global__ void __launch_bounds__(64, 1) wait_selftest_kernel(uint32_t* status, int64_t* out) {
  __shared__ __align__(8) uint64_t bars[3];
  __shared__ volatile int abort_flag;
  const uint32_t b_never0 = smem_u32(&bars[0]);
  const uint32_t b_never1 = smem_u32(&bars[1]);
  const uint32_t b_done = smem_u32(&bars[2]);
  if (threadIdx.x == 0) {
    mbar_init(b_never0, 1);
    mbar_init(b_never1, 1);
    mbar_init(b_done, 1);
    abort_flag = 0;
    fence_barrier_init();
  }
  __syncthreads();
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  if (warp == 0 && lane == 0) {
    // control: a barrier whose phase completes is seen as complete by the same wait
    mbar_arrive(b_done);
    out[4] = mbar_wait<kSelfTestLimitNs>(b_done, 0, &abort_flag) ? 1 : 0;
    const uint64_t t0 = globaltimer();
    const bool ok = mbar_wait<kSelfTestLimitNs>(b_never0, 0, &abort_flag);
    out[1] = (int64_t)(globaltimer() - t0);
    out[0] = ok ? 0 : 1;
    if (!ok) fail(&abort_flag, status);
  } else if (warp == 1 && lane == 0) {
    const uint64_t t0 = globaltimer();
    const bool ok = mbar_wait(b_never1, 0, &abort_flag);  // the kernels' 1 s limit
    out[3] = (int64_t)(globaltimer() - t0);
    out[2] = ok ? 0 : 1;
  }
}

}  // namespace tc

int launch_wait_selftest(uint32_t* status, int64_t* out, cudaStream_t stream, std::string* err) {
  tc::wait_selftest_kernel<<<1, 64, 0, stream>>>(status, out);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) { *err = std::string("wait self-test launch: ") + cudaGetErrorString(e); return 3; }
  return 0;
}

}  // namespace aqd
