// Diagnostic kernels of libturnopd.

#include "common.cuh"
#include "kernels.h"
#include "ptx.cuh"

namespace turnopd {
namespace {

// One CTA polls, with the bounded try_wait loop the kernels use, an mbarrier that
// nothing arrives on; after `limit` polls it records TURNOPD_ERR_TIMEOUT and
// returns.  The loop is bounded and the CTA holds nothing else, so it always ends.
__global__ void k_wait_selftest(uint32_t limit, int32_t *status)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0)
        mbar_init(&bar, 1);
    __syncthreads();
    uint32_t it = 0;
    while (!mbar_try_wait(&bar, 0) && ++it < limit) {
    }
    if (it >= limit && threadIdx.x == 0)
        set_status(status, TURNOPD_ERR_TIMEOUT);
}

}  // namespace

cudaError_t launch_wait_selftest(uint32_t limit, int32_t *status, cudaStream_t stream)
{
    k_wait_selftest<<<1, 32, 0, stream>>>(limit, status);
    return cudaGetLastError();
}

}  // namespace turnopd
