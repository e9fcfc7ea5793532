// The bf16 row path's entry: the row grids of rowkl_cluster.cuh for vocabularies that
// are a multiple of 8.  Other vocabularies take the same kernels compiled with a
// masked last vector, in their own translation unit (rowkl_cluster_tail.cu), so that
// neither set slows the other's build or changes its code.

#include "rowkl_cluster.cuh"

namespace turnopd {

cudaError_t launch_row_cluster(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used)
{
    if (p.vocab % 8 != 0)
        return launch_row_cluster_tail(p, fp32_grad, stream, used);
    return launch_row_cluster_t<false>(p, fp32_grad, stream, used);
}

}  // namespace turnopd
