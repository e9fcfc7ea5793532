// The bf16 row grids of rowkl_cluster.cuh for a vocabulary that is not a multiple of
// 8: the row's last vector is masked in the statistics and written column by column.

#include "rowkl_cluster.cuh"

namespace turnopd {

cudaError_t launch_row_cluster_tail(const RowIn &p, bool fp32_grad, cudaStream_t stream, bool *used)
{
    return launch_row_cluster_t<true>(p, fp32_grad, stream, used);
}

}  // namespace turnopd
