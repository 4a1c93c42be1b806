// qproj_d64.cu - instantiations of the Q-projection kernel (qproj.cuh) for
// head size 64.
#include "qproj.cuh"

namespace att {
template cudaError_t launch_qproj_mr<64, 1>(const QprojParams&, int, cudaStream_t);
template cudaError_t launch_qproj_mr<64, 2>(const QprojParams&, int, cudaStream_t);
}  // namespace att
