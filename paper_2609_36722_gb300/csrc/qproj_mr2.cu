// qproj_mr2.cu - instantiations of the Q-projection kernel (qproj.cuh) with
// two 128-row accumulators per CTA, head size 128.
#include "qproj.cuh"

namespace att {
template cudaError_t launch_qproj_mr<128, 2>(const QprojParams&, int, cudaStream_t);
}  // namespace att
