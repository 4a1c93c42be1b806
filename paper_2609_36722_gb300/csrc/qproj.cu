// qproj.cu - launch of the Q-projection kernel (qproj.cuh): the dispatch over
// (D, MR) and the D = 128, one-accumulator instantiations.
#include "qproj.cuh"

namespace att {

template cudaError_t launch_qproj_mr<128, 1>(const QprojParams&, int, cudaStream_t);
extern template cudaError_t launch_qproj_mr<128, 2>(const QprojParams&, int, cudaStream_t);
extern template cudaError_t launch_qproj_mr<64, 1>(const QprojParams&, int, cudaStream_t);
extern template cudaError_t launch_qproj_mr<64, 2>(const QprojParams&, int, cudaStream_t);

cudaError_t launch_qproj(const QprojParams& p, int D, int mr, int ks, cudaStream_t st) {
  if (!qproj_shape_supported(D, mr, ks, p.n_lora) || p.hidden / 64 < ks) return cudaErrorInvalidValue;
  if (D == 128) return mr == 2 ? launch_qproj_mr<128, 2>(p, ks, st) : launch_qproj_mr<128, 1>(p, ks, st);
  return mr == 2 ? launch_qproj_mr<64, 2>(p, ks, st) : launch_qproj_mr<64, 1>(p, ks, st);
}

}  // namespace att
