// Instantiations of the tcgen05 GEMM (gemm_kernel.cuh) with epilogue features kFeatPlain: one
// translation unit per feature set, so that they compile in parallel.
#include "gemm_kernel.cuh"

namespace sgd {
namespace gk {

template cudaError_t launch_tc<64, 256, 8, kFeatPlain>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 256, 4, kFeatPlain>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 224, 8, kFeatPlain>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 128, 8, kFeatPlain>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<32, 256, 8, kFeatPlain>(const GemmPlan&, const TcArgs&, cudaStream_t);

}  // namespace gk
}  // namespace sgd
