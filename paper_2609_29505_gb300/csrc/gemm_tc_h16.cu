// Instantiations of the tcgen05 GEMM (gemm_kernel.cuh) with epilogue features kFeatH16: one
// translation unit per feature set, so that they compile in parallel.
#include "gemm_kernel.cuh"

namespace sgd {
namespace gk {

template cudaError_t launch_tc<64, 256, 8, kFeatH16>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 256, 4, kFeatH16>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 224, 8, kFeatH16>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 128, 8, kFeatH16>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<32, 256, 8, kFeatH16>(const GemmPlan&, const TcArgs&, cudaStream_t);

}  // namespace gk
}  // namespace sgd
