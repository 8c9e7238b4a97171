// Instantiations of the tcgen05 GEMM (gemm_kernel.cuh) with epilogue features kFeatLn: one
// translation unit per feature set, so that they compile in parallel.
#include "gemm_kernel.cuh"

namespace sgd {
namespace gk {

template cudaError_t launch_tc<64, 256, 8, kFeatLn>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 256, 4, kFeatLn>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 224, 8, kFeatLn>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<64, 128, 8, kFeatLn>(const GemmPlan&, const TcArgs&, cudaStream_t);
template cudaError_t launch_tc<32, 256, 8, kFeatLn>(const GemmPlan&, const TcArgs&, cudaStream_t);

}  // namespace gk
}  // namespace sgd
