// gemm_tc_i8.cu -- the int8-A launch shapes of the tensor-core integer GEMM (the converter warps turn
// the int8 activation tile into the fp16 operand in shared memory) and the split-convolution shape;
// a translation unit of its own so that the two halves of the GEMM compile in parallel.
#include "gemm_tc.cuh"

namespace ilw {

template <int BN, int STAGES, int NB, bool GELU>
cudaError_t run_i8(const GemmProblem &gp, const EpiParams &ep, cudaStream_t s) {
    return run<BN, STAGES, NB, false, false, GELU>(gp, ep, s);
}

template cudaError_t run_i8<128, 5, kMaxBranches, false>(const GemmProblem &, const EpiParams &, cudaStream_t);
template cudaError_t run_i8<192, 3, 1, true>(const GemmProblem &, const EpiParams &, cudaStream_t);
template cudaError_t run_i8<192, 4, 1, false>(const GemmProblem &, const EpiParams &, cudaStream_t);
template cudaError_t run_i8<128, 3, 1, true>(const GemmProblem &, const EpiParams &, cudaStream_t);
template cudaError_t run_i8<128, 5, 1, false>(const GemmProblem &, const EpiParams &, cudaStream_t);

}  // namespace ilw
