// sq_gemv_int4.cu -- instantiations of the CUDA-core skinny linear layer for
// int4 weights (one translation unit per weight format so they compile in
// parallel).
#include "sq_gemv.cuh"
#include "sq_gemv_mma.cuh"

namespace sq {

cudaError_t launch_gemv_int4(const GemvArgs& a, int mr, int r, bool silu, int lpr, int64_t blocks_needed, size_t smem,
                           cudaStream_t st) {
  return launch_gemv_fmt<WK_INT4>(a, mr, r, silu, lpr, blocks_needed, smem, st);
}

cudaError_t launch_gemv_mma_int4(const GemvArgs& a, bool silu, cudaStream_t st) {
  return launch_gemv_mma_int4_impl(a, silu, st);
}

cudaError_t take_gemv_status_int4(uint32_t* bits) { return take_gemv_status_tu(bits); }

}  // namespace sq
