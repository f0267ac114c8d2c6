// sq_gemv_fp16.cu -- instantiations of the CUDA-core skinny linear layer for
// fp16 weights (one translation unit per weight format so they compile in
// parallel).
#include "sq_gemv.cuh"

namespace sq {

cudaError_t launch_gemv_fp16(const GemvArgs& a, int mr, int r, bool silu, int lpr, int64_t blocks_needed, size_t smem,
                           cudaStream_t st) {
  return launch_gemv_fmt<WK_FP16>(a, mr, r, silu, lpr, blocks_needed, smem, st);
}

cudaError_t take_gemv_status_fp16(uint32_t* bits) { return take_gemv_status_tu(bits); }

}  // namespace sq
