// The dense-basis transform's elementwise step (dense.cu), called by the C
// ABI; the product itself runs on the 16-bit GEMM (launch_fp16_gemm).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace starq {

// out[i][k] = fl16(fl32(X[i][k] * a_s[k])), s = mask[i] (1: a_m, 0 or no
// mask: a_u; a NULL vector is all ones). K % 8 == 0; X 16-byte aligned.
cudaError_t launch_scale_rows_f16(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                                  const float* a_u, __half* out, cudaStream_t stream);

}  // namespace starq
