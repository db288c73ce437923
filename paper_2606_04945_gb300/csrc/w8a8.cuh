// Launchers of the 8-bit GEMM (w4a4_gemm.cu, operand kind 3 of the TMA
// pair kernel) and of the weight codes' fp16 form (w8a8_gemm.cu), called by
// the C ABI after validation.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "common.cuh"

namespace starq {

// a.Xe: activation codes as fp16 [L][K]; a.We: weight codes as fp16 [N][K];
// N % 128 == 0, K % 128 == 0, K <= 65536.
cudaError_t launch_w8a8_gemm(const GemmArgs& a, cudaStream_t stream);
// 8-bit weight codes [N][K] -> the same codes as fp16 [N][K]; K % 8 == 0.
cudaError_t launch_w8_codes_f16(const uint8_t* Wq, uint8_t* We, size_t N, int K, cudaStream_t stream);

}  // namespace starq
