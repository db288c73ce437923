// Launchers of the 8-bit GEMM and of the weight-code split (w8a8_gemm.cu),
// called by the C ABI after validation.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "common.cuh"

namespace starq {

// a.Xe: activation code halves [L][2K] (E4M3 h in columns 0..K-1, l in
// K..2K-1); a.We: weight code halves [N][2K]; N % 128 == 0, K % 128 == 0,
// K <= 65536.
cudaError_t launch_w8a8_gemm(const GemmArgs& a, cudaStream_t stream);
// 8-bit weight codes [N][K] -> their E4M3 halves [N][2K]; K % 8 == 0.
cudaError_t launch_w8_split(const uint8_t* Wq, uint8_t* We, size_t N, int K, cudaStream_t stream);

}  // namespace starq
