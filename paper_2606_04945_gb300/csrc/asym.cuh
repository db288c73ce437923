// Weight side of the asymmetric activation path (asym.cu), called by the C
// ABI after validation.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace starq {

// Largest K for which 128 E4M3 columns can hold sum_k q_w (|sum| <= 7 K).
constexpr int ASYM_MAX_K = 7680;

// Packed int4 weight codes [N][K/2] -> E4M3 rows [N][K + 128]: the codes,
// then 128 E4M3 values that sum exactly to the row's code sum.
cudaError_t launch_zero_point_columns(const uint8_t* Wq, uint8_t* We, int N, int K, cudaStream_t stream);

}  // namespace starq
