// Weight rows for the asymmetric activation path (Eq. 2-4 for activations,
// symmetric per-channel weights, Eq. 3 and Eq. 5):
//   sum_k (q_a[k] - z) q_w[k] = sum_k q_a[k] q_w[k] + (-z) sum_k q_w[k].
// The activation rows carry 128 extra columns of -z (the quantiser writes
// them). The weight rows carry 128 extra E4M3 values w_j with
// sum_j w_j = sum_k q_w[k], so the 4-bit GEMM over K + 128 computes the
// left side exactly: every product is an integer and every partial sum stays
// below 2^24 (|acc| <= 105 K + 15 * 7 K).
//
// The decomposition: as many 448s (the largest E4M3 value) as fit, then the
// remainder r < 448 greedily by the largest E4M3 value <= r (an E4M3 value
// 2^e (1 + m/8) has its spacing 2^(e-3) <= r / 8, so each step leaves less
// than an eighth: at most four more values), with the sign of the sum; the
// rest are zeros. 7 K / 448 + 4 <= 128 for K <= 7680.
#include "asym.cuh"
#include "common.cuh"

namespace starq {
namespace {

// E4M3 byte of a non-negative integer that is an E4M3 number (<= 448)
__device__ __forceinline__ uint8_t e4m3_of_int(int v) {
    uint16_t h;
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %1;" : "=h"(h) : "f"((float)v));
    return (uint8_t)(h & 0xFF);
}

// largest E4M3 number <= r, for 1 <= r <= 448
__device__ __forceinline__ int e4m3_floor(int r) {
    if (r <= 16) return r;
    const int e = 31 - __clz(r);                  // 2^e <= r < 2^(e+1), e >= 4
    const int step = 1 << (e - 3);
    return min(r / step * step, 448);
}

// one warp per weight row
__global__ void __launch_bounds__(256) zero_point_columns_kernel(const uint8_t* Wq, uint8_t* We, int N, int K) {
    const int warp = (int)((blockIdx.x * blockDim.x + threadIdx.x) >> 5), lane = threadIdx.x & 31;
    if (warp >= N) return;
    const uint8_t* src = Wq + (size_t)warp * (K / 2);
    uint8_t* dst = We + (size_t)warp * (K + 128);
    int sum = 0;
    for (int i = lane; i < K / 8; i += 32) {      // eight codes per 32-bit word
        const uint32_t x = *reinterpret_cast<const uint32_t*>(src + 4 * i);
        #pragma unroll
        for (int k = 0; k < 8; ++k) sum += ((int)(x << (28 - 4 * k))) >> 28;
        uint32_t lo, hi;
        int4x8_to_e4m3x8(x, lo, hi);
        *reinterpret_cast<uint2*>(dst + 8 * i) = make_uint2(lo, hi);
    }
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, m);
    // lane l writes columns K + 4 l .. K + 4 l + 3: value j is 448 for
    // j < n448, then the greedy remainder terms, then 0
    const int neg = sum < 0, mag = neg ? -sum : sum;
    const int n448 = mag / 448;
    int rem = mag - 448 * n448;
    int terms[5] = {0, 0, 0, 0, 0};
    #pragma unroll
    for (int t = 0; t < 5; ++t) {
        if (rem > 0) {
            terms[t] = e4m3_floor(rem);
            rem -= terms[t];
        }
    }
    uint32_t w = 0;
    #pragma unroll
    for (int b = 0; b < 4; ++b) {
        const int j = 4 * lane + b;
        int val = 0;
        if (j < n448) val = 448;
        else if (j - n448 < 5) val = terms[j - n448];
        uint8_t byte = e4m3_of_int(val);
        if (neg && val != 0) byte |= 0x80;        // E4M3 sign bit
        w |= (uint32_t)byte << (8 * b);
    }
    *reinterpret_cast<uint32_t*>(dst + K + 4 * lane) = w;
}

}  // namespace

cudaError_t launch_zero_point_columns(const uint8_t* Wq, uint8_t* We, int N, int K, cudaStream_t stream) {
    if (N == 0) return cudaSuccess;
    const int blocks = (N + 7) / 8;               // eight warps (rows) per CTA
    zero_point_columns_kernel<<<blocks, 256, 0, stream>>>(Wq, We, N, K);
    return cudaGetLastError();
}

}  // namespace starq
