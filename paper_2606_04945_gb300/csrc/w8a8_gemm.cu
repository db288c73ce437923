// W8A8 GEMM: the 8-bit setting of the method (Tab. 5; Sec. 3.1 Eq. 2 with
// qmax = 127 for the per-token activation codes and the per-channel weight
// codes, Eq. 3 for the dequantisation):
//   acc[i][n] = sum_k qa[i][k] qw[n][k]          exact integers
//   Y[i][n]   = fl(fl(fl32(acc) * s_a[i]) * s_w[n]) (+ bias[n]) -> output type
//
// sm_103a has no integer tcgen05 MMA, and 8-bit codes are not E4M3 numbers,
// but every code |c| <= 127 is an fp16 number and so is every product's
// factor: the product runs as one kind::f16 GEMM on the codes held as fp16
// (the quantiser writes them so, [L][K]; w8_codes_f16 below the weights,
// [N][K]). A float32 accumulator stays exact while its partial sums are
// integers below 2^24; the GEMM (operand kind 3 of the TMA pair kernel in
// w4a4_gemm.cu) therefore accumulates runs of 512 K, each at most
// 512 * 127^2 < 2^23 in magnitude, and its epilogue adds the runs in int32
// (|acc| <= 127^2 K < 2^31 for K <= 65536) before dequantising.
//
// This costs one 16-bit product per 8-bit product: half the FP8 kind's rate,
// and the shared-memory bound of the 16-bit pair tiles. (An exact split into
// E4M3 halves, c = 16 h + l, takes four FP8 products per 8-bit product into
// three accumulators: the same tensor time, with four operand tiles per K
// block through shared memory instead of two.)
#include "common.cuh"
#include "w8a8.cuh"

namespace starq {
namespace {

// 8-bit weight codes [N][K] (two's complement bytes) -> the same codes as
// fp16 [N][K]: one thread per 8 codes (8 bytes in, 16 bytes out).
__global__ void __launch_bounds__(256) w8_codes_f16_kernel(const uint8_t* Wq, uint8_t* We, size_t N, int K) {
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;     // group of 8 codes
    const size_t groups = N * (size_t)(K / 8);
    if (i >= groups) return;
    const size_t row = i / (size_t)(K / 8);
    const int k0 = (int)(i - row * (size_t)(K / 8)) * 8;
    const uint2 w = *reinterpret_cast<const uint2*>(Wq + row * K + k0);
    uint32_t h[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t word = k < 2 ? w.x : w.y;
        const int q0 = (int)(int8_t)(word >> (16 * (k & 1))), q1 = (int)(int8_t)(word >> (16 * (k & 1) + 8));
        const __half2 p = __floats2half2_rn((float)q0, (float)q1);      // exact: |q| <= 128
        h[k] = *reinterpret_cast<const uint32_t*>(&p);
    }
    *reinterpret_cast<uint4*>(We + (row * K + k0) * 2) = make_uint4(h[0], h[1], h[2], h[3]);
}

}  // namespace

cudaError_t launch_w8_codes_f16(const uint8_t* Wq, uint8_t* We, size_t N, int K, cudaStream_t stream) {
    const size_t groups = N * (size_t)(K / 8);
    if (groups == 0) return cudaSuccess;
    w8_codes_f16_kernel<<<(unsigned)((groups + 255) / 256), 256, 0, stream>>>(Wq, We, N, K);
    return cudaGetLastError();
}

}  // namespace starq
