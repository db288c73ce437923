// Dense orthogonal basis (the learned P of App. B, W_f = Q_w(P^T W^T)): the
// transform X^s P is a 16-bit GEMM whose A operand is the scaled rows
// fl16(fl32(x * a_s)). This kernel forms that operand: eight elements per
// thread, one 16-byte store.
#include "common.cuh"
#include "dense.cuh"

namespace starq {
namespace {

template <typename T> __device__ __forceinline__ void load8(const T* p, float (&v)[8]);
template <> __device__ __forceinline__ void load8<__half>(const __half* p, float (&v)[8]) {
    const uint4 w = *reinterpret_cast<const uint4*>(p);
    const __half2* h = reinterpret_cast<const __half2*>(&w);
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 f = __half22float2(h[k]);
        v[2 * k] = f.x;
        v[2 * k + 1] = f.y;
    }
}
template <> __device__ __forceinline__ void load8<__nv_bfloat16>(const __nv_bfloat16* p, float (&v)[8]) {
    const uint4 w = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float2 f = __bfloat1622float2(h[k]);
        v[2 * k] = f.x;
        v[2 * k + 1] = f.y;
    }
}
template <> __device__ __forceinline__ void load8<float>(const float* p, float (&v)[8]) {
    const float4 a = reinterpret_cast<const float4*>(p)[0], b = reinterpret_cast<const float4*>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

template <typename Tin>
__global__ void __launch_bounds__(256) scale_rows_f16_kernel(const Tin* X, int L, int K, const uint8_t* mask,
                                                             const float* a_m, const float* a_u, __half* out) {
    const size_t g = (size_t)blockIdx.x * blockDim.x + threadIdx.x;     // group of 8 elements
    const size_t groups = (size_t)L * (size_t)(K / 8);
    if (g >= groups) return;
    const int row = (int)(g / (size_t)(K / 8));
    const int k0 = (int)(g - (size_t)row * (size_t)(K / 8)) * 8;
    const float* a = (mask != nullptr && mask[row] != 0) ? a_m : a_u;
    float v[8];
    load8<Tin>(X + (size_t)row * K + k0, v);
    if (a != nullptr) {
        const float4 s0 = __ldg(reinterpret_cast<const float4*>(a + k0)), s1 = __ldg(reinterpret_cast<const float4*>(a + k0 + 4));
        v[0] = __fmul_rn(v[0], s0.x); v[1] = __fmul_rn(v[1], s0.y); v[2] = __fmul_rn(v[2], s0.z); v[3] = __fmul_rn(v[3], s0.w);
        v[4] = __fmul_rn(v[4], s1.x); v[5] = __fmul_rn(v[5], s1.y); v[6] = __fmul_rn(v[6], s1.z); v[7] = __fmul_rn(v[7], s1.w);
    }
    uint32_t w[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        const __half2 h = __floats2half2_rn(v[2 * k], v[2 * k + 1]);
        w[k] = *reinterpret_cast<const uint32_t*>(&h);
    }
    *reinterpret_cast<uint4*>(out + (size_t)row * K + k0) = make_uint4(w[0], w[1], w[2], w[3]);
}

template <typename Tin>
cudaError_t launch_typed(const void* X, int L, int K, const uint8_t* mask, const float* a_m, const float* a_u,
                         __half* out, cudaStream_t stream) {
    const size_t groups = (size_t)L * (size_t)(K / 8);
    if (groups == 0) return cudaSuccess;
    scale_rows_f16_kernel<Tin><<<(unsigned)((groups + 255) / 256), 256, 0, stream>>>(
        static_cast<const Tin*>(X), L, K, mask, a_m, a_u, out);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_scale_rows_f16(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                                  const float* a_u, __half* out, cudaStream_t stream) {
    switch (x_dtype) {
        case STARQ_F16: return launch_typed<__half>(X, L, K, mask, a_m, a_u, out, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(X, L, K, mask, a_m, a_u, out, stream);
        case STARQ_F32: return launch_typed<float>(X, L, K, mask, a_m, a_u, out, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
