// Glue of the transformer blocks around the quantised linears: the residual
// add with RMSNorm, and rotary position embedding. Not part of the paper's
// method (Sec. 3 quantises the linears and the softmax-value product); the
// block runs them between its projections, and they are memory-bound
// element-wise passes.
//
// add_rmsnorm (one CTA of 128 threads per row, 16-byte vectors):
//   h = fl_T(x + r)                 (r = NULL: h = x; stored when h_out != NULL)
//   y = fl_T(fl32(h * inv) * w)     inv = 1 / sqrt(mean(h^2) + eps), float32
// rope (one thread per rotation pair and token):
//   for each head of 128 channels and i < 64, with angle = pos * f_i and
//   f_i = theta^(-2 i / 128) (computed in float64, rounded to float32):
//   (a, b) = (x_i, x_{i+64});  x_i = fl_T(a c - b s),  x_{i+64} = fl_T(b c + a s)
//   with c, s = cos, sin of the float32 angle, the products and sums in
//   float32 (the rotate-half form of the LLaMA / Qwen2 family).
#include "common.cuh"

namespace starq {
namespace {

constexpr int NORM_THREADS = 128;

template <typename T> struct Vec;
template <> struct Vec<__half> {
    static __device__ __forceinline__ void load(const uint4& w, float (&f)[8]) {
        const __half2* h = reinterpret_cast<const __half2*>(&w);
        #pragma unroll
        for (int k = 0; k < 4; ++k) { const float2 v = __half22float2(h[k]); f[2 * k] = v.x; f[2 * k + 1] = v.y; }
    }
    static __device__ __forceinline__ uint4 store(const float (&f)[8]) {
        uint4 w;
        __half2* h = reinterpret_cast<__half2*>(&w);
        #pragma unroll
        for (int k = 0; k < 4; ++k) h[k] = __floats2half2_rn(f[2 * k], f[2 * k + 1]);
        return w;
    }
};
template <> struct Vec<__nv_bfloat16> {
    static __device__ __forceinline__ void load(const uint4& w, float (&f)[8]) {
        const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
        #pragma unroll
        for (int k = 0; k < 4; ++k) { const float2 v = __bfloat1622float2(h[k]); f[2 * k] = v.x; f[2 * k + 1] = v.y; }
    }
    static __device__ __forceinline__ uint4 store(const float (&f)[8]) {
        uint4 w;
        __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&w);
        #pragma unroll
        for (int k = 0; k < 4; ++k) h[k] = __floats2bfloat162_rn(f[2 * k], f[2 * k + 1]);
        return w;
    }
};

// Up to MAXV 16-byte vectors per thread (K <= 8 * 128 * MAXV).
template <typename T, int MAXV>
// h_out may be X or R: every thread reads its own vectors before it writes
// them, so the in-place form needs no ordering between threads.
__global__ void __launch_bounds__(NORM_THREADS) add_rmsnorm_kernel(const T* X, const T* R, int K,
                                                                  const float* __restrict__ w, float eps, T* h_out,
                                                                  T* __restrict__ Y) {
    __shared__ float part[NORM_THREADS / 32];
    const size_t row = blockIdx.x;
    const int nv = K / 8;
    const uint4* x4 = reinterpret_cast<const uint4*>(X + row * K);
    const uint4* r4 = R != nullptr ? reinterpret_cast<const uint4*>(R + row * K) : nullptr;
    float v[MAXV][8];
    float ss = 0.f;
    #pragma unroll
    for (int j = 0; j < MAXV; ++j) {
        const int i = threadIdx.x + j * NORM_THREADS;
        if (i < nv) {
            Vec<T>::load(x4[i], v[j]);
            if (r4 != nullptr) {
                float r[8];
                Vec<T>::load(r4[i], r);
                #pragma unroll
                for (int k = 0; k < 8; ++k) v[j][k] = __fadd_rn(v[j][k], r[k]);
                const uint4 hw = Vec<T>::store(v[j]);      // h rounded to T, as the residual stream is stored
                Vec<T>::load(hw, v[j]);
                if (h_out != nullptr) reinterpret_cast<uint4*>(h_out + row * K)[i] = hw;
            }
            #pragma unroll
            for (int k = 0; k < 8; ++k) ss = fmaf(v[j][k], v[j][k], ss);
        }
    }
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, m);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = ss;
    __syncthreads();
    if (Y == nullptr) return;
    const float tot = (part[0] + part[1]) + (part[2] + part[3]);
    const float inv = rsqrtf(__fadd_rn(__fdiv_rn(tot, (float)K), eps));
    uint4* y4 = reinterpret_cast<uint4*>(Y + row * K);
    const float4* w4 = reinterpret_cast<const float4*>(w);
    #pragma unroll
    for (int j = 0; j < MAXV; ++j) {
        const int i = threadIdx.x + j * NORM_THREADS;
        if (i < nv) {
            const float4 a = __ldg(w4 + 2 * i), b = __ldg(w4 + 2 * i + 1);
            const float wv[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
            float o[8];
            #pragma unroll
            for (int k = 0; k < 8; ++k) o[k] = __fmul_rn(__fmul_rn(v[j][k], inv), wv[k]);
            y4[i] = Vec<T>::store(o);
        }
    }
}

template <typename T>
__global__ void __launch_bounds__(256) rope_kernel(T* QK, int L, int ld, int heads, const int* __restrict__ pos,
                                                   double theta) {
    __shared__ float freq[64];
    if (threadIdx.x < 64) freq[threadIdx.x] = (float)pow(theta, -(double)(2 * threadIdx.x) / 128.0);
    __syncthreads();
    // thread -> (token, head, i): 64 rotation pairs per head
    const size_t n = (size_t)L * heads * 64;
    for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < n; t += (size_t)gridDim.x * blockDim.x) {
        const int i = (int)(t & 63);
        const size_t th = t >> 6;
        const int h = (int)(th % heads);
        const size_t tok = th / heads;
        T* p = QK + tok * ld + h * 128;
        const float ang = __fmul_rn((float)pos[tok], freq[i]);
        float s, c;
        sincosf(ang, &s, &c);
        const float a = (float)p[i], b = (float)p[i + 64];
        p[i] = (T)__fsub_rn(__fmul_rn(a, c), __fmul_rn(b, s));
        p[i + 64] = (T)__fadd_rn(__fmul_rn(b, c), __fmul_rn(a, s));
    }
}

template <typename T>
cudaError_t launch_norm_typed(const void* X, const void* R, int L, int K, const float* w, float eps, void* h_out,
                              void* Y, cudaStream_t stream) {
    const T* x = static_cast<const T*>(X);
    const T* r = static_cast<const T*>(R);
    T* h = static_cast<T*>(h_out);
    T* y = static_cast<T*>(Y);
    const int nv = K / 8;
    if (nv <= NORM_THREADS * 4) add_rmsnorm_kernel<T, 4><<<L, NORM_THREADS, 0, stream>>>(x, r, K, w, eps, h, y);
    else add_rmsnorm_kernel<T, 20><<<L, NORM_THREADS, 0, stream>>>(x, r, K, w, eps, h, y);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_add_rmsnorm(const void* X, const void* R, int dtype, int L, int K, const float* w, float eps,
                               void* h_out, void* Y, cudaStream_t stream) {
    if (L == 0) return cudaSuccess;
    return dtype == STARQ_BF16 ? launch_norm_typed<__nv_bfloat16>(X, R, L, K, w, eps, h_out, Y, stream)
                               : launch_norm_typed<__half>(X, R, L, K, w, eps, h_out, Y, stream);
}

cudaError_t launch_rope(void* QK, int dtype, int L, int ld, int heads, const int* pos, double theta,
                        cudaStream_t stream) {
    if (L == 0) return cudaSuccess;
    const size_t n = (size_t)L * heads * 64;
    size_t blocks = (n + 255) / 256;
    const size_t cap = (size_t)num_sms() * 16;
    if (blocks > cap) blocks = cap;
    if (dtype == STARQ_BF16)
        rope_kernel<__nv_bfloat16><<<(unsigned)blocks, 256, 0, stream>>>(static_cast<__nv_bfloat16*>(QK), L, ld,
                                                                           heads, pos, theta);
    else
        rope_kernel<__half><<<(unsigned)blocks, 256, 0, stream>>>(static_cast<__half*>(QK), L, ld, heads, pos, theta);
    return cudaGetLastError();
}

}  // namespace starq
