// TAC: block-wise affine compensation (Sec. 3.3 Eq. 17, App. C row-major form)
//
//   out[i][b*g + r] = sum_j M[b][r][j] * Z[i][b*g + j] + d[b][r]
//
// Grid: (token tiles, blocks b). A CTA stages M_b transposed (Mt[j][r]) and a
// tile of TM tokens of block b in shared memory, then each thread computes
// RT = 4 tokens x RC = 8 channels with float32 FMAs, reading four j at a time
// (float4) from both tiles. TM = 8192 / g tokens, so the token tile is
// 32 KB (fp32) and the CTA holds g*g*4 + 32 KB of shared memory.
#include "common.cuh"

namespace starq {
namespace {

constexpr int TPB = 256;

template <typename T> __device__ __forceinline__ float to_f(T x);
template <> __device__ __forceinline__ float to_f<__half>(__half x) { return __half2float(x); }
template <> __device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 x) { return __bfloat162float(x); }
template <> __device__ __forceinline__ float to_f<float>(float x) { return x; }

template <typename T> __device__ __forceinline__ T from_f(float x);
template <> __device__ __forceinline__ __half from_f<__half>(float x) { return __float2half_rn(x); }
template <> __device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float x) { return __float2bfloat16_rn(x); }
template <> __device__ __forceinline__ float from_f<float>(float x) { return x; }

template <int G, typename TIn, typename TOut>
__global__ void __launch_bounds__(TPB)
tac_kernel(TacArgs a) {
    constexpr int RC = G < 8 ? G : 8;         // channels per thread
    constexpr int CG = G / RC;                // channel groups
    constexpr int TG = TPB / CG;              // token groups
    constexpr int RT = 4;                     // tokens per thread
    constexpr int TM = TG * RT;               // tokens per CTA
    constexpr int ZP = G + 4;                 // padded token-row length
    extern __shared__ float4 smem4[];
    float* Mt = reinterpret_cast<float*>(smem4);      // [G][G]  Mt[j][r] = M[b][r][j]
    float* zs = Mt + G * G;                           // [TM][ZP]

    const int b = blockIdx.y;
    const int tok0 = blockIdx.x * TM;
    const int C = a.C;
    const float* Mb = a.M + (size_t)b * G * G;
    const TIn* Z = static_cast<const TIn*>(a.Z);

    for (int idx = threadIdx.x; idx < G * G; idx += TPB) {
        const int r = idx % G, j = idx / G;       // consecutive threads: consecutive r
        Mt[j * G + r] = __ldg(Mb + (size_t)r * G + j);
    }
    for (int idx = threadIdx.x; idx < TM * G; idx += TPB) {
        const int t = idx / G, j = idx % G;
        const int tok = tok0 + t;
        zs[t * ZP + j] = tok < a.L ? to_f<TIn>(Z[(size_t)tok * C + b * G + j]) : 0.f;
    }
    __syncthreads();

    const int cg = threadIdx.x % CG;
    const int tg = threadIdx.x / CG;
    float acc[RT][RC];
    #pragma unroll
    for (int t = 0; t < RT; ++t)
        #pragma unroll
        for (int c = 0; c < RC; ++c) acc[t][c] = 0.f;

    #pragma unroll 2
    for (int j = 0; j < G; j += 4) {
        float z[RT][4];
        #pragma unroll
        for (int t = 0; t < RT; ++t) {
            const float4 v = *reinterpret_cast<const float4*>(&zs[(tg * RT + t) * ZP + j]);
            z[t][0] = v.x; z[t][1] = v.y; z[t][2] = v.z; z[t][3] = v.w;
        }
        #pragma unroll
        for (int jj = 0; jj < 4 && jj < G; ++jj) {
            float m[RC];
            #pragma unroll
            for (int c = 0; c < RC; c += 4) {
                const float4 v = *reinterpret_cast<const float4*>(&Mt[(j + jj) * G + cg * RC + c]);
                m[c] = v.x; m[c + 1] = v.y; m[c + 2] = v.z; m[c + 3] = v.w;
            }
            #pragma unroll
            for (int t = 0; t < RT; ++t)
                #pragma unroll
                for (int c = 0; c < RC; ++c) acc[t][c] = fmaf(z[t][jj], m[c], acc[t][c]);
        }
    }

    float dv[RC];
    #pragma unroll
    for (int c = 0; c < RC; ++c) dv[c] = a.d ? __ldg(a.d + (size_t)b * G + cg * RC + c) : 0.f;
    TOut* out = static_cast<TOut*>(a.out);
    #pragma unroll
    for (int t = 0; t < RT; ++t) {
        const int tok = tok0 + tg * RT + t;
        if (tok >= a.L) continue;
        TOut* o = out + (size_t)tok * C + b * G + cg * RC;
        #pragma unroll
        for (int c = 0; c < RC; ++c) o[c] = from_f<TOut>(acc[t][c] + dv[c]);
    }
}

template <int G, typename TIn, typename TOut>
cudaError_t launch_g(const TacArgs& a, cudaStream_t stream) {
    constexpr int RC = G < 8 ? G : 8;
    constexpr int TM = (TPB / (G / RC)) * 4;
    constexpr size_t smem = (size_t)G * G * 4 + (size_t)TM * (G + 4) * 4;
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 64 && !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(tac_kernel<G, TIn, TOut>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr_set[dev] = true;
    }
    dim3 grid((a.L + TM - 1) / TM, a.C / G);
    tac_kernel<G, TIn, TOut><<<grid, TPB, smem, stream>>>(a);
    return cudaGetLastError();
}

template <typename TIn, typename TOut>
cudaError_t launch_io(const TacArgs& a, cudaStream_t stream) {
    switch (a.g) {
        case 4: return launch_g<4, TIn, TOut>(a, stream);
        case 8: return launch_g<8, TIn, TOut>(a, stream);
        case 16: return launch_g<16, TIn, TOut>(a, stream);
        case 32: return launch_g<32, TIn, TOut>(a, stream);
        case 64: return launch_g<64, TIn, TOut>(a, stream);
        case 128: return launch_g<128, TIn, TOut>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <typename TIn>
cudaError_t launch_in(const TacArgs& a, cudaStream_t stream) {
    switch (a.out_dtype) {
        case STARQ_F16: return launch_io<TIn, __half>(a, stream);
        case STARQ_BF16: return launch_io<TIn, __nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_io<TIn, float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_tac(const TacArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    switch (a.z_dtype) {
        case STARQ_F16: return launch_in<__half>(a, stream);
        case STARQ_BF16: return launch_in<__nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_in<float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
