// SGAT activation transform + per-row symmetric int4 quantisation.
//
// One CTA per row (a token for Q_a, an output channel for Q_w). Each thread
// owns 16 consecutive elements per pass of 16 * blockDim elements; rows
// longer than 4096 take up to five passes, all held in registers so the row
// is read from HBM once.
//
// Per row (Sec. 3.2 Eq. 11 with P = diag(a_s) H_hb, Sec. 3.1 Eq. 2):
//   v = fl32(x * a_s)                      state picked by the row's mask bit
//   v = v H_hb                             fast Walsh-Hadamard transform
//   v = v * gate_s                          binary subspace gate (Eq. 9)
//   v = fl32(v * post_scale)               1/hb on the weight side (Eq. 12)
//   amax = max |v|; s = amax / qmax; r = qmax / amax; q = clamp(rne(v*r))
//
// The transform's butterfly network is the one of the fast Walsh-Hadamard
// transform in stage order h = 1, 2, 4, ..., hb/2, each butterfly
// (a, b) -> (a + b, a - b) in float32 round-to-nearest. Stages h <= 8 run
// inside a thread, 16 <= h <= 256 across lanes by shuffles, h >= 512 across
// warps through shared memory. Every float operation is an explicit
// round-to-nearest intrinsic so that no multiply is contracted into an add.
#include "common.cuh"

namespace starq {
namespace {

constexpr int EPT = 16;          // elements per thread per pass
constexpr int MAX_THREADS = 256; // threads per CTA for rows >= 4096
constexpr int MAX_PASSES = 5;    // rows up to 5 * 4096 = 20480 elements

template <typename T> struct In;
template <> struct In<__half> {
    static __device__ __forceinline__ void load16(const __half* p, float (&v)[EPT]) {
        const uint4* q = reinterpret_cast<const uint4*>(p);
        #pragma unroll
        for (int u = 0; u < 2; ++u) {
            uint4 w = __ldg(q + u);
            const __half2* h = reinterpret_cast<const __half2*>(&w);
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                float2 f = __half22float2(h[j]);
                v[8 * u + 2 * j] = f.x;
                v[8 * u + 2 * j + 1] = f.y;
            }
        }
    }
};
template <> struct In<__nv_bfloat16> {
    static __device__ __forceinline__ void load16(const __nv_bfloat16* p, float (&v)[EPT]) {
        const uint4* q = reinterpret_cast<const uint4*>(p);
        #pragma unroll
        for (int u = 0; u < 2; ++u) {
            uint4 w = __ldg(q + u);
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                float2 f = __bfloat1622float2(h[j]);
                v[8 * u + 2 * j] = f.x;
                v[8 * u + 2 * j + 1] = f.y;
            }
        }
    }
};
template <> struct In<float> {
    static __device__ __forceinline__ void load16(const float* p, float (&v)[EPT]) {
        const float4* q = reinterpret_cast<const float4*>(p);
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            float4 w = __ldg(q + u);
            v[4 * u] = w.x; v[4 * u + 1] = w.y; v[4 * u + 2] = w.z; v[4 * u + 3] = w.w;
        }
    }
};

__device__ __forceinline__ void butterfly(float& lo, float& hi) {
    const float a = lo, b = hi;
    lo = __fadd_rn(a, b);
    hi = __fsub_rn(a, b);
}

template <int PASSES, typename Tin>
__global__ void __launch_bounds__(MAX_THREADS)
sgat_quant_kernel(QuantArgs a) {
    __shared__ float xchg[EPT * MAX_THREADS];   // cross-warp butterfly exchange
    __shared__ float red[MAX_THREADS / 32];
    const int T = blockDim.x;
    const int t = threadIdx.x;
    const int lane = t & 31;
    const int row = blockIdx.x;
    const int K = a.K;
    const int hb = a.hb;
    const Tin* X = static_cast<const Tin*>(a.X) + (size_t)row * K;
    const bool masked = a.mask != nullptr && a.mask[row] != 0;
    const float* sm = masked ? a.a_m : a.a_u;
    // Active coordinates of the row's state (Eq. 9): masked rows keep
    // [0, d_sh + d_m), unmasked rows keep [0, d_sh) and [d_sh + d_m, K).
    const int own_lo = masked ? a.d_sh : a.d_sh + a.d_m;
    const int own_hi = masked ? a.d_sh + a.d_m : a.K;

    float v[PASSES][EPT];
    float amax = 0.f;
    #pragma unroll
    for (int p = 0; p < PASSES; ++p) {
        const int e0 = p * EPT * T + EPT * t;
        const bool live = e0 < K;
        if (live) {
            In<Tin>::load16(X + e0, v[p]);
            if (sm != nullptr) {
                const float4* s4 = reinterpret_cast<const float4*>(sm + e0);
                #pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const float4 w = __ldg(s4 + u);
                    v[p][4 * u] = __fmul_rn(v[p][4 * u], w.x);
                    v[p][4 * u + 1] = __fmul_rn(v[p][4 * u + 1], w.y);
                    v[p][4 * u + 2] = __fmul_rn(v[p][4 * u + 2], w.z);
                    v[p][4 * u + 3] = __fmul_rn(v[p][4 * u + 3], w.w);
                }
            }
        } else {
            #pragma unroll
            for (int i = 0; i < EPT; ++i) v[p][i] = 0.f;
        }
        // stages h = 1, 2, 4, 8 inside the thread
        #pragma unroll
        for (int h = 1; h < EPT; h <<= 1) {
            if (h < hb) {
                #pragma unroll
                for (int i = 0; i < EPT; ++i)
                    if ((i & h) == 0) butterfly(v[p][i], v[p][i + h]);
            }
        }
        // stages h = 16 .. 256 across lanes: partner lane = lane ^ (h / 16)
        #pragma unroll
        for (int m = 1; m < 32; m <<= 1) {
            if (EPT * m < hb) {
                const bool upper = (lane & m) != 0;
                #pragma unroll
                for (int i = 0; i < EPT; ++i) {
                    const float o = __shfl_xor_sync(0xffffffffu, v[p][i], m);
                    v[p][i] = upper ? __fsub_rn(o, v[p][i]) : __fadd_rn(v[p][i], o);
                }
            }
        }
        // stages h = 512 .. 2048 across warps: partner thread = t ^ (h / 16)
        for (int m = 32; EPT * m < hb; m <<= 1) {
            #pragma unroll
            for (int i = 0; i < EPT; ++i) xchg[i * T + t] = v[p][i];
            __syncthreads();
            const bool upper = (t & m) != 0;
            #pragma unroll
            for (int i = 0; i < EPT; ++i) {
                const float o = xchg[i * T + (t ^ m)];
                v[p][i] = upper ? __fsub_rn(o, v[p][i]) : __fadd_rn(v[p][i], o);
            }
            __syncthreads();
        }
        // gate, post-scale, optional debug copy, running amax
        #pragma unroll
        for (int i = 0; i < EPT; ++i) {
            const int e = e0 + i;
            const bool keep = live && (e < a.d_sh || (e >= own_lo && e < own_hi));
            float w = keep ? v[p][i] : 0.f;
            if (a.post_scale != 1.f) w = __fmul_rn(w, a.post_scale);
            v[p][i] = w;
            amax = fmaxf(amax, fabsf(w));
        }
        if (a.v_dbg != nullptr && live) {
            float4* d4 = reinterpret_cast<float4*>(a.v_dbg + (size_t)row * K + e0);
            #pragma unroll
            for (int u = 0; u < 4; ++u)
                d4[u] = make_float4(v[p][4 * u], v[p][4 * u + 1], v[p][4 * u + 2], v[p][4 * u + 3]);
        }
    }
    // row amax: warp shuffle, then across warps
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, m));
    if (lane == 0) red[t >> 5] = amax;
    __syncthreads();
    amax = 0.f;
    for (int w = 0; w < (T >> 5); ++w) amax = fmaxf(amax, red[w]);

    const float qmax = (float)a.qmax;
    const bool nz = amax > 0.f;
    const float s = nz ? __fdiv_rn(amax, qmax) : 0.f;
    const float r = nz ? __fdiv_rn(qmax, amax) : 0.f;
    if (t == 0) a.s[row] = s;
    #pragma unroll
    for (int p = 0; p < PASSES; ++p) {
        const int e0 = p * EPT * T + EPT * t;
        if (e0 >= K) continue;
        uint32_t packed[2] = {0u, 0u};
        #pragma unroll
        for (int i = 0; i < EPT; ++i) {
            int q = __float2int_rn(__fmul_rn(v[p][i], r));
            q = max(-a.qmax, min(a.qmax, q));
            packed[i >> 3] |= (uint32_t)(q & 0xF) << (4 * (i & 7));
        }
        *reinterpret_cast<uint2*>(a.Xq + (size_t)row * (K / 2) + e0 / 2) =
            make_uint2(packed[0], packed[1]);
    }
}

template <typename Tin>
cudaError_t launch_typed(const QuantArgs& a, cudaStream_t stream) {
    int threads, passes;
    if (a.K <= EPT * MAX_THREADS) {
        threads = ((a.K / EPT) + 31) / 32 * 32;
        passes = 1;
    } else {
        threads = MAX_THREADS;
        passes = (a.K + EPT * MAX_THREADS - 1) / (EPT * MAX_THREADS);
    }
    dim3 grid(a.L), block(threads);
    switch (passes) {
        case 1: sgat_quant_kernel<1, Tin><<<grid, block, 0, stream>>>(a); break;
        case 2: sgat_quant_kernel<2, Tin><<<grid, block, 0, stream>>>(a); break;
        case 3: sgat_quant_kernel<3, Tin><<<grid, block, 0, stream>>>(a); break;
        case 4: sgat_quant_kernel<4, Tin><<<grid, block, 0, stream>>>(a); break;
        case 5: sgat_quant_kernel<5, Tin><<<grid, block, 0, stream>>>(a); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_sgat_quant(const QuantArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    switch (a.x_dtype) {
        case STARQ_F16: return launch_typed<__half>(a, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_typed<float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
