// W8A8 GEMM: the 8-bit setting of the method (Tab. 5; Sec. 3.1 Eq. 2 with
// qmax = 127 for the per-token activation codes and the per-channel weight
// codes, Eq. 3 for the dequantisation):
//   acc[i][n] = sum_k qa[i][k] qw[n][k]          exact integers
//   Y[i][n]   = fl(fl(fl32(acc) * s_a[i]) * s_w[n]) (+ bias[n]) -> output type
//
// sm_103a has no integer tcgen05 MMA, and 8-bit codes are not E4M3 numbers.
// So each code is split as c = 16 h + l, with l = ((c + 8) mod 16) - 8 in
// [-8, 7] and h = (c - l) / 16 in [-8, 8]. Both halves are exact E4M3
// numbers; the quantiser writes them as [rows][2K] (h in columns 0..K-1, l in
// K..2K-1). Then
//   acc = 256 (H_a H_w^T) + 16 (H_a L_w^T + L_a H_w^T) + L_a L_w^T,
// four kind::f8f6f4 products into three TMEM accumulators. Each partial sum
// is an integer of magnitude at most 128 K < 2^24 (K <= 65536), so the
// float32 accumulation of the tensor cores is exact. The combination runs in
// int32 (|acc| <= 127^2 K < 2^31).
//
// One CTA per 128 x 128 output tile; the row tiles of one weight tile are
// consecutive in the grid, so a weight tile leaves DRAM once. Four epilogue
// warps (one TMEM lane quarter each), a TMA warp and an MMA warp. A
// pipeline stage holds the four 128 x 128-byte tiles (H_a, L_a, H_w, L_w)
// of one 128-wide K block (64 KB, 128-byte swizzle); three stages. Every
// MMA reads both operands from shared memory, whose bandwidth bounds the
// kernel: 192 KB per K block (16 MMAs of 8 KB, 64 KB of TMA writes) against
// 1024 cycles of MMA. (Copying the activation halves into TMEM first, so
// the MMAs read them there, was slower: eight more tcgen05 instructions per
// K block made the single issuing thread the bound.) Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "w8a8.cuh"

namespace starq {
namespace {

constexpr int W8_BM = 128, W8_BN = 128, W8_BK = 128;
constexpr int W8_TILE = W8_BM * W8_BK;              // bytes of one 128 x 128 E4M3 tile
constexpr int W8_STAGE = 4 * W8_TILE;
constexpr int W8_STAGES = 3;
constexpr int W8_THREADS = 192;                     // 4 epilogue warps, TMA warp, MMA warp
constexpr int W8_TMA_WARP = 4, W8_MMA_WARP = 5;
constexpr unsigned STATUS_TIMEOUT_W8 = 1u << 5;
// TMEM columns of the three accumulators
constexpr uint32_t TM_HH = 0, TM_MIX = 128, TM_LL = 256;

struct W8Sm {
    uint64_t full[W8_STAGES], empty[W8_STAGES], tmem_full;
    uint32_t tmem_base;
    int abort;
};
constexpr size_t W8_SMEM = (size_t)W8_STAGES * W8_STAGE + 1024 + sizeof(W8Sm);

// 32 float32 results -> 32 outputs at p (16-byte aligned)
template <typename T> struct W8Out;
template <> struct W8Out<__half> {
    static __device__ __forceinline__ void store(__half* p, const float (&y)[32]) {
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
            #pragma unroll
            for (int k = 0; k < 4; ++k) {
                const __half2 h = __floats2half2_rn(y[8 * u + 2 * k], y[8 * u + 2 * k + 1]);
                w[k] = *reinterpret_cast<const uint32_t*>(&h);
            }
            reinterpret_cast<uint4*>(p)[u] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
};
template <> struct W8Out<__nv_bfloat16> {
    static __device__ __forceinline__ void store(__nv_bfloat16* p, const float (&y)[32]) {
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
            #pragma unroll
            for (int k = 0; k < 4; ++k) {
                const __nv_bfloat162 h = __floats2bfloat162_rn(y[8 * u + 2 * k], y[8 * u + 2 * k + 1]);
                w[k] = *reinterpret_cast<const uint32_t*>(&h);
            }
            reinterpret_cast<uint4*>(p)[u] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
};
template <> struct W8Out<float> {
    static __device__ __forceinline__ void store(float* p, const float (&y)[32]) {
        #pragma unroll
        for (int u = 0; u < 8; ++u)
            reinterpret_cast<float4*>(p)[u] = make_float4(y[4 * u], y[4 * u + 1], y[4 * u + 2], y[4 * u + 3]);
    }
};

template <typename TOut>
__global__ void __launch_bounds__(W8_THREADS, 1)
w8a8_gemm_kernel(GemmArgs a, const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_w) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    W8Sm* sh = reinterpret_cast<W8Sm*>(smem_raw + (base - raw) + (size_t)W8_STAGES * W8_STAGE);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * W8_BM, n0 = blockIdx.y * W8_BN;
    const int K = a.K, nkb = K / W8_BK;
    volatile int* abort = &sh->abort;
    auto B = [](const uint64_t& bar) { return smem_addr(&bar); };

    if (threadIdx.x == 0) {
        for (int s = 0; s < W8_STAGES; ++s) {
            mbar_init(B(sh->full[s]), 1);
            mbar_init(B(sh->empty[s]), 1);
        }
        mbar_init(B(sh->tmem_full), 1);
        sh->abort = 0;
        mbar_fence_init();
    }
    if (warp == W8_MMA_WARP) {
        tmem_alloc(smem_addr(&sh->tmem_base), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;

    if (warp == W8_TMA_WARP) {
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; ++kb) {
            const int s = kb % W8_STAGES, n = kb / W8_STAGES;
            if (!mbar_wait_bounded_warp(B(sh->empty[s]), (uint32_t)(n & 1) ^ 1u, abort)) { ok = false; break; }
            const uint32_t st = base + (uint32_t)s * W8_STAGE, fb = B(sh->full[s]);
            if (elect_one()) {
                mbar_arrive_expect_tx(fb, W8_STAGE);
                tma_load_2d(st, &tm_a, kb * W8_BK, m0, fb);                       // H_a
                tma_load_2d(st + W8_TILE, &tm_a, K + kb * W8_BK, m0, fb);         // L_a
                tma_load_2d(st + 2 * W8_TILE, &tm_w, kb * W8_BK, n0, fb);         // H_w
                tma_load_2d(st + 3 * W8_TILE, &tm_w, K + kb * W8_BK, n0, fb);     // L_w
            }
            __syncwarp();
        }
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_W8); }
    } else if (warp == W8_MMA_WARP) {
        // E4M3 A and B (format 0), f32 D, N = 128 (bits 17..22), M = 128 (bits 24..28)
        constexpr uint32_t IDESC = (1u << 4) | ((uint32_t)(W8_BN >> 3) << 17) | ((uint32_t)(W8_BM >> 4) << 24);
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; ++kb) {
            const int s = kb % W8_STAGES, n = kb / W8_STAGES;
            if (!mbar_wait_bounded_warp(B(sh->full[s]), (uint32_t)(n & 1), abort)) { ok = false; break; }
            tc_fence_after();
            const uint32_t st = base + (uint32_t)s * W8_STAGE;
            if (elect_one()) {
                const uint64_t ah = smem_desc_sw128(st), al = smem_desc_sw128(st + W8_TILE);
                const uint64_t wh = smem_desc_sw128(st + 2 * W8_TILE), wl = smem_desc_sw128(st + 3 * W8_TILE);
                #pragma unroll
                for (int ks = 0; ks < W8_BK / 32; ++ks) {
                    // 32 bytes per K step, added to the start-address field
                    // (addresses below 2^18: the field never carries)
                    const uint64_t k = (uint64_t)(ks * 32 / 16);
                    const uint32_t acc = (kb > 0 || ks > 0) ? 1u : 0u;
                    mma_f8f6f4(tmem + TM_HH, ah + k, wh + k, IDESC, acc);
                    mma_f8f6f4(tmem + TM_MIX, ah + k, wl + k, IDESC, acc);
                    mma_f8f6f4(tmem + TM_MIX, al + k, wh + k, IDESC, 1u);
                    mma_f8f6f4(tmem + TM_LL, al + k, wl + k, IDESC, acc);
                }
                tc_commit(B(sh->empty[s]));
            }
            __syncwarp();
        }
        if (elect_one()) tc_commit(B(sh->tmem_full));
        __syncwarp();
        if (lane == 0) {
            // every MMA of this thread has completed before TMEM is released
            volatile int never = 0;
            if (!mbar_wait_bounded(B(sh->tmem_full), 0, &never)) ok = false;
        }
        __syncwarp();
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_W8); }
    } else {
        // epilogue: warp w reads TMEM lanes 32 w .. 32 w + 31 (tile rows)
        const bool ok = mbar_wait_bounded_warp(B(sh->tmem_full), 0, abort);
        if (ok) {
            tc_fence_after();
            const int row = m0 + warp * 32 + lane;
            const bool valid = row < a.L;
            const float sa = valid ? a.s_a[row] : 0.f;
            const uint32_t tl = tmem + ((uint32_t)(warp * 32) << 16);
            TOut* Y = static_cast<TOut*>(a.Y);
            #pragma unroll 1
            for (int c = 0; c < W8_BN / 32; ++c) {
                uint32_t hh[32], mx[32], ll[32];
                tmem_ld_32x32b_x32(tl + TM_HH + 32 * c, hh);
                tmem_ld_32x32b_x32(tl + TM_MIX + 32 * c, mx);
                tmem_ld_32x32b_x32(tl + TM_LL + 32 * c, ll);
                tmem_ld_wait();
                const int col0 = n0 + 32 * c;
                float y[32];
                int acc[32];
                #pragma unroll
                for (int k = 0; k < 32; ++k) {
                    acc[k] = 256 * __float2int_rn(__uint_as_float(hh[k])) + 16 * __float2int_rn(__uint_as_float(mx[k])) +
                             __float2int_rn(__uint_as_float(ll[k]));
                    y[k] = __fmul_rn(__fmul_rn(__int2float_rn(acc[k]), sa), __ldg(a.s_w + col0 + k));
                    if (a.bias != nullptr) y[k] = __fadd_rn(y[k], __ldg(a.bias + col0 + k));
                }
                if (valid) {
                    W8Out<TOut>::store(Y + (size_t)row * a.N + col0, y);
                    if (a.acc_dbg != nullptr) {
                        int4* d4 = reinterpret_cast<int4*>(a.acc_dbg + (size_t)row * a.N + col0);
                        #pragma unroll
                        for (int u = 0; u < 8; ++u) d4[u] = make_int4(acc[4 * u], acc[4 * u + 1], acc[4 * u + 2], acc[4 * u + 3]);
                    }
                }
            }
        }
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_W8); }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == W8_MMA_WARP) tmem_dealloc(tmem, 512);
}

// 8-bit weight codes [N][K] (bytes) -> their E4M3 split [N][2K]: one thread
// per 8 codes.
__global__ void __launch_bounds__(256) w8_split_kernel(const uint8_t* Wq, uint8_t* We, size_t N, int K) {
    const size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x;     // group of 8 codes
    const size_t groups = N * (size_t)(K / 8);
    if (i >= groups) return;
    const size_t row = i / (size_t)(K / 8);
    const int k0 = (int)(i - row * (size_t)(K / 8)) * 8;
    const uint2 w = *reinterpret_cast<const uint2*>(Wq + row * K + k0);
    uint16_t hh[4], ll[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        const uint32_t word = k < 2 ? w.x : w.y;
        const int q0 = (int)(int8_t)(word >> (16 * (k & 1))), q1 = (int)(int8_t)(word >> (16 * (k & 1) + 8));
        const int l0 = ((q0 + 8) & 15) - 8, l1 = ((q1 + 8) & 15) - 8;
        const int h0 = (q0 - l0) >> 4, h1 = (q1 - l1) >> 4;
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(hh[k]) : "f"((float)h1), "f"((float)h0));
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(ll[k]) : "f"((float)l1), "f"((float)l0));
    }
    *reinterpret_cast<uint2*>(We + row * 2 * K + k0) =
        make_uint2((uint32_t)hh[0] | ((uint32_t)hh[1] << 16), (uint32_t)hh[2] | ((uint32_t)hh[3] << 16));
    *reinterpret_cast<uint2*>(We + row * 2 * K + K + k0) =
        make_uint2((uint32_t)ll[0] | ((uint32_t)ll[1] << 16), (uint32_t)ll[2] | ((uint32_t)ll[3] << 16));
}

bool encode_split_tmap(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols};
    const cuuint32_t box[2] = {W8_BK, 128};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <typename TOut>
cudaError_t launch_typed(const GemmArgs& a, const CUtensorMap& ta, const CUtensorMap& tw, cudaStream_t stream) {
    static DeviceCache<int> attr;
    int done = 0;
    const cudaError_t e = attr.get(&done, [](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(w8a8_gemm_kernel<TOut>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)W8_SMEM);
    });
    if (e != cudaSuccess) return e;
    const dim3 grid((a.L + W8_BM - 1) / W8_BM, a.N / W8_BN);
    w8a8_gemm_kernel<TOut><<<grid, W8_THREADS, W8_SMEM, stream>>>(a, ta, tw);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_w8a8_gemm(const GemmArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    CUtensorMap ta, tw;
    if (!encode_split_tmap(&ta, a.Xe, (uint64_t)a.L, 2 * (uint64_t)a.K) ||
        !encode_split_tmap(&tw, a.We, (uint64_t)a.N, 2 * (uint64_t)a.K))
        return cudaErrorInvalidValue;
    switch (a.y_dtype) {
        case STARQ_F16: return launch_typed<__half>(a, ta, tw, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(a, ta, tw, stream);
        case STARQ_F32: return launch_typed<float>(a, ta, tw, stream);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_w8_split(const uint8_t* Wq, uint8_t* We, size_t N, int K, cudaStream_t stream) {
    const size_t groups = N * (size_t)(K / 8);
    if (groups == 0) return cudaSuccess;
    w8_split_kernel<<<(unsigned)((groups + 255) / 256), 256, 0, stream>>>(Wq, We, N, K);
    return cudaGetLastError();
}

}  // namespace starq
