// W4A4 GEMM with fused dequantisation (Sec. 3.2 Eq. 13, Sec. 3.1 Eq. 3, 5).
//
//   acc[i][n] = sum_k qa[i][k] qw[n][k]        exact integer accumulation
//   Y[i][n]   = fl(fl(acc * s_a[i]) * s_w[n]) (+ bias[n]) -> output type
//
// sm_103a has no integer tcgen05 MMA, so the codes are multiplied as E4M3:
// every int4 value in [-8, 7] is exact in E4M3, each product (|p| <= 64)
// is exact, and every partial sum is an integer below 49 * 65536 < 2^22,
// which float32 holds exactly. The tensor core accumulates in float32 in
// TMEM; the epilogue reads back exact integers.
//
// One persistent CTA per SM, warp-specialised:
//   warps 0-3   epilogue: tcgen05.ld of the accumulator (warp w reads TMEM
//               lanes 32w..32w+31 = tile rows), dequantise, store Y.
//   warp 4      TMEM allocation; lane 0 issues tcgen05.mma and commits.
//   warps 5-12  converters: 128-bit loads of packed int4 rows from global
//               memory, nibble -> E4M3 by byte permutes, stores into the
//               128-byte-swizzled K-major layout the MMA descriptors read.
// Tiles are 128 tokens x 256 output channels; K runs in 128-element stages
// through a 4-deep shared-memory ring (48 KB per stage). Two 256-column
// accumulators in TMEM let the epilogue of tile t overlap the MMAs of t+1.
// Every mbarrier wait is bounded; a CTA that gives up records it in the
// status word, drains its MMAs and frees TMEM before returning.
#include "common.cuh"

namespace starq {
namespace {

constexpr int BM = 128;               // tokens per tile (MMA M)
constexpr int BN = 256;               // output channels per tile (MMA N)
constexpr int BK = 128;               // K elements per stage (bytes of E4M3)
constexpr int UMMA_K = 32;            // K per tcgen05.mma for 8-bit inputs
constexpr int STAGES = 4;
constexpr int A_STAGE_BYTES = BM * BK;                   // 16 KB
constexpr int B_STAGE_BYTES = BN * BK;                   // 32 KB
constexpr int STAGE_BYTES = A_STAGE_BYTES + B_STAGE_BYTES;
constexpr int NUM_EPI_WARPS = 4;
constexpr int MMA_WARP = 4;
constexpr int FIRST_CONV_WARP = 5;
constexpr int NUM_CONV_WARPS = 8;
constexpr int NUM_CONV_THREADS = NUM_CONV_WARPS * 32;
constexpr int THREADS = (FIRST_CONV_WARP + NUM_CONV_WARPS) * 32;   // 416
constexpr int TMEM_COLS = 512;                            // 2 x 256 fp32 columns
constexpr int A_LOADS = BM * (BK / 2) / 16;               // 16-byte packed loads: 512
constexpr int B_LOADS = BN * (BK / 2) / 16;               // 1024
constexpr int A_PER_THREAD = A_LOADS / NUM_CONV_THREADS;  // 2
constexpr int B_PER_THREAD = B_LOADS / NUM_CONV_THREADS;  // 4
constexpr size_t SMEM_BYTES = (size_t)STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;

static_assert(A_LOADS % NUM_CONV_THREADS == 0 && B_LOADS % NUM_CONV_THREADS == 0, "");

// Instruction descriptor: F32 accumulator, A = B = E4M3, both K-major,
// N = BN, M = BM.
constexpr uint32_t IDESC = (1u << 4) | (0u << 7) | (0u << 10) |
                           ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);

struct Smem {
    uint64_t full[STAGES];
    uint64_t empty[STAGES];
    uint64_t tmem_full[2];
    uint64_t tmem_empty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

// Convert one 16-byte load (32 codes of one row, K elements 32q..32q+31 of
// the stage) and store it as two 16-byte chunks of E4M3.
__device__ __forceinline__ void convert_store(uint32_t tile, int row, int q, uint4 w) {
    uint32_t o[8];
    int4x8_to_e4m3x8(w.x, o[0], o[1]);
    int4x8_to_e4m3x8(w.y, o[2], o[3]);
    int4x8_to_e4m3x8(w.z, o[4], o[5]);
    int4x8_to_e4m3x8(w.w, o[6], o[7]);
    st_shared_v4(tile + sw128_offset(row, 2 * q), o[0], o[1], o[2], o[3]);
    st_shared_v4(tile + sw128_offset(row, 2 * q + 1), o[4], o[5], o[6], o[7]);
}

template <typename TOut> struct Out;
template <> struct Out<__half> {
    static __device__ __forceinline__ void store32(__half* p, const float (&y)[32]) {
        uint4* q = reinterpret_cast<uint4*>(p);
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                __half2 h = __floats2half2_rn(y[8 * u + 2 * j], y[8 * u + 2 * j + 1]);
                w[j] = *reinterpret_cast<uint32_t*>(&h);
            }
            q[u] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
};
template <> struct Out<__nv_bfloat16> {
    static __device__ __forceinline__ void store32(__nv_bfloat16* p, const float (&y)[32]) {
        uint4* q = reinterpret_cast<uint4*>(p);
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            uint32_t w[4];
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                __nv_bfloat162 h = __floats2bfloat162_rn(y[8 * u + 2 * j], y[8 * u + 2 * j + 1]);
                w[j] = *reinterpret_cast<uint32_t*>(&h);
            }
            q[u] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
};
template <> struct Out<float> {
    static __device__ __forceinline__ void store32(float* p, const float (&y)[32]) {
        float4* q = reinterpret_cast<float4*>(p);
        #pragma unroll
        for (int u = 0; u < 8; ++u) q[u] = make_float4(y[4 * u], y[4 * u + 1], y[4 * u + 2], y[4 * u + 3]);
    }
};

template <typename TOut>
__global__ void __launch_bounds__(THREADS, 1)
w4a4_gemm_kernel(GemmArgs a) {
    extern __shared__ uint8_t smem_raw[];
    // 1024-byte alignment for the swizzle atoms
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* base_ptr = smem_raw + (base - raw);
    Smem* sh = reinterpret_cast<Smem*>(base_ptr + STAGES * STAGE_BYTES);
    volatile int* abort = &sh->abort;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int L = a.L, N = a.N, K = a.K;
    const int num_m = (L + BM - 1) / BM;
    const int num_n = (N + BN - 1) / BN;
    const int num_tiles = num_m * num_n;
    const int num_k = K / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_addr(&sh->full[s]), NUM_CONV_THREADS);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tmem_full[b]), 1);
            mbar_init(smem_addr(&sh->tmem_empty[b]), NUM_EPI_WARPS * 32);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        sh->abort = 0;
        mbar_fence_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc(smem_addr(&sh->tmem_base), TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = sh->tmem_base;

    if (warp >= FIRST_CONV_WARP) {
        // ------------------------------------------------------------------
        // Converters
        // ------------------------------------------------------------------
        const int ct = threadIdx.x - FIRST_CONV_WARP * 32;
        const size_t row_bytes = (size_t)K / 2;
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x) {
            const int m0 = (tile % num_m) * BM;
            const int n0 = (tile / num_m) * BN;
            for (int kc = 0; kc < num_k; ++kc) {
                uint4 wa[A_PER_THREAD], wb[B_PER_THREAD];
                #pragma unroll
                for (int u = 0; u < A_PER_THREAD; ++u) {
                    const int idx = ct + u * NUM_CONV_THREADS;
                    const int r = idx >> 2, q = idx & 3;
                    wa[u] = (m0 + r < L)
                        ? ld_global_nc_v4(a.Xq + (size_t)(m0 + r) * row_bytes + kc * (BK / 2) + q * 16)
                        : make_uint4(0, 0, 0, 0);
                }
                #pragma unroll
                for (int u = 0; u < B_PER_THREAD; ++u) {
                    const int idx = ct + u * NUM_CONV_THREADS;
                    const int r = idx >> 2, q = idx & 3;
                    wb[u] = (n0 + r < N)
                        ? ld_global_nc_v4(a.Wq + (size_t)(n0 + r) * row_bytes + kc * (BK / 2) + q * 16)
                        : make_uint4(0, 0, 0, 0);
                }
                if (!mbar_wait_bounded(smem_addr(&sh->empty[stage]), phase ^ 1u, abort)) {
                    ok = false;
                    break;
                }
                const uint32_t sA = base + stage * STAGE_BYTES;
                const uint32_t sB = sA + A_STAGE_BYTES;
                #pragma unroll
                for (int u = 0; u < A_PER_THREAD; ++u) {
                    const int idx = ct + u * NUM_CONV_THREADS;
                    convert_store(sA, idx >> 2, idx & 3, wa[u]);
                }
                #pragma unroll
                for (int u = 0; u < B_PER_THREAD; ++u) {
                    const int idx = ct + u * NUM_CONV_THREADS;
                    convert_store(sB, idx >> 2, idx & 3, wb[u]);
                }
                fence_proxy_async_smem();
                mbar_arrive(smem_addr(&sh->full[stage]));
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
        }
        if (!ok) {
            sh->abort = 1;
            atomicOr(a.status, STATUS_TIMEOUT_GEMM);
        }
    } else if (warp == MMA_WARP) {
        // ------------------------------------------------------------------
        // MMA issuer (one thread)
        // ------------------------------------------------------------------
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int it = 0;
            for (int tile = blockIdx.x; tile < num_tiles && ok; tile += gridDim.x, ++it) {
                const int acc = it & 1;
                const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
                if (!mbar_wait_bounded(smem_addr(&sh->tmem_empty[acc]), acc_phase ^ 1u, abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
                for (int kc = 0; kc < num_k; ++kc) {
                    if (!mbar_wait_bounded(smem_addr(&sh->full[stage]), phase, abort)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sA = base + stage * STAGE_BYTES;
                    const uint32_t sB = sA + A_STAGE_BYTES;
                    #pragma unroll
                    for (int ks = 0; ks < BK / UMMA_K; ++ks) {
                        mma_f8f6f4(d_tmem, smem_desc_sw128(sA + ks * UMMA_K),
                                   smem_desc_sw128(sB + ks * UMMA_K), IDESC,
                                   (kc > 0 || ks > 0) ? 1u : 0u);
                    }
                    tc_commit(smem_addr(&sh->empty[stage]));
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                tc_commit(smem_addr(&sh->tmem_full[acc]));
            }
            // Wait for every MMA this thread issued before TMEM is released.
            tc_commit(smem_addr(&sh->drain));
            volatile int never = 0;
            if (!mbar_wait_bounded(smem_addr(&sh->drain), 0, &never)) ok = false;
            if (!ok) {
                sh->abort = 1;
                atomicOr(a.status, STATUS_TIMEOUT_GEMM);
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------------
        // Epilogue: warp w owns TMEM lanes / tile rows 32w .. 32w + 31
        // ------------------------------------------------------------------
        bool ok = true;
        int it = 0;
        TOut* Y = static_cast<TOut*>(a.Y);
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++it) {
            const int m0 = (tile % num_m) * BM;
            const int n0 = (tile / num_m) * BN;
            const int acc = it & 1;
            const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
            if (!mbar_wait_bounded(smem_addr(&sh->tmem_full[acc]), acc_phase, abort)) {
                ok = false;
                break;
            }
            tc_fence_after();
            const int row = m0 + warp * 32 + lane;
            const bool valid = row < L;
            const float sa = valid ? __ldg(a.s_a + row) : 0.f;
            const uint32_t t_row = tmem_base + ((uint32_t)(warp * 32) << 16) + (uint32_t)(acc * BN);
            #pragma unroll 1
            for (int c = 0; c < BN / 32; ++c) {
                const int nc = n0 + c * 32;
                if (nc >= N) break;
                uint32_t r[32];
                tmem_ld_32x32b_x32(t_row + c * 32, r);
                tmem_ld_wait();
                if (valid) {
                    float y[32];
                    const float4* sw4 = reinterpret_cast<const float4*>(a.s_w + nc);
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 sw = __ldg(sw4 + u);
                        y[4 * u] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u]), sa), sw.x);
                        y[4 * u + 1] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 1]), sa), sw.y);
                        y[4 * u + 2] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 2]), sa), sw.z);
                        y[4 * u + 3] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 3]), sa), sw.w);
                    }
                    if (a.bias != nullptr) {
                        const float4* b4 = reinterpret_cast<const float4*>(a.bias + nc);
                        #pragma unroll
                        for (int u = 0; u < 8; ++u) {
                            const float4 b = __ldg(b4 + u);
                            y[4 * u] = __fadd_rn(y[4 * u], b.x);
                            y[4 * u + 1] = __fadd_rn(y[4 * u + 1], b.y);
                            y[4 * u + 2] = __fadd_rn(y[4 * u + 2], b.z);
                            y[4 * u + 3] = __fadd_rn(y[4 * u + 3], b.w);
                        }
                    }
                    Out<TOut>::store32(Y + (size_t)row * N + nc, y);
                    if (a.acc_dbg != nullptr) {
                        int4* d4 = reinterpret_cast<int4*>(a.acc_dbg + (size_t)row * N + nc);
                        #pragma unroll
                        for (int u = 0; u < 8; ++u)
                            d4[u] = make_int4(__float2int_rn(__uint_as_float(r[4 * u])),
                                              __float2int_rn(__uint_as_float(r[4 * u + 1])),
                                              __float2int_rn(__uint_as_float(r[4 * u + 2])),
                                              __float2int_rn(__uint_as_float(r[4 * u + 3])));
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(smem_addr(&sh->tmem_empty[acc]));
        }
        if (!ok) {
            sh->abort = 1;
            atomicOr(a.status, STATUS_TIMEOUT_GEMM);
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == MMA_WARP) tmem_dealloc(tmem_base, TMEM_COLS);
}

template <typename TOut>
cudaError_t launch_typed(const GemmArgs& a, cudaStream_t stream) {
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 64 && !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(w4a4_gemm_kernel<TOut>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set[dev] = true;
    }
    const int num_tiles = ((a.L + BM - 1) / BM) * ((a.N + BN - 1) / BN);
    const int grid = num_tiles < num_sms() ? num_tiles : num_sms();
    w4a4_gemm_kernel<TOut><<<grid, THREADS, SMEM_BYTES, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    switch (a.y_dtype) {
        case STARQ_F16: return launch_typed<__half>(a, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_typed<float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
