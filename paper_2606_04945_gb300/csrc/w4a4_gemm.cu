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
#include <cuda.h>
#include <cudaTypedefs.h>

#include "common.cuh"
#include "w8a8.cuh"

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
// (a s, b s) then (. * t0, . * t1): two packed round-to-nearest multiplies,
// each half rounding like the scalar operation.
__device__ __forceinline__ void mul2_rn(float a, float b, float s, float t0, float t1, float& y0, float& y1) {
    asm("{\n\t.reg .b64 V, S, T;\n\t"
        "mov.b64 V, {%2, %3};\n\t"
        "mov.b64 S, {%4, %4};\n\t"
        "mov.b64 T, {%5, %6};\n\t"
        "mul.rn.f32x2 V, V, S;\n\t"
        "mul.rn.f32x2 V, V, T;\n\t"
        "mov.b64 {%0, %1}, V;\n\t}"
        : "=f"(y0), "=f"(y1) : "f"(a), "f"(b), "f"(s), "f"(t0), "f"(t1));
}

// Row `row` (32 values) of a 32 x 32 output box staged for a TMA store:
// 16-bit types use 64-byte rows with the 64-byte swizzle (16-byte group g at
// g ^ ((row >> 1) & 3)), float uses 128-byte rows with the 128-byte swizzle
// (g ^ (row & 7)); either way the 32 lanes of a warp write without bank
// conflicts.
template <typename T2, typename Cvt>
__device__ __forceinline__ void stage_row16(uint32_t box, int row, const float (&y)[32], Cvt cvt) {
    #pragma unroll
    for (int g = 0; g < 4; ++g) {
        uint32_t w[4];
        #pragma unroll
        for (int j = 0; j < 4; ++j) {
            T2 h = cvt(y[8 * g + 2 * j], y[8 * g + 2 * j + 1]);
            w[j] = *reinterpret_cast<uint32_t*>(&h);
        }
        st_shared_v4(box + row * 64 + 16 * (g ^ ((row >> 1) & 3)), w[0], w[1], w[2], w[3]);
    }
}
// Row `row` (16 values) of a 32 x 16 box of a 16-bit type: 32-byte rows
// with the 32-byte swizzle (16-byte group g at g ^ ((row >> 2) & 1)), which
// keeps the 32 lanes' stores free of bank conflicts.
template <typename T2, typename Cvt>
__device__ __forceinline__ void stage_row16_half(uint32_t box, int row, const float (&h)[16], Cvt cvt) {
    #pragma unroll
    for (int g = 0; g < 2; ++g) {
        uint32_t w[4];
        #pragma unroll
        for (int j = 0; j < 4; ++j) {
            T2 v = cvt(h[8 * g + 2 * j], h[8 * g + 2 * j + 1]);
            w[j] = *reinterpret_cast<uint32_t*>(&v);
        }
        st_shared_v4(box + row * 32 + 16 * (g ^ ((row >> 2) & 1)), w[0], w[1], w[2], w[3]);
    }
}
template <> struct Out<__half> {
    static constexpr CUtensorMapDataType TMAP_TYPE = CU_TENSOR_MAP_DATA_TYPE_FLOAT16;
    static constexpr CUtensorMapSwizzle TMAP_SWIZZLE = CU_TENSOR_MAP_SWIZZLE_64B;
    static __device__ __forceinline__ void stage32(uint32_t box, int row, const float (&y)[32]) {
        stage_row16<__half2>(box, row, y, [](float a, float b) { return __floats2half2_rn(a, b); });
    }
    static __device__ __forceinline__ void stage16(uint32_t box, int row, const float (&h)[16]) {
        stage_row16_half<__half2>(box, row, h, [](float a, float b) { return __floats2half2_rn(a, b); });
    }
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
    static constexpr CUtensorMapDataType TMAP_TYPE = CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    static constexpr CUtensorMapSwizzle TMAP_SWIZZLE = CU_TENSOR_MAP_SWIZZLE_64B;
    static __device__ __forceinline__ void stage32(uint32_t box, int row, const float (&y)[32]) {
        stage_row16<__nv_bfloat162>(box, row, y, [](float a, float b) { return __floats2bfloat162_rn(a, b); });
    }
    static __device__ __forceinline__ void stage16(uint32_t box, int row, const float (&h)[16]) {
        stage_row16_half<__nv_bfloat162>(box, row, h, [](float a, float b) { return __floats2bfloat162_rn(a, b); });
    }
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
    static constexpr CUtensorMapDataType TMAP_TYPE = CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
    static constexpr CUtensorMapSwizzle TMAP_SWIZZLE = CU_TENSOR_MAP_SWIZZLE_128B;
    static __device__ __forceinline__ void stage16(uint32_t, int, const float (&)[16]) {}   // 16-bit outputs only
    static __device__ __forceinline__ void stage32(uint32_t box, int row, const float (&y)[32]) {
        #pragma unroll
        for (int g = 0; g < 8; ++g)
            st_shared_v4(box + row * 128 + 16 * (g ^ (row & 7)), __float_as_uint(y[4 * g]),
                         __float_as_uint(y[4 * g + 1]), __float_as_uint(y[4 * g + 2]), __float_as_uint(y[4 * g + 3]));
    }
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

// ---------------------------------------------------------------------------
// CTA-pair kernel: activation codes as E4M3 bytes by TMA, packed int4
// weights by TMA into a staging buffer and converted in shared memory.
//
// Two CTAs of a cluster share one 256 x 256 output tile through
// tcgen05.mma.cta_group::2 (M = 256, N = 256, K = 32 per instruction): CTA r
// holds tokens m0 + 128 r .. + 127 of A and output channels n0 + 128 r ..
// + 127 of B, and receives rows 128 r .. of the accumulator in its own TMEM.
// Each CTA therefore converts only its half of the weight tile. The leader
// (rank 0) issues the MMAs once both CTAs' converters have arrived on its
// stage barrier, and its commits arrive on the stage / accumulator barriers
// of both CTAs. Roles per CTA (20 warps): 0-7 epilogue, 8 TMA producers
// (activations; raw weights), 9 TMEM allocation + (leader) MMA issue, 10-19
// converters, two per stage buffer. Every CTA loads its own activation rows
// (no cluster multicast).
// ---------------------------------------------------------------------------
namespace pairk {
constexpr int BM = 128;                    // token rows per CTA (M = 256 per pair)
constexpr int BN = 256;                    // output channels per pair tile
constexpr int BN_CTA = 128;                // ... per CTA
constexpr int BK = 128;                    // K elements per stage
constexpr int UMMA_K = 32;
constexpr int STAGES = 5;
constexpr int A_BYTES = BM * BK;                       // 16 KB E4M3
constexpr int B_BYTES = BN_CTA * BK;                   // 16 KB E4M3 (converted)
constexpr int BRAW_BYTES = BN_CTA * BK / 2;            // 8 KB packed int4
constexpr int STAGE_BYTES = A_BYTES + B_BYTES + BRAW_BYTES;
constexpr int NUM_EPI_WARPS = 8;           // lane quarter w % 4, column half w / 4
constexpr int TMA_WARP = 8;                // lane 0: activation tiles, lane 1: raw weight tiles
constexpr int MMA_WARP = 9;
constexpr int FIRST_CONV_WARP = 10;
constexpr int CONV_WARPS_PER_STAGE = 2;    // each converts half of a stage's rows
constexpr int NUM_CONV_WARPS = CONV_WARPS_PER_STAGE * STAGES;
constexpr int THREADS = (FIRST_CONV_WARP + NUM_CONV_WARPS) * 32;   // 640
constexpr int TMEM_COLS = 512;
constexpr int EPI_PARAM_BYTES = NUM_EPI_WARPS * 2 * (BN / 2) * 4;   // s_w and bias, 128 columns per warp
constexpr size_t SMEM_BYTES = (size_t)STAGES * STAGE_BYTES + EPI_PARAM_BYTES + 1024 + 512;
constexpr uint32_t IDESC = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)((2 * BM) >> 4) << 24);
static_assert(BRAW_BYTES % (16 * 32 * CONV_WARPS_PER_STAGE) == 0, "");

struct Smem {
    uint64_t a_full[STAGES];      // activation tile landed (TMA bytes)
    uint64_t raw_full[STAGES];    // packed weight tile landed (TMA bytes)
    uint64_t raw_empty[STAGES];   // converters done reading the packed tile
    uint64_t full[STAGES];        // leader: converter warps of the pair
    uint64_t empty[STAGES];       // MMA commit (to both CTAs of the pair)
    uint64_t tmem_full[2];        // MMA commit (to both CTAs of the pair)
    uint64_t tmem_empty[2];       // leader: epilogue warps of the pair
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};
}  // namespace pairk

template <typename TOut>
__global__ void __launch_bounds__(pairk::THREADS, 1)
w4a4_gemm_pair_kernel(GemmArgs a, const __grid_constant__ CUtensorMap tmap_a,
                      const __grid_constant__ CUtensorMap tmap_b) {
    constexpr int BM = pairk::BM, BN = pairk::BN, BN_CTA = pairk::BN_CTA, BK = pairk::BK;
    constexpr int UMMA_K = pairk::UMMA_K, STAGES = pairk::STAGES, STAGE_BYTES = pairk::STAGE_BYTES;
    constexpr int A_BYTES = pairk::A_BYTES, B_BYTES = pairk::B_BYTES, BRAW_BYTES = pairk::BRAW_BYTES;
    constexpr int TMA_WARP = pairk::TMA_WARP, MMA_WARP = pairk::MMA_WARP;
    constexpr int FIRST_CONV_WARP = pairk::FIRST_CONV_WARP;
    constexpr int CONV_WARPS_PER_STAGE = pairk::CONV_WARPS_PER_STAGE;
    constexpr int NUM_EPI_WARPS = pairk::NUM_EPI_WARPS;
    constexpr int TMEM_COLS = pairk::TMEM_COLS;
    constexpr uint32_t IDESC = pairk::IDESC;
    constexpr uint16_t PAIR = 3u;                 // both CTAs of the cluster (one pair)
    using Smem = pairk::Smem;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    Smem* sh = reinterpret_cast<Smem*>(smem_raw + (base - raw) + STAGES * STAGE_BYTES);
    volatile int* abort = &sh->abort;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t half = cluster_ctarank();     // position inside the CTA pair
    const uint32_t leader = 0;
    const int L = a.L, N = a.N, K = a.K;
    // Pair tile: 256 tokens x 256 channels.
    const int num_m = (L + 2 * BM - 1) / (2 * BM);
    const int num_n = (N + BN - 1) / BN;
    const int num_tiles = num_m * num_n;
    const int num_k = K / BK;
    const int cluster = blockIdx.x / 2;
    const int num_clusters = gridDim.x / 2;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_addr(&sh->a_full[s]), 1);
            mbar_init(smem_addr(&sh->raw_full[s]), 1);
            mbar_init(smem_addr(&sh->raw_empty[s]), CONV_WARPS_PER_STAGE);
            mbar_init(smem_addr(&sh->full[s]), 2 * CONV_WARPS_PER_STAGE);  // converter warps of the pair
            mbar_init(smem_addr(&sh->empty[s]), 1);                        // the pair's MMA commit
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tmem_full[b]), 1);
            mbar_init(smem_addr(&sh->tmem_empty[b]), 2 * NUM_EPI_WARPS);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        sh->abort = 0;
        mbar_fence_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc_pair(smem_addr(&sh->tmem_base), TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();              // barriers of every CTA initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem_base = sh->tmem_base;

    if (warp == TMA_WARP) {
        // Lane 0 streams activation tiles into a stage once every pair of
        // the cluster has finished the MMAs on it; lane 1 streams packed
        // weight tiles into the staging buffer as soon as the converters have
        // read the previous one, so the raw weights of a stage arrive well
        // before its MMA slot frees.
        if (lane < 2) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int tile = cluster; tile < num_tiles && ok; tile += num_clusters) {
                const int m_rows = (tile % num_m) * 2 * BM + (int)half * BM;
                const int n_rows = (tile / num_m) * BN + (int)half * BN_CTA;
                for (int kc = 0; kc < num_k; ++kc) {
                    const uint32_t st = base + stage * STAGE_BYTES;
                    if (lane == 0) {
                        if (!mbar_wait_bounded(smem_addr(&sh->empty[stage]), phase ^ 1u, abort)) { ok = false; break; }
                        const uint32_t bar = smem_addr(&sh->a_full[stage]);
                        mbar_arrive_expect_tx(bar, A_BYTES);
                        tma_load_2d(st, &tmap_a, kc * BK, m_rows, bar);
                    } else {
                        if (!mbar_wait_bounded(smem_addr(&sh->raw_empty[stage]), phase ^ 1u, abort)) { ok = false; break; }
                        const uint32_t bar = smem_addr(&sh->raw_full[stage]);
                        mbar_arrive_expect_tx(bar, BRAW_BYTES);
                        tma_load_2d(st + A_BYTES + B_BYTES, &tmap_b, kc * (BK / 2), n_rows, bar);
                    }
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
        }
        __syncwarp();
    } else if (warp >= FIRST_CONV_WARP) {
        // Converter warps (cw % STAGES) own stage buffer cw % STAGES and
        // convert its phases in order (stages g = buffer, buffer + STAGES,
        // ... of the CTA's sequence), each the half of the rows given by
        // cw / STAGES. All stage buffers convert concurrently, and a parity
        // wait can never be two phases ahead of its barrier. One
        // cluster-scope arrive per warp and stage tells the pair's leader
        // that its rows are ready.
        const int cw = warp - FIRST_CONV_WARP;
        const int buf = cw % STAGES;
        const int row0 = (cw / STAGES) * (BN_CTA / CONV_WARPS_PER_STAGE);
        const uint32_t leader_full0 = mapa_shared(smem_addr(&sh->full[0]), leader);
        const int my_tiles = cluster < num_tiles ? (num_tiles - 1 - cluster) / num_clusters + 1 : 0;
        const int total = my_tiles * num_k;
        bool ok = true;
        for (int g = buf; g < total; g += STAGES) {
            const int stage = buf;
            const uint32_t k = (uint32_t)(g / STAGES);          // phase index of this buffer
            if (!mbar_wait_bounded(smem_addr(&sh->raw_full[stage]), k & 1u, abort)) { ok = false; break; }
            // the converted tile overwrites the previous phase's MMA operand
            if (k > 0 && !mbar_wait_bounded(smem_addr(&sh->empty[stage]), (k - 1) & 1u, abort)) { ok = false; break; }
            const uint32_t st = base + stage * STAGE_BYTES;
            const uint32_t sB = st + A_BYTES, sRaw = st + A_BYTES + B_BYTES;
            #pragma unroll 4
            for (int u = 0; u < BRAW_BYTES / 16 / 32 / CONV_WARPS_PER_STAGE; ++u) {
                const int idx = lane + 32 * u;
                const int r = row0 + (idx >> 2), q = idx & 3;
                convert_store(sB, r, q, ld_shared_v4(sRaw + r * (BK / 2) + q * 16));
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_addr(&sh->raw_empty[stage]));
            fence_proxy_async_smem();
            // the stage is ready for the MMA once this CTA's activation tile landed too
            if (!mbar_wait_bounded(smem_addr(&sh->a_full[stage]), k & 1u, abort)) { ok = false; break; }
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(leader_full0 + stage * 8);
        }
        if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
    } else if (warp == MMA_WARP) {
        if (lane == 0 && half == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int it = 0;
            for (int tile = cluster; tile < num_tiles && ok; tile += num_clusters, ++it) {
                const int acc = it & 1;
                const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
                if (!mbar_wait_bounded(smem_addr(&sh->tmem_empty[acc]), acc_phase ^ 1u, abort)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
                for (int kc = 0; kc < num_k; ++kc) {
                    if (!mbar_wait_bounded(smem_addr(&sh->full[stage]), phase, abort)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t sA = base + stage * STAGE_BYTES;
                    const uint32_t sB = sA + A_BYTES;
                    #pragma unroll
                    for (int ks = 0; ks < BK / UMMA_K; ++ks)
                        mma_f8f6f4_pair(d_tmem, smem_desc_sw128(sA + ks * UMMA_K),
                                        smem_desc_sw128(sB + ks * UMMA_K), IDESC,
                                        (kc > 0 || ks > 0) ? 1u : 0u);
                    // the stage may be refilled once the pair's MMAs are done with it
                    tc_commit_pair_multicast(smem_addr(&sh->empty[stage]), PAIR);
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                tc_commit_pair_multicast(smem_addr(&sh->tmem_full[acc]), PAIR);
            }
            tc_commit_pair_multicast(smem_addr(&sh->drain), PAIR);
            if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
        }
        __syncwarp();
    } else {
        // epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31 of this CTA,
        // columns (w / 4) * 128 .. + 127 of the tile. Its per-channel scales
        // and biases are staged in its own shared slice while the tile's
        // MMAs run, so no global-load latency follows the accumulator.
        const uint32_t leader_tmem_empty0 = mapa_shared(smem_addr(&sh->tmem_empty[0]), leader);
        float* epi_sw = reinterpret_cast<float*>(smem_raw + (base - raw) + STAGES * STAGE_BYTES + sizeof(Smem) +
                                                 (16 - sizeof(Smem) % 16) % 16) + warp * 2 * (BN / 2);
        float* epi_b = epi_sw + BN / 2;
        const int quarter = warp & 3, chalf = warp >> 2;
        bool ok = true;
        int it = 0;
        TOut* Y = static_cast<TOut*>(a.Y);
        for (int tile = cluster; tile < num_tiles; tile += num_clusters, ++it) {
            const int m0 = (tile % num_m) * 2 * BM + (int)half * BM;
            const int n0 = (tile / num_m) * BN;
            const int acc = it & 1;
            const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
            const int row = m0 + quarter * 32 + lane;
            const bool valid = row < L;
            const float sa = valid ? __ldg(a.s_a + row) : 0.f;
            {
                const int ncol = n0 + chalf * (BN / 2) + 4 * lane;      // 4 columns per lane
                float4 w = make_float4(0.f, 0.f, 0.f, 0.f), b = w;
                if (ncol < N) {
                    w = __ldg(reinterpret_cast<const float4*>(a.s_w + ncol));
                    if (a.bias != nullptr) b = __ldg(reinterpret_cast<const float4*>(a.bias + ncol));
                }
                __syncwarp();          // the previous tile's reads of the slice are done
                reinterpret_cast<float4*>(epi_sw)[lane] = w;
                reinterpret_cast<float4*>(epi_b)[lane] = b;
                __syncwarp();
            }
            if (!mbar_wait_bounded(smem_addr(&sh->tmem_full[acc]), acc_phase, abort)) { ok = false; break; }
            tc_fence_after();
            const uint32_t t_row = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * BN);
            #pragma unroll 1
            for (int cc = 0; cc < BN / 64; ++cc) {
                const int c = chalf * (BN / 64) + cc;
                const int nc = n0 + c * 32;
                if (nc >= N) break;
                uint32_t r[32];
                tmem_ld_32x32b_x32(t_row + c * 32, r);
                tmem_ld_wait();
                if (valid) {
                    float y[32];
                    const float4* sw4 = reinterpret_cast<const float4*>(epi_sw + cc * 32);
                    const float4* b4 = reinterpret_cast<const float4*>(epi_b + cc * 32);
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 sw = sw4[u];
                        y[4 * u] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u]), sa), sw.x);
                        y[4 * u + 1] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 1]), sa), sw.y);
                        y[4 * u + 2] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 2]), sa), sw.z);
                        y[4 * u + 3] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 3]), sa), sw.w);
                    }
                    if (a.bias != nullptr) {
                        #pragma unroll
                        for (int u = 0; u < 8; ++u) {
                            const float4 b = b4[u];
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
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(leader_tmem_empty0 + acc * 8);
        }
        if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
    }

    // every MMA the pair's leader issued has completed before TMEM is released
    if (warp == MMA_WARP && lane == 0) {
        volatile int never = 0;
        if (!mbar_wait_bounded(smem_addr(&sh->drain), 0, &never)) atomicOr(a.status, STATUS_TIMEOUT_GEMM);
    }
    __syncwarp();
    tc_fence_before();
    cluster_sync();              // no CTA leaves while another may still signal it
    tc_fence_after();
    if (warp == MMA_WARP) tmem_dealloc_pair(tmem_base, TMEM_COLS);
}

// Tensor map of a row-major uint8 matrix [rows][cols] with a box of
// box_rows x box_cols bytes.
bool encode_u8_tmap(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                    uint32_t box_cols, CUtensorMapSwizzle swz) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of a row-major K-major operand [rows][cols] of 1- or 2-byte
// elements, box box_rows x box_cols elements, 128-byte swizzle.
bool encode_operand_tmap(CUtensorMap* m, const void* ptr, CUtensorMapDataType type, size_t elem, uint64_t rows,
                         uint64_t cols, uint32_t box_rows, uint32_t box_cols) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * elem};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, type, 2, const_cast<void*>(ptr), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of the row-major output Y [rows][cols] with 32 x 32 boxes.
bool encode_out_tmap(CUtensorMap* m, void* ptr, CUtensorMapDataType type, size_t elem, uint64_t rows,
                     uint64_t cols, CUtensorMapSwizzle swz, uint32_t box_cols = 32) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * elem};
    const cuuint32_t box[2] = {box_cols, 32};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, type, 2, ptr, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
              CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// ---------------------------------------------------------------------------
// CTA-pair GEMM with both operands as E4M3 bytes by TMA (activation codes
// from the quantiser, weight codes from w4_unpack_e4m3).
//
// The standard two-barrier pipeline: the TMA producer of each CTA waits for
// the stage to be free (the pair's MMA commit, which arrives in both CTAs)
// and loads its 128 activation rows and BN / 2 weight rows, the bytes
// counted on the pair leader's stage barrier (cta_group::2); the leader's
// MMA thread waits there and issues the four K = 32 MMAs of the stage
// (M 256, N BN). Every CTA loads only its own rows: no cluster multicast.
// Up to 6 stages of 32 KB; 8 epilogue warps.
// ---------------------------------------------------------------------------
namespace tmak {
constexpr int BM = 128, BK = 128, UMMA_K = 32;
constexpr int A_BYTES = BM * BK;
constexpr int NUM_EPI_WARPS = 8;
constexpr int TMA_WARP = 8, MMA_WARP = 9;
constexpr int THREADS = 10 * 32;
constexpr int TMEM_COLS = 512;
constexpr int ACC_STRIDE = 256;                // TMEM columns from one accumulator to the other
constexpr int EPI_CHUNKS = 4;                  // 32-column chunks per epilogue warp and tile
constexpr int EPI_PARAM_BYTES = NUM_EPI_WARPS * 2 * (EPI_CHUNKS * 32) * 4;
// A CTA pair's output tile is 256 tokens x BN channels; each CTA holds
// BN / 2 weight rows of every stage.
template <int BN>
struct Tile {
    static_assert(BN % 32 == 0 && BN >= 64 && BN <= 256, "pair tile width");
    static constexpr int BN_CTA = BN / 2;
    static constexpr int B_BYTES = BN_CTA * BK;
    static constexpr int STAGE_BYTES = A_BYTES + B_BYTES;       // 32 KB at BN = 256
    static_assert(STAGE_BYTES % 1024 == 0, "stages keep the 1024-byte swizzle alignment");
    static constexpr uint32_t IDESC = (1u << 4) | ((uint32_t)(BN >> 3) << 17) | ((uint32_t)((2 * BM) >> 4) << 24);
};
template <int S>
struct Smem {
    uint64_t full[S];             // pair leader: both CTAs' TMA bytes
    uint64_t empty[S];            // the pair's MMA commit
    uint64_t tmem_full[2];
    uint64_t tmem_empty[2];       // pair leader: epilogue warps of the pair
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};
// Per output element size and tile width: one 32 x 32 staging box per
// epilogue warp, and as many stages (up to 6) as the rest of the 227 KB
// allows: at BN = 256, 6 for 16-bit outputs and 5 for float; at BN = 224, 6.
template <int OUT_BYTES, int BN>
struct Cfg {
    static constexpr int EPI_BOX_WARP_BYTES = 32 * 32 * OUT_BYTES;
    static constexpr int EPI_STAGE_BYTES = NUM_EPI_WARPS * EPI_BOX_WARP_BYTES;
    static constexpr int FIXED = EPI_STAGE_BYTES + EPI_PARAM_BYTES + 1024 + 512;
    static constexpr int FIT = (227 * 1024 - FIXED) / Tile<BN>::STAGE_BYTES;
    static constexpr int STAGES = FIT < 6 ? FIT : 6;
    static constexpr size_t SMEM_BYTES = (size_t)STAGES * Tile<BN>::STAGE_BYTES + FIXED;
    static_assert(STAGES >= 4 && SMEM_BYTES <= 227 * 1024, "shared memory");
};
}  // namespace tmak

// OPK: operand kind -- 0 = E4M3 codes (dequantising epilogue), 1 = fp16,
// 2 = bf16 (plain float32 accumulator cast to the output type), 3 = 8-bit
// codes held as fp16 (exact: |c| <= 127), accumulated in runs of 256 K that
// the epilogue sums in int32 before dequantising. Every kind reads 128-byte
// K rows and advances 32 bytes of K per MMA.
// Tile of the calling thread's last TMA pair GEMM launch: BN * 10 + 2 (CTAs
// per cluster).
thread_local int g_last_tile = 0;
// Most CTA pairs a TMA pair GEMM launched from this thread may use (0 = as
// many as are resident).
thread_local int g_pair_limit = 0;

// Output tiles of the pair GEMM: 256-token rows x BN-channel pair tiles.
int tma_tiles(int L, int N, int BN) {
    const int num_n = (N + BN - 1) / BN;
    return ((L + 2 * tmak::BM - 1) / (2 * tmak::BM)) * num_n;
}
// Estimated cycles of a launch (twice the model's stage cycles per round).
long long tma_round_cost(int L, int N, int BN, int clusters) {
    const long long tiles = tma_tiles(L, N, BN);
    const long long used = clusters < 1 ? 1 : clusters;
    const long long rounds = (tiles + used - 1) / used;
    const long long stage2 = 4LL * BN > 512LL + 3LL * BN ? 4LL * BN : 512LL + 3LL * BN;
    return rounds * stage2;
}

// SWIGLU: the weight rows come interleaved in groups of 16 (gate rows
// 16 k .. 16 k + 15, then the matching up rows), so every 32-column chunk
// of the accumulator holds 16 gate and 16 up channels; the epilogue writes
// silu(gate) * up, rounded once, to column nc / 2 of an [L][N / 2] output.
// G2: a second, independent problem b (the same L, K and output type) whose
// tiles follow a's in the one persistent tile stream, so that a short
// problem's pipeline fill and drain hide behind the other's tiles.
template <typename TOut, int OPK, int BN, bool SWIGLU = false, bool G2 = false>
__global__ void __launch_bounds__(tmak::THREADS, 1)
w4a4_gemm_tma_pair_kernel(GemmArgs a, const __grid_constant__ CUtensorMap tmap_a,
                          const __grid_constant__ CUtensorMap tmap_b, const __grid_constant__ CUtensorMap tmap_y,
                          GemmArgs b, const __grid_constant__ CUtensorMap tmap_a2,
                          const __grid_constant__ CUtensorMap tmap_b2, const __grid_constant__ CUtensorMap tmap_y2) {
    using Tile = tmak::Tile<BN>;
    using Cfg = tmak::Cfg<sizeof(TOut), BN>;
    constexpr int BM = tmak::BM, BN_CTA = Tile::BN_CTA, BK = tmak::BK;
    constexpr int UMMA_K = tmak::UMMA_K, STAGES = Cfg::STAGES, STAGE_BYTES = Tile::STAGE_BYTES;
    constexpr int A_BYTES = tmak::A_BYTES, B_BYTES = Tile::B_BYTES;
    constexpr int TMA_WARP = tmak::TMA_WARP, MMA_WARP = tmak::MMA_WARP;
    constexpr int NUM_EPI_WARPS = tmak::NUM_EPI_WARPS, TMEM_COLS = tmak::TMEM_COLS;
    constexpr int ACC_STRIDE = tmak::ACC_STRIDE, EPI_CHUNKS = tmak::EPI_CHUNKS;
    static_assert(ACC_STRIDE >= BN && ACC_STRIDE + BN <= TMEM_COLS, "two accumulators in TMEM");
    static_assert(2 * EPI_CHUNKS * 32 >= BN, "two epilogue warps per row quarter cover the tile");
    constexpr uint32_t IDESC = Tile::IDESC | (OPK == 2 ? ((1u << 7) | (1u << 10)) : 0u);
    constexpr int BKE = OPK == 0 ? BK : BK / 2;          // K elements per stage row
    constexpr bool DEQUANT = OPK == 0 || OPK == 3;
    // OPK 3: each accumulator takes a run of RUN_K K (KRUN K blocks) and
    // the epilogue adds the runs in int32. A run's sum is an integer of
    // magnitude at most RUN_K * 127^2 < 2^22 at RUN_K = 256: exact in float32,
    // and fl(v + 1.5 * 2^23) = 2^23 + 2^22 + v exactly, whose bits are
    // 0x4B400000 + v (MAGIC: the conversion is one add). The offsets are
    // summed in wrapping 32-bit arithmetic and removed once per tile.
    // OPK 0-2: one run per tile (KRUN 0).
    constexpr int RUN_K = 512;
    constexpr bool MAGIC = (long long)RUN_K * 127 * 127 < (1LL << 22);
    static_assert(OPK != 3 || (long long)RUN_K * 127 * 127 < (1LL << 24), "a run's float32 sum is exact");
    constexpr int KRUN = OPK == 3 ? RUN_K / BKE : 0;
    static_assert(OPK != 3 || (BN > (EPI_CHUNKS - 1) * 32 && BN + 32 <= ACC_STRIDE && BN <= 2 * EPI_CHUNKS * 32 - 32),
                  "kind 3: the fourth box of the first column half keeps its sum in the 32 TMEM columns after BN");
    constexpr uint16_t PAIR = 3u;                        // both CTAs of the cluster (one pair)
    using Smem = tmak::Smem<STAGES>;

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    constexpr int EPI_STAGE_BYTES = Cfg::EPI_STAGE_BYTES;
    constexpr int EPI_BOX_WARP_BYTES = Cfg::EPI_BOX_WARP_BYTES;
    Smem* sh = reinterpret_cast<Smem*>(smem_raw + (base - raw) + STAGES * STAGE_BYTES + EPI_STAGE_BYTES);
    volatile int* abort = &sh->abort;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t half = cluster_ctarank(), leader = 0;
    const int L = a.L, N = a.N, K = a.K;
    const int num_m = (L + 2 * BM - 1) / (2 * BM);
    const int num_tiles0 = num_m * ((N + BN - 1) / BN);  // problem a's tiles, then problem b's
    const int num_tiles = num_tiles0 + (G2 ? num_m * ((b.N + BN - 1) / BN) : 0);
    const int num_k = K / BKE;
    const int cluster = blockIdx.x / 2, num_clusters = gridDim.x / 2;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_addr(&sh->full[s]), 1);
            mbar_init(smem_addr(&sh->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&sh->tmem_full[b]), 1);
            mbar_init(smem_addr(&sh->tmem_empty[b]), 2 * NUM_EPI_WARPS);
        }
        mbar_init(smem_addr(&sh->drain), 1);
        sh->abort = 0;
        mbar_fence_init();
    }
    if (warp == MMA_WARP) {
        tmem_alloc_pair(smem_addr(&sh->tmem_base), TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync();              // barriers of every CTA initialised, TMEM allocated
    tc_fence_after();
    const uint32_t tmem_base = sh->tmem_base;
    // the prologue above may overlap the previous kernel; no global memory
    // is touched before its results are visible (except the weight tiles
    // of the first stages when the caller vouches for them: see below)
    if (warp != TMA_WARP) grid_dependency_wait();
    grid_launch_dependents();

    // The producer and MMA roles run their loops with the whole warp (warp-
    // uniform control flow and descriptors); one elected lane issues.
    if (warp == TMA_WARP) {
        const uint32_t leader_full0 = mapa_shared(smem_addr(&sh->full[0]), leader);
        // weight tiles of the first stages ahead of the wait for the previous
        // kernel (their stage barriers are fresh, so no empty wait is due)
        int pre = 0;
        if (a.weights_ready && cluster < num_tiles) {
            pre = num_k < STAGES ? num_k : STAGES;
            const bool p1 = G2 && cluster >= num_tiles0;
            const int lt = p1 ? cluster - num_tiles0 : cluster;
            const void* mb = p1 ? (const void*)&tmap_b2 : (const void*)&tmap_b;
            const int n_rows = (lt / num_m) * BN + (int)half * BN_CTA;
            for (int kc = 0; kc < pre; ++kc) {
                if (elect_one()) {
                    if (half == 0) mbar_arrive_expect_tx(smem_addr(&sh->full[kc]), 2 * (A_BYTES + B_BYTES));
                    tma_load_2d_pair(base + kc * STAGE_BYTES + A_BYTES, mb, kc * BKE, n_rows,
                                     leader_full0 + kc * 8);
                }
                __syncwarp();
            }
        }
        grid_dependency_wait();
        int stage = 0;
        uint32_t phase = 0;
        bool ok = true;
        for (int tile = cluster; tile < num_tiles && ok; tile += num_clusters) {
            const bool p1 = G2 && tile >= num_tiles0;
            const int lt = p1 ? tile - num_tiles0 : tile;
            const void* ma = p1 ? (const void*)&tmap_a2 : (const void*)&tmap_a;
            const void* mb = p1 ? (const void*)&tmap_b2 : (const void*)&tmap_b;
            const int m_rows = (lt % num_m) * 2 * BM + (int)half * BM;
            const int n_rows = (lt / num_m) * BN + (int)half * BN_CTA;
            for (int kc = 0; kc < num_k; ++kc) {
                const bool early = tile == cluster && kc < pre;  // weights already in flight
                if (!early && !mbar_wait_bounded_warp(smem_addr(&sh->empty[stage]), phase ^ 1u, abort)) { ok = false; break; }
                const uint32_t st = base + stage * STAGE_BYTES;
                const uint32_t bar = leader_full0 + stage * 8;
                if (elect_one()) {
                    if (half == 0 && !early) mbar_arrive_expect_tx(smem_addr(&sh->full[stage]), 2 * (A_BYTES + B_BYTES));
                    tma_load_2d_pair(st, ma, kc * BKE, m_rows, bar);
                    if (!early) tma_load_2d_pair(st + A_BYTES, mb, kc * BKE, n_rows, bar);
                }
                __syncwarp();
                if (++stage == STAGES) { stage = 0; phase ^= 1u; }
            }
        }
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
        __syncwarp();
    } else if (warp == MMA_WARP) {
        if (half == 0) {
            const uint64_t desc0 = smem_desc_sw128(base);     // start-address field: base >> 4
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int it = 0;          // accumulator runs issued (a tile each, or a K run of a tile: see KRUN)
            for (int tile = cluster; tile < num_tiles && ok; tile += num_clusters) {
                uint32_t d_tmem = 0;
                for (int kc = 0; kc < num_k; ++kc) {
                    const int kk = KRUN > 0 ? kc % KRUN : kc;    // K block within the run
                    if (kk == 0) {
                        const int acc = it & 1;
                        const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
                        if (!mbar_wait_bounded_warp(smem_addr(&sh->tmem_empty[acc]), acc_phase ^ 1u, abort)) { ok = false; break; }
                        tc_fence_after();
                        d_tmem = tmem_base + (uint32_t)(acc * ACC_STRIDE);
                    }
                    if (!mbar_wait_bounded_warp(smem_addr(&sh->full[stage]), phase, abort)) { ok = false; break; }
                    tc_fence_after();
                    // stage offsets stay below 2^18 bytes, so adding them to
                    // the start-address field never carries out of it
                    const uint64_t ad = desc0 + (uint64_t)((stage * STAGE_BYTES) >> 4);
                    const uint64_t bd = ad + (uint64_t)(A_BYTES >> 4);
                    if (elect_one()) {
                        #pragma unroll
                        for (int ks = 0; ks < BK / UMMA_K; ++ks) {
                            const uint64_t adk = ad + (uint64_t)(ks * UMMA_K / 16), bdk = bd + (uint64_t)(ks * UMMA_K / 16);
                            if (OPK == 0) mma_f8f6f4_pair(d_tmem, adk, bdk, IDESC, (kk > 0 || ks > 0) ? 1u : 0u);
                            else mma_f16_pair(d_tmem, adk, bdk, IDESC, (kk > 0 || ks > 0) ? 1u : 0u);
                        }
                        tc_commit_pair_multicast(smem_addr(&sh->empty[stage]), PAIR);
                    }
                    __syncwarp();
                    if (++stage == STAGES) { stage = 0; phase ^= 1u; }
                    if (kc + 1 == num_k || (KRUN > 0 && kk + 1 == KRUN)) {   // the run is complete
                        if (elect_one()) tc_commit_pair_multicast(smem_addr(&sh->tmem_full[it & 1]), PAIR);
                        __syncwarp();
                        ++it;
                    }
                }
            }
            if (elect_one()) tc_commit_pair_multicast(smem_addr(&sh->drain), PAIR);
            __syncwarp();
            if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
        }
        __syncwarp();
    } else if (OPK == 3) {
        // epilogue of the 8-bit kind: the same lanes, columns and boxes as
        // below; every K run of the tile is read from TMEM, converted
        // (exact integers) and added in int32 registers, and its accumulator
        // handed back at once; after the last run the int32 sums are
        // dequantised, fl(fl(fl32(acc) s_a) s_w) (+ bias), and stored.
        constexpr int BOX_BYTES = 32 * 32 * (int)sizeof(TOut);
        constexpr int NBUF = EPI_BOX_WARP_BYTES / BOX_BYTES;
        const uint32_t leader_tmem_empty0 = mapa_shared(smem_addr(&sh->tmem_empty[0]), leader);
        const uint32_t ybox0 = base + STAGES * STAGE_BYTES + warp * EPI_BOX_WARP_BYTES;
        float* epi_sw = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(sh) + sizeof(Smem) +
                                                 (16 - sizeof(Smem) % 16) % 16) + warp * 2 * (EPI_CHUNKS * 32);
        float* epi_b = epi_sw + EPI_CHUNKS * 32;
        const int quarter = warp & 3, chalf = warp >> 2;
        const int runs = KRUN > 0 ? (num_k + KRUN - 1) / KRUN : 1;
        bool ok = true;
        int it = 0;
        int nbox = 0;
        for (int tile = cluster; tile < num_tiles && ok; tile += num_clusters) {
            const bool p1 = G2 && tile >= num_tiles0;
            const int lt = p1 ? tile - num_tiles0 : tile;
            const GemmArgs& P = p1 ? b : a;
            const void* my = p1 ? (const void*)&tmap_y2 : (const void*)&tmap_y;
            const int N = P.N;
            const int m0 = (lt % num_m) * 2 * BM + (int)half * BM;
            const int n0 = (lt / num_m) * BN;
            const int row = m0 + quarter * 32 + lane;
            const bool valid = row < L;
            const float sa = valid ? __ldg(P.s_a + row) : 0.f;
            {
                const int ncol = n0 + chalf * (EPI_CHUNKS * 32) + 4 * lane;
                float4 w = make_float4(0.f, 0.f, 0.f, 0.f), bb = w;
                if (ncol < N) {
                    w = __ldg(reinterpret_cast<const float4*>(P.s_w + ncol));
                    if (P.bias != nullptr) bb = __ldg(reinterpret_cast<const float4*>(P.bias + ncol));
                }
                __syncwarp();
                reinterpret_cast<float4*>(epi_sw)[lane] = w;
                reinterpret_cast<float4*>(epi_b)[lane] = bb;
                __syncwarp();
            }
            // boxes 0-2 of the warp: int32 sums in registers; box 3 (the
            // warps of the first column half): in the free TMEM columns
            // BN .. BN + 31 beside accumulator 0, on the warp's own lanes
            uint32_t sum[EPI_CHUNKS - 1][32];
            const uint32_t corr = MAGIC ? (uint32_t)runs * 0x4B400000u : 0u;   // the runs' offsets
            auto run_bits = [](uint32_t x) -> uint32_t {   // a run's exact integer (plus the offset)
                return MAGIC ? __float_as_uint(__fadd_rn(__uint_as_float(x), 12582912.f))
                             : (uint32_t)__float2int_rn(__uint_as_float(x));
            };
            const uint32_t t_sum = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)BN;
            for (int run = 0; run < runs; ++run, ++it) {
                const int acc = it & 1;
                const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
                if (!mbar_wait_bounded_sleepy(smem_addr(&sh->tmem_full[acc]), acc_phase, abort, 64)) { ok = false; break; }
                tc_fence_after();
                const uint32_t t_row = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * ACC_STRIDE);
                #pragma unroll
                for (int cc = 0; cc < EPI_CHUNKS; ++cc) {
                    const int c = chalf * EPI_CHUNKS + cc;
                    if (c * 32 < BN && n0 + c * 32 < N) {          // warp-uniform
                        if (cc < EPI_CHUNKS - 1) {                 // a register box: one load
                            uint32_t r[32];
                            tmem_ld_32x32b_x32(t_row + c * 32, r);
                            tmem_ld_wait();
                            #pragma unroll
                            for (int t = 0; t < 32; ++t) {
                                const uint32_t v = run_bits(r[t]);
                                uint32_t& sv = sum[cc < EPI_CHUNKS - 1 ? cc : 0][t];
                                sv = run == 0 ? v : sv + v;
                            }
                        } else {                                   // the TMEM box: 8 columns at a time
                            #pragma unroll
                            for (int h = 0; h < 4; ++h) {
                                uint32_t r[8], s8[8];
                                tmem_ld_32x32b_x8(t_row + c * 32 + 8 * h, r);
                                if (run > 0) tmem_ld_32x32b_x8(t_sum + 8 * h, s8);
                                tmem_ld_wait();
                                #pragma unroll
                                for (int t = 0; t < 8; ++t)
                                    s8[t] = run_bits(r[t]) + (run > 0 ? s8[t] : 0u);
                                tmem_st_32x32b_x8(t_sum + 8 * h, s8);
                            }
                            tmem_st_wait();                        // before the next run reads them back
                        }
                    }
                }
                // the run's TMEM reads are complete (tcgen05.wait::ld) and ordered
                // by the fence: a relaxed arrive hands the accumulator back
                // without a memory barrier
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster_relaxed(leader_tmem_empty0 + acc * 8);
            }
            if (!ok) break;
            // dequantise one box of sums and store it
            auto emit = [&](const uint32_t (&qs)[32], int cc, int nc) {
                auto q = [&](int t) { return (int)(qs[t] - corr); };
                if (P.acc_dbg != nullptr && valid) {
                    int4* d4 = reinterpret_cast<int4*>(P.acc_dbg + (size_t)row * N + nc);
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) d4[u] = make_int4(q(4 * u), q(4 * u + 1), q(4 * u + 2), q(4 * u + 3));
                }
                float y[32];
                const float4* sw4 = reinterpret_cast<const float4*>(epi_sw + cc * 32);
                const float4* b4 = reinterpret_cast<const float4*>(epi_b + cc * 32);
                #pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const float4 sw = sw4[u];
                    y[4 * u] = __fmul_rn(__fmul_rn(__int2float_rn(q(4 * u)), sa), sw.x);
                    y[4 * u + 1] = __fmul_rn(__fmul_rn(__int2float_rn(q(4 * u + 1)), sa), sw.y);
                    y[4 * u + 2] = __fmul_rn(__fmul_rn(__int2float_rn(q(4 * u + 2)), sa), sw.z);
                    y[4 * u + 3] = __fmul_rn(__fmul_rn(__int2float_rn(q(4 * u + 3)), sa), sw.w);
                }
                if (P.bias != nullptr) {
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 bq = b4[u];
                        y[4 * u] = __fadd_rn(y[4 * u], bq.x);
                        y[4 * u + 1] = __fadd_rn(y[4 * u + 1], bq.y);
                        y[4 * u + 2] = __fadd_rn(y[4 * u + 2], bq.z);
                        y[4 * u + 3] = __fadd_rn(y[4 * u + 3], bq.w);
                    }
                }
                // the buffer's previous store has read it
                const uint32_t box = ybox0 + (uint32_t)((nbox % NBUF) * BOX_BYTES);
                if (nbox >= NBUF) {
                    if (lane == 0) {
                        if (NBUF == 2) bulk_wait_read1(); else bulk_wait_read0();
                    }
                    __syncwarp();
                }
                Out<TOut>::stage32(box, lane, y);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(my, nc, m0 + quarter * 32, box);
                    bulk_commit();
                }
                ++nbox;
            };
            #pragma unroll
            for (int cc = 0; cc < EPI_CHUNKS - 1; ++cc) {
                const int c = chalf * EPI_CHUNKS + cc;
                if (c * 32 < BN && n0 + c * 32 < N) emit(sum[cc], cc, n0 + c * 32);
            }
            {
                constexpr int cc = EPI_CHUNKS - 1;
                const int c = chalf * EPI_CHUNKS + cc;
                if (c * 32 < BN && n0 + c * 32 < N) {
                    uint32_t q[32];
                    #pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        uint32_t s8[8];
                        tmem_ld_32x32b_x8(t_sum + 8 * h, s8);
                        tmem_ld_wait();
                        #pragma unroll
                        for (int t = 0; t < 8; ++t) q[8 * h + t] = s8[t];
                    }
                    emit(q, cc, n0 + c * 32);
                }
            }
        }
        if (lane == 0) bulk_wait0();     // this warp's stores are complete
        __syncwarp();
        if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
    } else {
        // epilogue: warp w reads TMEM lanes 32 (w % 4) .. + 31, columns
        // (w / 4) * 128 .. + 127 below BN, in 32 x 32 boxes; scales and biases are
        // staged before the accumulator wait. Each box is dequantised into
        // the warp's swizzled staging buffer and written by one TMA store
        // (rows past L and columns past N are clipped by the tensor map).
        constexpr int BOX_BYTES = 32 * 32 * (int)sizeof(TOut);
        constexpr int NBUF = EPI_BOX_WARP_BYTES / BOX_BYTES;
        const uint32_t leader_tmem_empty0 = mapa_shared(smem_addr(&sh->tmem_empty[0]), leader);
        const uint32_t ybox0 = base + STAGES * STAGE_BYTES + warp * EPI_BOX_WARP_BYTES;
        float* epi_sw = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(sh) + sizeof(Smem) +
                                                 (16 - sizeof(Smem) % 16) % 16) + warp * 2 * (EPI_CHUNKS * 32);
        float* epi_b = epi_sw + EPI_CHUNKS * 32;
        const int quarter = warp & 3, chalf = warp >> 2;
        bool ok = true;
        int it = 0;
        int nbox = 0;
        for (int tile = cluster; tile < num_tiles; tile += num_clusters, ++it) {
            const bool p1 = G2 && tile >= num_tiles0;
            const int lt = p1 ? tile - num_tiles0 : tile;
            const GemmArgs& P = p1 ? b : a;
            const void* my = p1 ? (const void*)&tmap_y2 : (const void*)&tmap_y;
            const int N = P.N;
            const int m0 = (lt % num_m) * 2 * BM + (int)half * BM;
            const int n0 = (lt / num_m) * BN;
            const int acc = it & 1;
            const uint32_t acc_phase = (uint32_t)(it >> 1) & 1u;
            const int row = m0 + quarter * 32 + lane;
            const bool valid = row < L;
            const float sa = (DEQUANT && valid) ? __ldg(P.s_a + row) : 0.f;
            if (DEQUANT) {
                const int ncol = n0 + chalf * (EPI_CHUNKS * 32) + 4 * lane;
                float4 w = make_float4(0.f, 0.f, 0.f, 0.f), bb = w;
                if (ncol < N) {
                    w = __ldg(reinterpret_cast<const float4*>(P.s_w + ncol));
                    if (P.bias != nullptr) bb = __ldg(reinterpret_cast<const float4*>(P.bias + ncol));
                }
                __syncwarp();
                reinterpret_cast<float4*>(epi_sw)[lane] = w;
                reinterpret_cast<float4*>(epi_b)[lane] = bb;
                __syncwarp();
            }
            // a whole tile of MMAs away: poll gently, the MMA warp shares the scheduler
            if (!mbar_wait_bounded_sleepy(smem_addr(&sh->tmem_full[acc]), acc_phase, abort, 256)) { ok = false; break; }
            tc_fence_after();
            const uint32_t t_row = tmem_base + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(acc * ACC_STRIDE);
            #pragma unroll 1
            for (int cc = 0; cc < EPI_CHUNKS; ++cc) {
                const int c = chalf * EPI_CHUNKS + cc;
                const int nc = n0 + c * 32;
                if (c * 32 >= BN || nc >= N) break;
                uint32_t r[32];
                tmem_ld_32x32b_x32(t_row + c * 32, r);
                tmem_ld_wait();
                float y[32];
                const float4* sw4 = reinterpret_cast<const float4*>(epi_sw + cc * 32);
                const float4* b4 = reinterpret_cast<const float4*>(epi_b + cc * 32);
                #pragma unroll
                for (int u = 0; u < 8 && !DEQUANT; ++u) {
                    y[4 * u] = __uint_as_float(r[4 * u]);
                    y[4 * u + 1] = __uint_as_float(r[4 * u + 1]);
                    y[4 * u + 2] = __uint_as_float(r[4 * u + 2]);
                    y[4 * u + 3] = __uint_as_float(r[4 * u + 3]);
                }
                if (DEQUANT && P.bias == nullptr) {
                    // fl(fl(acc s_a) s_w) on packed pairs (two multiplies: nothing to contract)
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 sw = sw4[u];
                        mul2_rn(__uint_as_float(r[4 * u]), __uint_as_float(r[4 * u + 1]), sa, sw.x, sw.y,
                                y[4 * u], y[4 * u + 1]);
                        mul2_rn(__uint_as_float(r[4 * u + 2]), __uint_as_float(r[4 * u + 3]), sa, sw.z, sw.w,
                                y[4 * u + 2], y[4 * u + 3]);
                    }
                } else if (DEQUANT) {
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 sw = sw4[u];
                        y[4 * u] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u]), sa), sw.x);
                        y[4 * u + 1] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 1]), sa), sw.y);
                        y[4 * u + 2] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 2]), sa), sw.z);
                        y[4 * u + 3] = __fmul_rn(__fmul_rn(__uint_as_float(r[4 * u + 3]), sa), sw.w);
                    }
                }
                if (DEQUANT && P.bias != nullptr) {
                    #pragma unroll
                    for (int u = 0; u < 8; ++u) {
                        const float4 bq = b4[u];
                        y[4 * u] = __fadd_rn(y[4 * u], bq.x);
                        y[4 * u + 1] = __fadd_rn(y[4 * u + 1], bq.y);
                        y[4 * u + 2] = __fadd_rn(y[4 * u + 2], bq.z);
                        y[4 * u + 3] = __fadd_rn(y[4 * u + 3], bq.w);
                    }
                }
                // the buffer's previous store has read it
                const uint32_t box = ybox0 + (uint32_t)((nbox % NBUF) * BOX_BYTES);
                if (nbox >= NBUF) {
                    if (lane == 0) {
                        if (NBUF == 2) bulk_wait_read1(); else bulk_wait_read0();
                    }
                    __syncwarp();
                }
                if (SWIGLU) {
                    float h[16];
                    #pragma unroll
                    for (int t = 0; t < 16; ++t) h[t] = y[t] / (1.f + expf(-y[t])) * y[16 + t];
                    Out<TOut>::stage16(box, lane, h);
                } else {
                    Out<TOut>::stage32(box, lane, y);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(my, SWIGLU ? nc / 2 : nc, m0 + quarter * 32, box);
                    bulk_commit();
                }
                ++nbox;
                if (P.acc_dbg != nullptr && valid) {
                    int4* d4 = reinterpret_cast<int4*>(P.acc_dbg + (size_t)row * N + nc);
                    #pragma unroll
                    for (int u = 0; u < 8; ++u)
                        d4[u] = make_int4(__float2int_rn(__uint_as_float(r[4 * u])),
                                          __float2int_rn(__uint_as_float(r[4 * u + 1])),
                                          __float2int_rn(__uint_as_float(r[4 * u + 2])),
                                          __float2int_rn(__uint_as_float(r[4 * u + 3])));
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(leader_tmem_empty0 + acc * 8);
        }
        if (lane == 0) bulk_wait0();     // this warp's stores are complete
        __syncwarp();
        if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_GEMM); }
    }

    // every MMA the pair's leader issued has completed before TMEM is released
    if (warp == MMA_WARP && lane == 0) {
        volatile int never = 0;
        if (!mbar_wait_bounded(smem_addr(&sh->drain), 0, &never)) atomicOr(a.status, STATUS_TIMEOUT_GEMM);
    }
    __syncwarp();
    tc_fence_before();
    cluster_sync();              // no CTA leaves while another may still signal it
    tc_fence_after();
    if (warp == MMA_WARP) tmem_dealloc_pair(tmem_base, TMEM_COLS);
}

// Clusters (CTA pairs) of this instantiation resident at once on the current
// device (queried once per device; also sets the kernel's shared-memory
// limit).
template <typename TOut, int OPK, int BN, bool SW, bool G2 = false>
cudaError_t tma_max_clusters(int* clusters) {
    constexpr size_t SMEM_BYTES = tmak::Cfg<sizeof(TOut), BN>::SMEM_BYTES;
    static DeviceCache<int> cache;
    return cache.get(clusters, [](int, int* v) {
        auto kernel = w4a4_gemm_tma_pair_kernel<TOut, OPK, BN, SW, G2>;
        cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 2;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.blockDim = dim3(tmak::THREADS);
        cfg.dynamicSmemBytes = SMEM_BYTES;
        cfg.attrs = attr;
        cfg.numAttrs = 1;                // the occupancy query takes the cluster shape only
        cfg.gridDim = dim3(2 * 32);
        int n = 0;
        e = cudaOccupancyMaxActiveClusters(&n, kernel, &cfg);
        if (e != cudaSuccess) return e;
        *v = n > 0 ? n : 1;
        return cudaSuccess;
    });
}

// b: the second problem of a grouped launch (G2), else unused.
template <typename TOut, int OPK, int BN, bool SW, bool G2 = false>
cudaError_t launch_tma_cl(const GemmArgs& a, cudaStream_t stream, int clusters, const GemmArgs* b = nullptr) {
    constexpr int BM = tmak::BM, BN_CTA = tmak::Tile<BN>::BN_CTA, BK = tmak::BK;
    constexpr int ELEM = OPK == 0 ? 1 : 2;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1] = pdl_attribute();
    cfg.blockDim = dim3(tmak::THREADS);
    cfg.dynamicSmemBytes = tmak::Cfg<sizeof(TOut), BN>::SMEM_BYTES;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    CUtensorMap ta, tb, ty, ta2, tb2, ty2;
    const CUtensorMapDataType opt = OPK == 0 ? CU_TENSOR_MAP_DATA_TYPE_UINT8 : CU_TENSOR_MAP_DATA_TYPE_UINT16;
    auto maps = [&](const GemmArgs& p, CUtensorMap* xa, CUtensorMap* xb, CUtensorMap* xy) {
        return encode_operand_tmap(xa, p.Xe, opt, ELEM, (uint64_t)p.L, (uint64_t)p.K, BM, BK / ELEM) &&
               encode_operand_tmap(xb, p.We, opt, ELEM, (uint64_t)p.N, (uint64_t)p.K, BN_CTA, BK / ELEM) &&
               (SW ? encode_out_tmap(xy, p.Y, Out<TOut>::TMAP_TYPE, sizeof(TOut), (uint64_t)p.L, (uint64_t)p.N / 2,
                                     CU_TENSOR_MAP_SWIZZLE_32B, 16)
                   : encode_out_tmap(xy, p.Y, Out<TOut>::TMAP_TYPE, sizeof(TOut), (uint64_t)p.L, (uint64_t)p.N,
                                     Out<TOut>::TMAP_SWIZZLE));
    };
    if (!maps(a, &ta, &tb, &ty)) return cudaErrorInvalidValue;
    int num_tiles = tma_tiles(a.L, a.N, BN);
    if (G2) {
        if (b == nullptr || !maps(*b, &ta2, &tb2, &ty2)) return cudaErrorInvalidValue;
        num_tiles += tma_tiles(b->L, b->N, BN);
    } else {
        ta2 = ta;
        tb2 = tb;
        ty2 = ty;
    }
    if (num_tiles < clusters) clusters = num_tiles;
    cfg.gridDim = dim3(2 * clusters);
    return cudaLaunchKernelEx(&cfg, w4a4_gemm_tma_pair_kernel<TOut, OPK, BN, SW, G2>, a, ta, tb, ty,
                              G2 ? *b : a, ta2, tb2, ty2);
}

// Tile shape per problem. A stage's steady state is bound by shared memory:
// per CTA the MMAs read the 16 KB activation tile and the CTA's weight half
// twice (for itself and for its pair peer) while TMA writes both, i.e.
// 256 + 1.5 BN cycles at 128 bytes per clock against 2 BN cycles of tensor
// work. A launch takes ceil(tiles / pairs) rounds of a tile's stages.
// Candidates: 256- and 224-channel pair tiles (224 fills the 76 pairs of
// the LLaDA projections better); the cheaper estimate wins, ties keep 256.
template <typename TOut, int OPK, bool SW>
cudaError_t launch_tma_shape(const GemmArgs& a, cudaStream_t stream) {
    if constexpr (OPK == 3) {            // 224-wide tiles only: their free TMEM columns hold a box of sums
        int c224 = 0;
        const cudaError_t e = tma_max_clusters<TOut, OPK, 224, SW>(&c224);
        if (e != cudaSuccess) return e;
        if (g_pair_limit > 0 && c224 > g_pair_limit) c224 = g_pair_limit;
        g_last_tile = 224 * 10 + 2;
        return launch_tma_cl<TOut, OPK, 224, SW>(a, stream, c224);
    } else {
        int c256 = 0, c224 = 0;
        cudaError_t e = tma_max_clusters<TOut, OPK, 256, SW>(&c256);
        if (e != cudaSuccess) return e;
        if ((e = tma_max_clusters<TOut, OPK, 224, SW>(&c224)) != cudaSuccess) return e;
        if (g_pair_limit > 0) {
            if (c256 > g_pair_limit) c256 = g_pair_limit;
            if (c224 > g_pair_limit) c224 = g_pair_limit;
        }
        const long long t256 = tma_round_cost(a.L, a.N, 256, c256);
        const long long t224 = tma_round_cost(a.L, a.N, 224, c224);
        if (t224 < t256) {
            g_last_tile = 224 * 10 + 2;
            return launch_tma_cl<TOut, OPK, 224, SW>(a, stream, c224);
        }
        g_last_tile = 256 * 10 + 2;
        return launch_tma_cl<TOut, OPK, 256, SW>(a, stream, c256);
    }
}

// Two independent problems (same L, K and output type, E4M3 operands, no
// SwiGLU) in one persistent launch: the tile width is chosen for the two
// together.
template <typename TOut>
cudaError_t launch_tma_grouped(const GemmArgs& a, const GemmArgs& b, cudaStream_t stream) {
    int c256 = 0, c224 = 0;
    cudaError_t e = tma_max_clusters<TOut, 0, 256, false, true>(&c256);
    if (e != cudaSuccess) return e;
    if ((e = tma_max_clusters<TOut, 0, 224, false, true>(&c224)) != cudaSuccess) return e;
    if (g_pair_limit > 0) {
        if (c256 > g_pair_limit) c256 = g_pair_limit;
        if (c224 > g_pair_limit) c224 = g_pair_limit;
    }
    auto cost = [&](int bn, int cl) {
        const long long tiles = tma_tiles(a.L, a.N, bn) + tma_tiles(b.L, b.N, bn);
        const long long used = cl < 1 ? 1 : cl;
        const long long stage2 = 4LL * bn > 512LL + 3LL * bn ? 4LL * bn : 512LL + 3LL * bn;
        return (tiles + used - 1) / used * stage2;
    };
    if (cost(224, c224) < cost(256, c256)) {
        g_last_tile = 224 * 10 + 2;
        return launch_tma_cl<TOut, 0, 224, false, true>(a, stream, c224, &b);
    }
    g_last_tile = 256 * 10 + 2;
    return launch_tma_cl<TOut, 0, 256, false, true>(a, stream, c256, &b);
}

template <typename TOut, int OPK = 0>
cudaError_t launch_tma_typed(const GemmArgs& a, cudaStream_t stream) {
    if constexpr (OPK == 0 && sizeof(TOut) == 2) {
        if (a.swiglu) return launch_tma_shape<TOut, OPK, true>(a, stream);
    }
    if (a.swiglu) return cudaErrorInvalidValue;
    return launch_tma_shape<TOut, OPK, false>(a, stream);
}

// Packed int4 -> E4M3: each thread turns 16 packed bytes into 32 E4M3 bytes.
__global__ void __launch_bounds__(256) unpack_e4m3_kernel(const uint4* __restrict__ packed,
                                                          uint4* __restrict__ out, size_t n16) {
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += (size_t)gridDim.x * blockDim.x) {
        const uint4 w = ld_global_nc_v4(packed + i);
        uint32_t o[8];
        int4x8_to_e4m3x8(w.x, o[0], o[1]);
        int4x8_to_e4m3x8(w.y, o[2], o[3]);
        int4x8_to_e4m3x8(w.z, o[4], o[5]);
        int4x8_to_e4m3x8(w.w, o[6], o[7]);
        out[2 * i] = make_uint4(o[0], o[1], o[2], o[3]);
        out[2 * i + 1] = make_uint4(o[4], o[5], o[6], o[7]);
    }
}

// The CTA-pair GEMM that converts packed weights: one pair per cluster, as
// many clusters as are resident at once (queried once per device).
template <typename TOut>
cudaError_t launch_pair_typed(const GemmArgs& a, cudaStream_t stream) {
    constexpr int BM = pairk::BM, BN = pairk::BN, BN_CTA = pairk::BN_CTA, BK = pairk::BK;
    constexpr int THREADS = pairk::THREADS;
    constexpr size_t SMEM_BYTES = pairk::SMEM_BYTES;
    CUtensorMap ta, tb;
    if (!encode_u8_tmap(&ta, a.Xe, (uint64_t)a.L, (uint64_t)a.K, BM, BK, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_u8_tmap(&tb, a.Wq, (uint64_t)a.N, (uint64_t)a.K / 2, BN_CTA, BK / 2, CU_TENSOR_MAP_SWIZZLE_NONE))
        return cudaErrorInvalidValue;
    auto kernel = w4a4_gemm_pair_kernel<TOut>;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = SMEM_BYTES;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    static DeviceCache<int> cache;
    int clusters = 0;
    cudaError_t e = cache.get(&clusters, [&](int, int* v) {
        cudaError_t r = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)SMEM_BYTES);
        if (r != cudaSuccess) return r;
        cudaLaunchConfig_t q = cfg;
        q.gridDim = dim3(2 * 64);
        int n = 0;
        r = cudaOccupancyMaxActiveClusters(&n, kernel, &q);
        if (r != cudaSuccess) return r;
        *v = n > 0 ? n : 1;
        return cudaSuccess;
    });
    if (e != cudaSuccess) return e;
    const int num_tiles = ((a.L + 2 * BM - 1) / (2 * BM)) * ((a.N + BN - 1) / BN);
    if (num_tiles < clusters) clusters = num_tiles;
    cfg.gridDim = dim3(2 * clusters);
    return cudaLaunchKernelEx(&cfg, kernel, a, ta, tb);
}

template <typename TOut>
cudaError_t launch_typed(const GemmArgs& a, cudaStream_t stream) {
    static DeviceCache<int> attr;
    int done = 0;
    cudaError_t e = attr.get(&done, [](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(w4a4_gemm_kernel<TOut>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)SMEM_BYTES);
    });
    if (e != cudaSuccess) return e;
    const int num_tiles = ((a.L + BM - 1) / BM) * ((a.N + BN - 1) / BN);
    const int grid = num_tiles < num_sms() ? num_tiles : num_sms();
    w4a4_gemm_kernel<TOut><<<grid, THREADS, SMEM_BYTES, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_unpack_e4m3(const uint8_t* packed, uint8_t* e4m3, size_t rows, int K, cudaStream_t stream) {
    const size_t n16 = rows * (size_t)K / 32;
    if (n16 == 0) return cudaSuccess;
    size_t blocks = (n16 + 255) / 256;
    const size_t cap = (size_t)num_sms() * 8;
    if (blocks > cap) blocks = cap;
    unpack_e4m3_kernel<<<(unsigned)blocks, 256, 0, stream>>>(reinterpret_cast<const uint4*>(packed),
                                                               reinterpret_cast<uint4*>(e4m3), n16);
    return cudaGetLastError();
}

int last_gemm_tile() { return g_last_tile; }

cudaError_t launch_fp16_gemm(const GemmArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    switch (a.y_dtype) {
        case STARQ_F16: return launch_tma_typed<__half, 1>(a, stream);
        case STARQ_BF16: return launch_tma_typed<__nv_bfloat16, 2>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_w8a8_gemm(const GemmArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    if (a.Xe == nullptr || a.We == nullptr || a.swiglu) return cudaErrorInvalidValue;
    switch (a.y_dtype) {
        case STARQ_F16: return launch_tma_typed<__half, 3>(a, stream);
        case STARQ_BF16: return launch_tma_typed<__nv_bfloat16, 3>(a, stream);
        case STARQ_F32: return launch_tma_typed<float, 3>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

int set_gemm_pair_limit(int pairs) {
    const int prev = g_pair_limit;
    g_pair_limit = pairs;
    return prev;
}

cudaError_t launch_w4a4_gemm_grouped(const GemmArgs& a, const GemmArgs& b, cudaStream_t stream) {
    if (a.L != b.L || a.K != b.K || a.y_dtype != b.y_dtype || !a.Xe || !a.We || !b.Xe || !b.We || a.swiglu ||
        b.swiglu)
        return cudaErrorInvalidValue;
    if (a.L == 0) return cudaSuccess;
    switch (a.y_dtype) {
        case STARQ_F16: return launch_tma_grouped<__half>(a, b, stream);
        case STARQ_BF16: return launch_tma_grouped<__nv_bfloat16>(a, b, stream);
        case STARQ_F32: return launch_tma_grouped<float>(a, b, stream);
        default: return cudaErrorInvalidValue;
    }
}

cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    if (a.Xe != nullptr && a.We != nullptr) {
        switch (a.y_dtype) {
            case STARQ_F16: return launch_tma_typed<__half>(a, stream);
            case STARQ_BF16: return launch_tma_typed<__nv_bfloat16>(a, stream);
            case STARQ_F32: return launch_tma_typed<float>(a, stream);
            default: return cudaErrorInvalidValue;
        }
    }
    if (a.Xe != nullptr) {
        switch (a.y_dtype) {
            case STARQ_F16: return launch_pair_typed<__half>(a, stream);
            case STARQ_BF16: return launch_pair_typed<__nv_bfloat16>(a, stream);
            case STARQ_F32: return launch_pair_typed<float>(a, stream);
            default: return cudaErrorInvalidValue;
        }
    }
    switch (a.y_dtype) {
        case STARQ_F16: return launch_typed<__half>(a, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_typed<float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
