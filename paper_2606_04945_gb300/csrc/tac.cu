// TAC: block-wise affine compensation (Sec. 3.3 Eq. 17, App. C row-major form)
//
//   out[i][b*g + r] = sum_j M[b][r][j] * Z[i][b*g + j] + d[b][r]
//
// 16-bit inputs with g = 64 or 128 run on the tensor cores (tac_tc_kernel
// below). Otherwise, the CUDA-core kernel: grid (token tiles, blocks b). A
// CTA stages M_b transposed (Mt[j][r]) and a tile of TM tokens of block b in shared memory, then each thread computes
// RT = 4 tokens x RC = 8 channels with float32 FMAs, reading four j at a time
// (float4) from both tiles. TM = 8192 / g tokens, so the token tile is
// 32 KB (fp32) and the CTA holds g*g*4 + 32 KB of shared memory.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <type_traits>

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
    static DeviceCache<int> attr;
    int done = 0;
    const cudaError_t e = attr.get(&done, [](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(tac_kernel<G, TIn, TOut>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    });
    if (e != cudaSuccess) return e;
    dim3 grid((a.L + TM - 1) / TM, a.C / G);
    tac_kernel<G, TIn, TOut><<<grid, TPB, smem, stream>>>(a);
    return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Tensor-core TAC for g in {64, 128} with 16-bit inputs.
//
// Block b is a GEMM out_b[L x g] = Z_b[L x g] M_b^T[g x g] + d_b with the
// contraction over the block's g channels. Z is exact in its 16-bit type; M
// is split into M_hi = 16bit(M) and M_lo = 16bit(M - M_hi) of the same type
// (the MMA takes equal A and B types), and the tensor core accumulates
// Z M_hi^T + Z M_lo^T in float32 in TMEM; the residual of the split is
// below 2^-22 |M| for fp16 and 2^-16 |M| for bf16. A CTA owns one block b and
// a run of 128-token tiles: it converts M_b once into 128-byte-swizzled
// K-major shared tiles, streams the Z tiles by TMA (two buffers), runs
// 2 g/16 MMAs (M = 128, N = g, K = 16) per tile, and its four warps add d_b
// to the rows read back from TMEM. float32 outputs are staged as
// 128-byte-swizzled 32 x 32 boxes and written by TMA stores; 16-bit outputs
// by 16-byte row stores.
// ---------------------------------------------------------------------------
constexpr int TC_TM = 128;              // tokens per tile (MMA M)
constexpr int TC_THREADS = 256;

template <int G>
struct TacTc {
    static_assert(G * G / 8 % TC_THREADS == 0, "whole load rounds per thread");
    static constexpr int ATOMS = G / 64;                      // 64 16-bit elements = 128 B per atom row
    static constexpr int Z_BYTES = TC_TM * G * 2;             // the Z tile
    static constexpr int M_BYTES = G * G * 2;                 // one of M_hi / M_lo
    static constexpr int OUT_BYTES = (TC_THREADS / 32) * 32 * 32 * 4;   // one float 32 x 32 box per warp
    // the Z tile's space holds the output boxes once the MMAs have read it
    static constexpr int REGION = Z_BYTES > OUT_BYTES ? Z_BYTES : OUT_BYTES;
    static constexpr size_t SMEM = (size_t)REGION + 2 * (size_t)M_BYTES + 1024;
    static constexpr int TMEM_COLS = G;
};

template <typename T> struct Split16;
template <> struct Split16<__half> {
    static __device__ __forceinline__ void split(float m, uint16_t& hi, uint16_t& lo) {
        const __half h = __float2half_rn(m);
        const __half l = __float2half_rn(m - __half2float(h));
        hi = __half_as_ushort(h);
        lo = __half_as_ushort(l);
    }
    static constexpr uint32_t KIND = 0;
};
template <> struct Split16<__nv_bfloat16> {
    static __device__ __forceinline__ void split(float m, uint16_t& hi, uint16_t& lo) {
        const __nv_bfloat16 h = __float2bfloat16_rn(m);
        const __nv_bfloat16 l = __float2bfloat16_rn(m - __bfloat162float(h));
        hi = __bfloat16_as_ushort(h);
        lo = __bfloat16_as_ushort(l);
    }
    static constexpr uint32_t KIND = 1;
};

template <typename TOut> struct TacStore;
// float32 output: 32 x 32 boxes staged 128-byte-swizzled and written by TMA
template <> struct TacStore<float> {
    static constexpr bool TMA = true;
};
// 16-bit output: 32 x 32 boxes of 64-byte rows with the 64-byte swizzle
template <> struct TacStore<__half> { static constexpr bool TMA = true; };
template <> struct TacStore<__nv_bfloat16> { static constexpr bool TMA = true; };

// M_b (float32 [g][g]) -> its two 16-bit halves, K-major (row r = output
// channel, 8 inputs per 16-byte chunk, 128-byte swizzle) at shared
// addresses sMh / sMl; every load of the thread is issued before the first
// convert.
template <int G, typename TIn>
__device__ __forceinline__ void tac_split_block(const float* Mb, uint32_t sMh, uint32_t sMl) {
    constexpr int NIT = G * G / 8 / TC_THREADS;
    float4 w0[NIT], w1[NIT];
    #pragma unroll
    for (int it = 0; it < NIT; ++it) {
        const int idx = threadIdx.x + it * TC_THREADS;
        const int r = idx / (G / 8), jc = idx % (G / 8);
        w0[it] = __ldg(reinterpret_cast<const float4*>(Mb + (size_t)r * G + 8 * jc));
        w1[it] = __ldg(reinterpret_cast<const float4*>(Mb + (size_t)r * G + 8 * jc + 4));
    }
    #pragma unroll
    for (int it = 0; it < NIT; ++it) {
        const int idx = threadIdx.x + it * TC_THREADS;
        const int r = idx / (G / 8), jc = idx % (G / 8);      // inputs j = 8 jc .. 8 jc + 7
        const float mv[8] = {w0[it].x, w0[it].y, w0[it].z, w0[it].w, w1[it].x, w1[it].y, w1[it].z, w1[it].w};
        uint32_t hi[4], lo[4];
        #pragma unroll
        for (int e = 0; e < 4; ++e) {
            uint16_t h0, l0, h1, l1;
            Split16<TIn>::split(mv[2 * e], h0, l0);
            Split16<TIn>::split(mv[2 * e + 1], h1, l1);
            hi[e] = (uint32_t)h0 | ((uint32_t)h1 << 16);
            lo[e] = (uint32_t)l0 | ((uint32_t)l1 << 16);
        }
        const uint32_t off = (jc / 8) * (G * 128) + sw128_offset(r, jc % 8);
        st_shared_v4(sMh + off, hi[0], hi[1], hi[2], hi[3]);
        st_shared_v4(sMl + off, lo[0], lo[1], lo[2], lo[3]);
    }
}

// The same halves written once to global memory, byte for byte the shared
// image tac_tc_kernel builds (hi then lo per block), for a bulk copy.
template <int G, typename TIn>
__global__ void __launch_bounds__(256)
tac_prepare_kernel(const float* __restrict__ M, uint8_t* __restrict__ Mp) {
    constexpr int M_BYTES = G * G * 2;
    const int b = blockIdx.x;
    const float* Mb = M + (size_t)b * G * G;
    uint8_t* hi = Mp + (size_t)b * 2 * M_BYTES;
    uint8_t* lo = hi + M_BYTES;
    for (int idx = threadIdx.x; idx < G * G / 8; idx += blockDim.x) {
        const int r = idx / (G / 8), jc = idx % (G / 8);
        const float4 w0 = __ldg(reinterpret_cast<const float4*>(Mb + (size_t)r * G + 8 * jc));
        const float4 w1 = __ldg(reinterpret_cast<const float4*>(Mb + (size_t)r * G + 8 * jc + 4));
        const float mv[8] = {w0.x, w0.y, w0.z, w0.w, w1.x, w1.y, w1.z, w1.w};
        uint32_t h[4], l[4];
        #pragma unroll
        for (int e = 0; e < 4; ++e) {
            uint16_t h0, l0, h1, l1;
            Split16<TIn>::split(mv[2 * e], h0, l0);
            Split16<TIn>::split(mv[2 * e + 1], h1, l1);
            h[e] = (uint32_t)h0 | ((uint32_t)h1 << 16);
            l[e] = (uint32_t)l0 | ((uint32_t)l1 << 16);
        }
        const uint32_t off = (jc / 8) * (G * 128) + sw128_offset(r, jc % 8);
        *reinterpret_cast<uint4*>(hi + off) = make_uint4(h[0], h[1], h[2], h[3]);
        *reinterpret_cast<uint4*>(lo + off) = make_uint4(l[0], l[1], l[2], l[3]);
    }
}

// Tensor-core TAC: one CTA per (block b, tile of 128 tokens), 8 warps.
//   * the tile Z[rows][b g .. b g + g) arrives by TMA (128-byte swizzle);
//   * meanwhile all threads read M_b (float32) with coalesced 32-byte loads
//     and write its two 16-bit halves hi = rn(M), lo = rn(M - hi) (the
//     input's type) into the K-major swizzled operand layout -- or, with a
//     prepared M (tac_prepare), one bulk copy brings both halves;
//   * one thread issues g/16 pairs of kind::f16 MMAs (Z hi^T and Z lo^T,
//     float32 accumulation in TMEM: relative error about 2^-22);
//   * each warp reads 32 tokens x g/2 channels of the accumulator, adds d,
//     and stores: float output through 32 x 32 boxes (staged in the Z
//     tile's space, which the MMAs no longer need) and TMA stores, 16-bit
//     output with direct row stores.
// About 97 KB of shared memory at g = 128, so two CTAs share an SM.
template <int G, typename TIn, typename TOut>
__global__ void __launch_bounds__(TC_THREADS)
tac_tc_kernel(TacArgs a, const __grid_constant__ CUtensorMap tmap_z, const __grid_constant__ CUtensorMap tmap_out,
              unsigned* status) {
    using P = TacTc<G>;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t zfull, mfull, mdone;
    __shared__ __align__(16) float dsm[G];
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    const uint32_t sZ = base;                                  // Z tile, then output boxes
    const uint32_t sMh = base + P::REGION, sMl = sMh + P::M_BYTES;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int b = blockIdx.x;
    const int row0 = blockIdx.y * TC_TM;
    volatile int* abort = &abort_flag;

    if (threadIdx.x == 0) {
        mbar_init(smem_addr(&zfull), 1);
        mbar_init(smem_addr(&mfull), 1);
        mbar_init(smem_addr(&mdone), 1);
        abort_flag = 0;
        mbar_fence_init();
    }
    const bool prepared = a.Mp != nullptr;
    if (warp == 0) {
        tmem_alloc(smem_addr(&tmem_slot), P::TMEM_COLS);
        tmem_relinquish();
    }
    __syncthreads();
    // both 16-bit halves of M_b (prepared) on their own barrier, and d_b in
    // shared memory; ahead of the wait for the previous kernel when the
    // caller vouches that it does not write them
    auto fetch_params = [&]() {
        if (threadIdx.x == 0 && prepared) {
            mbar_arrive_expect_tx(smem_addr(&mfull), 2 * P::M_BYTES);
            bulk_load(sMh, static_cast<const uint8_t*>(a.Mp) + (size_t)b * 2 * P::M_BYTES, 2 * P::M_BYTES,
                      smem_addr(&mfull));
        }
        if (!prepared) tac_split_block<G, TIn>(a.M + (size_t)b * G * G, sMh, sMl);
        if (threadIdx.x < G / 4)
            reinterpret_cast<float4*>(dsm)[threadIdx.x] =
                a.d ? __ldg(reinterpret_cast<const float4*>(a.d + (size_t)b * G) + threadIdx.x)
                    : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    if (a.params_ready) fetch_params();
    // the prologue above may overlap the previous kernel (programmatic launch)
    grid_dependency_wait();
    grid_launch_dependents();
    if (!a.params_ready) fetch_params();
    if (threadIdx.x == 0) {
        mbar_arrive_expect_tx(smem_addr(&zfull), P::Z_BYTES);
        for (int at = 0; at < P::ATOMS; ++at)
            tma_load_2d(sZ + at * (TC_TM * 128), &tmap_z, b * G + at * 64, row0, smem_addr(&zfull));
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    constexpr uint32_t IDESC = (1u << 4) | (Split16<TIn>::KIND << 7) | (Split16<TIn>::KIND << 10) |
                               ((uint32_t)(G >> 3) << 17) | ((uint32_t)(TC_TM >> 4) << 24);
    if (threadIdx.x == 0) {
        if (!mbar_wait_bounded(smem_addr(&zfull), 0, abort) ||
            (prepared && !mbar_wait_bounded(smem_addr(&mfull), 0, abort))) {
            *abort = 1;
        } else {
            tc_fence_after();
            #pragma unroll
            for (int ks = 0; ks < G / 16; ++ks) {
                const uint32_t koff = (ks / 4) * (TC_TM * 128) + (ks % 4) * 32;
                const uint32_t moff = (ks / 4) * (G * 128) + (ks % 4) * 32;
                const uint64_t ad = smem_desc_sw128(sZ + koff);
                mma_f16(tmem, ad, smem_desc_sw128(sMh + moff), IDESC, ks > 0 ? 1u : 0u);
                mma_f16(tmem, ad, smem_desc_sw128(sMl + moff), IDESC, 1u);
            }
        }
        tc_commit(smem_addr(&mdone));       // also after a failed wait: nothing was issued
    }
    bool ok = mbar_wait_bounded(smem_addr(&mdone), 0, abort) && !*abort;
    tc_fence_after();
    if (ok) {
        const int quarter = warp & 3, chalf = warp >> 2;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const int tok = row0 + quarter * 32 + lane;
        const uint32_t box = sZ + warp * (32 * 32 * 4);
        TOut* out = static_cast<TOut*>(a.out);
        #pragma unroll 1
        for (int c = 0; c < G / 64; ++c) {
            const int col = chalf * (G / 2) + c * 32;
            uint32_t r[32];
            tmem_ld_32x32b_x32(trow + col, r);
            tmem_ld_wait();
            float v[32];
            #pragma unroll
            for (int j = 0; j < 32; j += 4) {
                const float4 dd = reinterpret_cast<const float4*>(dsm + col)[j / 4];
                v[j] = __uint_as_float(r[j]) + dd.x;
                v[j + 1] = __uint_as_float(r[j + 1]) + dd.y;
                v[j + 2] = __uint_as_float(r[j + 2]) + dd.z;
                v[j + 3] = __uint_as_float(r[j + 3]) + dd.w;
            }
            if (TacStore<TOut>::TMA) {
                if (c > 0) {                                     // the previous box has been read
                    if (lane == 0) bulk_wait_read0();
                    __syncwarp();
                }
                if (sizeof(TOut) == 4) {                         // 128-byte rows: group q at q ^ (row & 7)
                    #pragma unroll
                    for (int q = 0; q < 8; ++q)
                        st_shared_v4(box + lane * 128 + ((q ^ (lane & 7)) << 4), __float_as_uint(v[4 * q]),
                                     __float_as_uint(v[4 * q + 1]), __float_as_uint(v[4 * q + 2]),
                                     __float_as_uint(v[4 * q + 3]));
                } else {                                         // 64-byte rows: group q at q ^ ((row >> 1) & 3)
                    #pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint32_t w[4];
                        #pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            TOut x0 = from_f<TOut>(v[8 * q + 2 * e]), x1 = from_f<TOut>(v[8 * q + 2 * e + 1]);
                            w[e] = (uint32_t)(*reinterpret_cast<uint16_t*>(&x0)) |
                                   ((uint32_t)(*reinterpret_cast<uint16_t*>(&x1)) << 16);
                        }
                        st_shared_v4(box + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4), w[0], w[1], w[2], w[3]);
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tmap_out, b * G + col, row0 + quarter * 32, box);
                    bulk_commit();
                }
            } else if (tok < a.L) {
                TOut* o = out + (size_t)tok * a.C + b * G + col;
                #pragma unroll
                for (int u = 0; u < 4; ++u) {
                    uint32_t w[4];
                    #pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        TOut x0 = from_f<TOut>(v[8 * u + 2 * e]), x1 = from_f<TOut>(v[8 * u + 2 * e + 1]);
                        w[e] = (uint32_t)(*reinterpret_cast<uint16_t*>(&x0)) |
                               ((uint32_t)(*reinterpret_cast<uint16_t*>(&x1)) << 16);
                    }
                    reinterpret_cast<uint4*>(o)[u] = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
        }
        if (TacStore<TOut>::TMA && lane == 0) bulk_wait0();
        __syncwarp();
    } else if (threadIdx.x == 0) {
        atomicOr(status, STATUS_TIMEOUT_TAC);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, P::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Streaming tensor-core TAC (prepared M, 16-bit Z, g = 64 or 128): the same
// products as tac_tc_kernel, in the same order, so the same bits. Persistent
// CTAs each take a contiguous run of the (block b, 128-token tile) jobs in
// block-major order, at most two blocks per run:
//   TMA warp   M_b's halves once per block (one bulk copy; the second block's
//              after the MMAs of the first have completed), then the Z tiles
//              through a ring of ZS stages;
//   MMA warp   per tile 2 g / 16 MMAs (Z M_hi^T, Z M_lo^T per K step) into one
//              of two TMEM accumulators;
//   8 warps    read the accumulator (a TMEM lane quarter, half the columns),
//              free it, add d_b, round to the output type and store 32 x 32
//              boxes by TMA from two staging boxes per warp.
// Loads, products and stores of consecutive tiles overlap.
// ---------------------------------------------------------------------------
constexpr int TS_EPI_WARPS = 8;
constexpr int TS_TMA_WARP = TS_EPI_WARPS, TS_MMA_WARP = TS_EPI_WARPS + 1;
constexpr int TS_THREADS = (TS_EPI_WARPS + 2) * 32;

template <int G, typename TOut>
struct TacStream {
    static constexpr int ATOMS = G / 64;
    static constexpr int Z_BYTES = TC_TM * G * 2;
    static constexpr int M_BYTES = G * G * 2;                          // one half
    static constexpr int BOX_BYTES = 32 * 32 * (int)sizeof(TOut);
    static constexpr int ZS = sizeof(TOut) == 4 ? 2 : 3;               // Z ring stages
    static constexpr int OFF_Z = 2 * M_BYTES;
    static constexpr int OFF_BOX = OFF_Z + ZS * Z_BYTES;
    static constexpr size_t SMEM = (size_t)OFF_BOX + (size_t)TS_EPI_WARPS * 2 * BOX_BYTES + 1024;
    static constexpr int TMEM_COLS = 2 * G;
    static_assert(SMEM <= 227 * 1024, "shared memory");
};

template <int G, typename TIn, typename TOut>
__global__ void __launch_bounds__(TS_THREADS, 1)
tac_stream_kernel(TacArgs a, const __grid_constant__ CUtensorMap tmap_z, const __grid_constant__ CUtensorMap tmap_out,
                  unsigned* status, int nt, long long jobs) {
    using P = TacStream<G, TOut>;
    extern __shared__ uint8_t smem_raw[];
    __shared__ __align__(8) uint64_t zfull[P::ZS], zempty[P::ZS], accfull[2], accempty[2], mfull, mempty;
    __shared__ __align__(16) float dsm[2][G];
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_flag;
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    const uint32_t sMh = base, sMl = base + P::M_BYTES;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    volatile int* abort = &abort_flag;
    auto B = [](const uint64_t& bar) { return smem_addr(&bar); };
    // this CTA's jobs [j0, j1): block j / nt, tile j mod nt
    const long long j0 = jobs * blockIdx.x / gridDim.x, j1 = jobs * (blockIdx.x + 1) / gridDim.x;
    const int n = (int)(j1 - j0);
    const int b0 = (int)(j0 / nt);

    if (threadIdx.x == 0) {
        for (int k = 0; k < P::ZS; ++k) {
            mbar_init(B(zfull[k]), 1);
            mbar_init(B(zempty[k]), 1);
        }
        for (int k = 0; k < 2; ++k) {
            mbar_init(B(accfull[k]), 1);
            mbar_init(B(accempty[k]), TS_EPI_WARPS);
        }
        mbar_init(B(mfull), 1);
        mbar_init(B(mempty), 1);
        abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == TS_MMA_WARP) {
        tmem_alloc(smem_addr(&tmem_slot), P::TMEM_COLS);
        tmem_relinquish();
    }
    grid_dependency_wait();            // launched with programmatic serialisation
    grid_launch_dependents();
    // d of the run's (at most two) blocks
    for (int i = threadIdx.x; i < 2 * G; i += blockDim.x) {
        const int bb = b0 + i / G;
        dsm[i / G][i % G] = (a.d != nullptr && bb < a.C / G) ? a.d[(size_t)bb * G + i % G] : 0.f;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;

    if (warp == TS_TMA_WARP) {
        bool ok = true;
        if (elect_one()) {
            int mb = -1, mloads = 0;
            for (int i = 0; i < n && ok; ++i) {
                const long long j = j0 + i;
                const int b = (int)(j / nt), t = (int)(j % nt);
                if (b != mb) {                               // the block's M halves (after the previous block's MMAs)
                    if (mloads > 0 && !mbar_wait_bounded(B(mempty), (uint32_t)((mloads - 1) & 1), abort)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(B(mfull), 2 * P::M_BYTES);
                    bulk_load(sMh, static_cast<const uint8_t*>(a.Mp) + (size_t)b * 2 * P::M_BYTES, 2 * P::M_BYTES,
                              B(mfull));
                    mb = b;
                    ++mloads;
                }
                const int k = i % P::ZS;
                if (!mbar_wait_bounded(B(zempty[k]), (uint32_t)(((i / P::ZS) & 1) ^ 1), abort)) { ok = false; break; }
                const uint32_t sZ = base + P::OFF_Z + (uint32_t)k * P::Z_BYTES;
                mbar_arrive_expect_tx(B(zfull[k]), P::Z_BYTES);
                for (int at = 0; at < P::ATOMS; ++at)
                    tma_load_2d(sZ + at * (TC_TM * 128), &tmap_z, b * G + at * 64, t * TC_TM, B(zfull[k]));
            }
            // the last commits on the Z ring have arrived before the CTA exits
            for (int i = n - P::ZS; i < n && ok; ++i)
                if (i >= 0) ok = mbar_wait_bounded(B(zempty[i % P::ZS]), (uint32_t)((i / P::ZS) & 1), abort);
            if (!ok) { *abort = 1; atomicOr(status, STATUS_TIMEOUT_TAC); }
        }
        __syncwarp();
    } else if (warp == TS_MMA_WARP) {
        if (elect_one()) {
            constexpr uint32_t IDESC = (1u << 4) | (Split16<TIn>::KIND << 7) | (Split16<TIn>::KIND << 10) |
                                       ((uint32_t)(G >> 3) << 17) | ((uint32_t)(TC_TM >> 4) << 24);
            bool ok = true;
            int mb = -1, mloads = 0, issued = 0;
            for (int i = 0; i < n && ok; ++i) {
                const int b = (int)((j0 + i) / nt);
                if (b != mb) {
                    if (mloads > 0) tc_commit(B(mempty));      // the previous block's MMAs done with M
                    if (!mbar_wait_bounded(B(mfull), (uint32_t)(mloads & 1), abort)) { ok = false; break; }
                    mb = b;
                    ++mloads;
                }
                const int k = i % P::ZS, acc = i & 1;
                if (!mbar_wait_bounded(B(zfull[k]), (uint32_t)((i / P::ZS) & 1), abort) ||
                    !mbar_wait_bounded(B(accempty[acc]), (uint32_t)(((i >> 1) & 1) ^ 1), abort)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sZ = base + P::OFF_Z + (uint32_t)k * P::Z_BYTES;
                #pragma unroll
                for (int ks = 0; ks < G / 16; ++ks) {
                    const uint32_t koff = (ks / 4) * (TC_TM * 128) + (ks % 4) * 32;
                    const uint32_t moff = (ks / 4) * (G * 128) + (ks % 4) * 32;
                    const uint64_t ad = smem_desc_sw128(sZ + koff);
                    mma_f16(tmem + (uint32_t)(acc * G), ad, smem_desc_sw128(sMh + moff), IDESC, ks > 0 ? 1u : 0u);
                    mma_f16(tmem + (uint32_t)(acc * G), ad, smem_desc_sw128(sMl + moff), IDESC, 1u);
                }
                tc_commit(B(zempty[k]));
                tc_commit(B(accfull[acc]));
                ++issued;
            }
            if (issued > 0) {                 // every MMA has completed before TMEM is released
                volatile int never = 0;
                if (!mbar_wait_bounded(B(accfull[(issued - 1) & 1]), (uint32_t)(((issued - 1) >> 1) & 1), &never))
                    ok = false;
            }
            if (!ok) { *abort = 1; atomicOr(status, STATUS_TIMEOUT_TAC); }
        }
        __syncwarp();
    } else {
        const int quarter = warp & 3, chalf = warp >> 2;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const uint32_t boxes = base + P::OFF_BOX + (uint32_t)warp * 2 * P::BOX_BYTES;
        int stores = 0;
        bool ok = true;
        for (int i = 0; i < n && ok; ++i) {
            const long long j = j0 + i;
            const int b = (int)(j / nt), t = (int)(j % nt);
            const int acc = i & 1;
            if (!mbar_wait_bounded_warp(B(accfull[acc]), (uint32_t)((i >> 1) & 1), abort)) { ok = false; break; }
            tc_fence_after();
            uint32_t r[G / 64][32];
            #pragma unroll
            for (int c = 0; c < G / 64; ++c)
                tmem_ld_32x32b_x32(trow + (uint32_t)(acc * G + chalf * (G / 2) + c * 32), r[c]);
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(accempty[acc]));      // the accumulator may take the next tile
            const float* dd = dsm[b - b0];
            #pragma unroll
            for (int c = 0; c < G / 64; ++c) {
                const int col = chalf * (G / 2) + c * 32;
                float v[32];
                #pragma unroll
                for (int q = 0; q < 32; ++q) v[q] = __uint_as_float(r[c][q]) + dd[col + q];
                const uint32_t box = boxes + (uint32_t)(stores & 1) * P::BOX_BYTES;
                if (stores >= 2) {                               // the store from this box two boxes ago has read it
                    if (lane == 0) bulk_wait_read1();
                    __syncwarp();
                }
                if (sizeof(TOut) == 4) {                         // 128-byte rows: group q at q ^ (row & 7)
                    #pragma unroll
                    for (int q = 0; q < 8; ++q)
                        st_shared_v4(box + lane * 128 + ((q ^ (lane & 7)) << 4), __float_as_uint(v[4 * q]),
                                     __float_as_uint(v[4 * q + 1]), __float_as_uint(v[4 * q + 2]),
                                     __float_as_uint(v[4 * q + 3]));
                } else {                                         // 64-byte rows: group q at q ^ ((row >> 1) & 3)
                    #pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        uint32_t w[4];
                        #pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            TOut x0 = from_f<TOut>(v[8 * q + 2 * e]), x1 = from_f<TOut>(v[8 * q + 2 * e + 1]);
                            w[e] = (uint32_t)(*reinterpret_cast<uint16_t*>(&x0)) |
                                   ((uint32_t)(*reinterpret_cast<uint16_t*>(&x1)) << 16);
                        }
                        st_shared_v4(box + lane * 64 + ((q ^ ((lane >> 1) & 3)) << 4), w[0], w[1], w[2], w[3]);
                    }
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tmap_out, b * G + col, t * TC_TM + quarter * 32, box);
                    bulk_commit();
                }
                ++stores;
            }
        }
        if (lane == 0) bulk_wait0();
        __syncwarp();
        if (!ok && lane == 0) { *abort = 1; atomicOr(status, STATUS_TIMEOUT_TAC); }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == TS_MMA_WARP) tmem_dealloc(tmem, P::TMEM_COLS);
}

bool encode_u16_tmap(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint32_t box_rows,
                     uint32_t box_cols) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * 2};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Output tensor map with 32 x 32 boxes: float (128-byte rows, 128-byte
// swizzle) or a 16-bit type (64-byte rows, 64-byte swizzle).
bool encode_out_tmap16or32(CUtensorMap* m, void* ptr, size_t elem, bool is_f16, uint64_t rows, uint64_t cols) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {cols * elem};
    const cuuint32_t box[2] = {32, 32};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapDataType type = elem == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32
                                     : (is_f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16);
    return fn(m, type, 2, ptr, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
              elem == 4 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int G, typename TIn, typename TOut>
cudaError_t launch_tc(const TacArgs& a, cudaStream_t stream) {
    using P = TacTc<G>;
    static DeviceCache<int> attr;
    int done = 0;
    const cudaError_t e = attr.get(&done, [](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(tac_tc_kernel<G, TIn, TOut>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)P::SMEM);
    });
    if (e != cudaSuccess) return e;
    CUtensorMap tz, to;
    if (!encode_u16_tmap(&tz, a.Z, (uint64_t)a.L, (uint64_t)a.C, TC_TM, 64)) return cudaErrorInvalidValue;
    if (!encode_out_tmap16or32(&to, a.out, sizeof(TOut), std::is_same<TOut, __half>::value, (uint64_t)a.L,
                               (uint64_t)a.C))
        return cudaErrorInvalidValue;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1] = {pdl_attribute()};
    cfg.gridDim = dim3(a.C / G, (a.L + TC_TM - 1) / TC_TM);
    cfg.blockDim = dim3(TC_THREADS);
    cfg.dynamicSmemBytes = P::SMEM;
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tac_tc_kernel<G, TIn, TOut>, a, tz, to, a.status);
}

template <int G, typename TIn, typename TOut>
cudaError_t launch_stream(const TacArgs& a, cudaStream_t stream) {
    using P = TacStream<G, TOut>;
    static DeviceCache<int> attr;
    int done = 0;
    const cudaError_t e = attr.get(&done, [](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(tac_stream_kernel<G, TIn, TOut>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)P::SMEM);
    });
    if (e != cudaSuccess) return e;
    CUtensorMap tz, to;
    if (!encode_u16_tmap(&tz, a.Z, (uint64_t)a.L, (uint64_t)a.C, TC_TM, 64)) return cudaErrorInvalidValue;
    if (!encode_out_tmap16or32(&to, a.out, sizeof(TOut), std::is_same<TOut, __half>::value, (uint64_t)a.L,
                               (uint64_t)a.C))
        return cudaErrorInvalidValue;
    // at least one CTA per block, so that a CTA's run of jobs (at most nt
    // long) spans at most two blocks
    const int nb = a.C / G, nt = (a.L + TC_TM - 1) / TC_TM;
    const long long jobs = (long long)nb * nt;
    long long ctas = jobs < num_sms() ? jobs : num_sms();
    if (ctas < nb) ctas = nb;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1] = {pdl_attribute()};
    cfg.gridDim = dim3((unsigned)ctas);
    cfg.blockDim = dim3(TS_THREADS);
    cfg.dynamicSmemBytes = P::SMEM;
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, tac_stream_kernel<G, TIn, TOut>, a, tz, to, a.status, nt, jobs);
}

template <typename TIn, typename TOut>
cudaError_t launch_io(const TacArgs& a, cudaStream_t stream) {
    if constexpr (!std::is_same<TIn, float>::value) {
        if (a.status != nullptr && (a.g == 64 || a.g == 128)) {
            // prepared halves and more jobs than one wave of the per-tile
            // kernel (two CTAs per SM) holds: the streaming kernel
            const long long jobs = (long long)(a.C / a.g) * ((a.L + TC_TM - 1) / TC_TM);
            if (a.Mp != nullptr && jobs > 2LL * num_sms())
                return a.g == 64 ? launch_stream<64, TIn, TOut>(a, stream) : launch_stream<128, TIn, TOut>(a, stream);
            return a.g == 64 ? launch_tc<64, TIn, TOut>(a, stream) : launch_tc<128, TIn, TOut>(a, stream);
        }
    }
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

cudaError_t launch_tac_prepare(const float* M, int C, int g, int z_dtype, void* Mp, cudaStream_t stream) {
    if (C == 0) return cudaSuccess;
    uint8_t* out = static_cast<uint8_t*>(Mp);
    dim3 grid(C / g);
    if (z_dtype == STARQ_F16) {
        if (g == 64) tac_prepare_kernel<64, __half><<<grid, 256, 0, stream>>>(M, out);
        else tac_prepare_kernel<128, __half><<<grid, 256, 0, stream>>>(M, out);
    } else {
        if (g == 64) tac_prepare_kernel<64, __nv_bfloat16><<<grid, 256, 0, stream>>>(M, out);
        else tac_prepare_kernel<128, __nv_bfloat16><<<grid, 256, 0, stream>>>(M, out);
    }
    return cudaGetLastError();
}

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
