// Tensor-core rate probe: the denominators of the GEMM rooflines, measured
// on the device that runs the library (the paper has no counterpart).
//
// Kinds (every CTA issues `iters` rounds of back-to-back MMAs on operands
// resident in shared memory or registers, then checks its accumulators):
//   0  tcgen05.mma cta_group::1 kind::f8f6f4, E4M3 x E4M3 -> F32, M 128,
//      N 256, K 32 (the W4A4 path's instruction kind); operands all
//      E4M3(7), so every accumulator must come back as 49 * 128 * iters,
//      an integer below 2^24: the raw integer-exactness check of the FP8
//      tensor-core accumulation.
//   1  the same as a CTA pair, cta_group::2 (M 256 over the pair, N 256),
//      the form the W4A4 GEMM issues.
//   2  tcgen05.mma cta_group::1 kind::f16 with bf16 operands (1.0), M 128,
//      N 256, K 16: the 16-bit rate (accumulators 64 * iters).
//   3  mma.sync m16n8k32 s8.s8.s32 (the integer MMA that sm_103a still
//      offers, through the warp-level instruction; eight independent
//      accumulator chains per warp; accumulators 32 * iters).
//   4  mma.sync m16n8k64 s4.s4.s32 (accumulators 64 * iters).
// Each CTA records its cycles from the first issue to the last completion;
// the caller times the launch with events. Every wait is bounded.
#include "common.cuh"

namespace starq {
namespace {

constexpr unsigned STATUS_TIMEOUT_PROBE = 1u << 6;
constexpr int PROBE_THREADS = 128;
constexpr int PROBE_SMEM = 64 * 1024 + 1024;     // A at 0 (16 KB), B at 32 KB (32 KB)
constexpr int SYNC_WARPS = 4;                    // warps per CTA of the mma.sync kinds
constexpr int SYNC_CHAINS = 8;                   // independent accumulators per warp

template <int KIND>
__global__ void __launch_bounds__(PROBE_THREADS, 1)
probe_tc_kernel(int iters, unsigned long long* cycles, int* errors, unsigned* status) {
    constexpr bool PAIR = KIND == 1;
    constexpr bool F16 = KIND == 2;
    constexpr int M = PAIR ? 256 : 128, N = 256;
    extern __shared__ uint8_t probe_smem[];
    __shared__ __align__(8) uint64_t done;
    __shared__ uint32_t tmem_slot;
    const uint32_t raw = smem_addr(probe_smem);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint32_t* const words = reinterpret_cast<uint32_t*>(probe_smem + (base - raw));
    // E4M3(7) = 0x4E in every byte; bf16(1.0) = 0x3F80 in every half
    const uint32_t fill = F16 ? 0x3F803F80u : 0x4E4E4E4Eu;
    for (int i = threadIdx.x; i < 64 * 1024 / 4; i += PROBE_THREADS) words[i] = fill;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = PAIR ? cluster_ctarank() : 0u;
    if (threadIdx.x == 0) {
        mbar_init(smem_addr(&done), 1);
        mbar_fence_init();
    }
    if (warp == 0) {
        if (PAIR) { tmem_alloc_pair(smem_addr(&tmem_slot), 256); tmem_relinquish_pair(); }
        else { tmem_alloc(smem_addr(&tmem_slot), 256); tmem_relinquish(); }
    }
    fence_proxy_async_smem();
    tc_fence_before();
    if (PAIR) cluster_sync(); else __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    // f32 accumulator (bit 4), bf16 inputs (bits 7, 10) for the 16-bit kind
    constexpr uint32_t IDESC = (1u << 4) | (F16 ? ((1u << 7) | (1u << 10)) : 0u) |
                               ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
    const long long t0 = clock64();
    if (threadIdx.x == 0 && rank == 0) {
        const uint64_t ad = smem_desc_sw128(base), bd = smem_desc_sw128(base + 32768);
        for (int i = 0; i < iters; ++i) {
            #pragma unroll
            for (int j = 0; j < 4; ++j) {            // four K steps of one 128-byte row
                const uint32_t acc = (i | j) ? 1u : 0u;
                const uint64_t step = (uint64_t)(j * 2);    // 32 bytes in 16-byte units
                if (KIND == 0) mma_f8f6f4(tmem, ad + step, bd + step, IDESC, acc);
                if (KIND == 1) mma_f8f6f4_pair(tmem, ad + step, bd + step, IDESC, acc);
                if (KIND == 2) mma_f16(tmem, ad + step, bd + step, IDESC, acc);
            }
        }
        if (PAIR) tc_commit_pair_multicast(smem_addr(&done), 3u);
        else tc_commit(smem_addr(&done));
    }
    volatile int never = 0;
    const bool ok = mbar_wait_bounded(smem_addr(&done), 0, &never);
    const long long t1 = clock64();
    if (threadIdx.x == 0) {
        cycles[blockIdx.x] = ok ? (unsigned long long)(t1 - t0) : 0ull;
        if (!ok) atomicOr(status, STATUS_TIMEOUT_PROBE);
    }
    if (ok) {
        // every accumulator of this CTA's 128 lanes: lanes 32 w .. of warp w
        tc_fence_after();
        const float expect = F16 ? 64.f * (float)iters : 49.f * 128.f * (float)iters;
        int bad = 0;
        #pragma unroll 1
        for (int c = 0; c < N; c += 32) {
            uint32_t r[32];
            tmem_ld_32x32b_x32(tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)c, r);
            tmem_ld_wait();
            #pragma unroll
            for (int k = 0; k < 32; ++k) bad += __uint_as_float(r[k]) != expect;
        }
        if (bad) atomicAdd(errors, bad);
    }
    (void)lane;
    tc_fence_before();
    if (PAIR) cluster_sync(); else __syncthreads();
    tc_fence_after();
    if (warp == 0) {
        if (PAIR) tmem_dealloc_pair(tmem, 256);
        else tmem_dealloc(tmem, 256);
    }
}

// mma.sync rates: SYNC_CHAINS independent accumulators per warp, A and B
// of all ones (s8: 0x01 bytes; s4: 0x1 nibbles), so every accumulator of
// the k32 s8 instruction grows by 32 and of the k64 s4 one by 64 per issue.
template <bool S4>
__global__ void __launch_bounds__(32 * SYNC_WARPS)
probe_sync_kernel(int iters, unsigned long long* cycles, int* errors, uint32_t one) {
    // one = 0x11111111 (s4) or 0x01010101 (s8), passed at run time so that
    // nothing about the operands is known when the kernel is compiled
    uint32_t a0 = one, a1 = one, a2 = one, a3 = one, b0 = one, b1 = one;
    int c[SYNC_CHAINS][4];
    #pragma unroll
    for (int q = 0; q < SYNC_CHAINS; ++q) c[q][0] = c[q][1] = c[q][2] = c[q][3] = 0;
    __syncthreads();
    const long long t0 = clock64();
    #pragma unroll 1
    for (int i = 0; i < iters; ++i) {
        #pragma unroll
        for (int q = 0; q < SYNC_CHAINS; ++q) {
            if (S4)
                asm volatile("mma.sync.aligned.m16n8k64.row.col.s32.s4.s4.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
                             "{%8,%9}, {%0,%1,%2,%3};"
                             : "+r"(c[q][0]), "+r"(c[q][1]), "+r"(c[q][2]), "+r"(c[q][3])
                             : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
            else
                asm volatile("mma.sync.aligned.m16n8k32.row.col.s32.s8.s8.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
                             "{%8,%9}, {%0,%1,%2,%3};"
                             : "+r"(c[q][0]), "+r"(c[q][1]), "+r"(c[q][2]), "+r"(c[q][3])
                             : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
        }
    }
    __syncthreads();
    const long long t1 = clock64();
    if (threadIdx.x == 0) cycles[blockIdx.x] = (unsigned long long)(t1 - t0);
    const int expect = (S4 ? 64 : 32) * iters;
    int bad = 0;
    #pragma unroll
    for (int q = 0; q < SYNC_CHAINS; ++q)
        #pragma unroll
        for (int k = 0; k < 4; ++k) bad += c[q][k] != expect;
    if (bad) atomicAdd(errors, bad);
}

}  // namespace

cudaError_t launch_probe_mma(int kind, int iters, unsigned long long* cycles, int* errors, unsigned* status,
                             int* ctas, double* macs_per_cta, cudaStream_t stream) {
    const int sms = num_sms();
    if (kind <= 2) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute at[1];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = kind == 1 ? 2 : 1;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(kind == 1 ? sms - (sms & 1) : sms);
        cfg.blockDim = dim3(PROBE_THREADS);
        cfg.dynamicSmemBytes = PROBE_SMEM;
        cfg.stream = stream;
        cfg.attrs = at;
        cfg.numAttrs = 1;
        static DeviceCache<int> attr;
        int done = 0;
        cudaError_t e = attr.get(&done, [](int, int* v) {
            *v = 1;
            cudaError_t r = cudaFuncSetAttribute(probe_tc_kernel<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, PROBE_SMEM);
            if (r == cudaSuccess)
                r = cudaFuncSetAttribute(probe_tc_kernel<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, PROBE_SMEM);
            if (r == cudaSuccess)
                r = cudaFuncSetAttribute(probe_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize, PROBE_SMEM);
            return r;
        });
        if (e != cudaSuccess) return e;
        *ctas = (int)cfg.gridDim.x;
        // per CTA: 128 rows x 256 columns x (32 or 16) K per MMA, 4 MMAs per round
        *macs_per_cta = 128.0 * 256.0 * (kind == 2 ? 16.0 : 32.0) * 4.0 * iters;
        switch (kind) {
            case 0: return cudaLaunchKernelEx(&cfg, probe_tc_kernel<0>, iters, cycles, errors, status);
            case 1: return cudaLaunchKernelEx(&cfg, probe_tc_kernel<1>, iters, cycles, errors, status);
            default: return cudaLaunchKernelEx(&cfg, probe_tc_kernel<2>, iters, cycles, errors, status);
        }
    }
    const int grid = 4 * sms;
    *ctas = grid;
    *macs_per_cta = (double)SYNC_WARPS * SYNC_CHAINS * iters * (16.0 * 8.0 * (kind == 4 ? 64.0 : 32.0));
    if (kind == 3) probe_sync_kernel<false><<<grid, 32 * SYNC_WARPS, 0, stream>>>(iters, cycles, errors, 0x01010101u);
    else probe_sync_kernel<true><<<grid, 32 * SYNC_WARPS, 0, stream>>>(iters, cycles, errors, 0x11111111u);
    return cudaGetLastError();
}

}  // namespace starq
