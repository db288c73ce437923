// The W4A4 GEMM on the warp-level integer MMA (mma.sync m16n8k64 s4.s4.s32,
// the only int4 tensor-core instruction sm_103a offers): the comparison
// point of the integer-path choice (Sec. 3.2 Eq. 13 / Eq. 5; the same
// contract as w4a4_gemm with packed operands).
//
//   acc[i][n] = sum_k q_a[i][k] q_w[n][k]     int32, exact
//   Y[i][n]   = fl(fl((float)acc s_a[i]) s_w[n]) (+ bias[n]) rounded to the
//               output type
//
// A CTA of 8 warps computes a 128 x 128 output tile; warp (wm, wn) a 64 x 32
// block as 4 x 4 MMA tiles of 16 x 8. The packed codes (two per byte, low
// nibble = even k) are exactly the s4 fragment format: eight consecutive
// codes of a row are one 32-bit register. K advances 64 codes (32 bytes per
// row) per step through two shared-memory stages filled by 16-byte cp.async;
// rows are padded to 48 bytes so the fragment loads (row = lane / 4, word =
// lane % 4) fall in distinct banks.
#include "common.cuh"

namespace starq {
namespace {

constexpr int MS_BM = 128, MS_BN = 128, MS_BK = 64;       // codes
constexpr int MS_ROW = 48;                                // bytes per padded smem row (32 used)
constexpr int MS_TILE = MS_BM * MS_ROW;                   // bytes per operand stage
constexpr int MS_THREADS = 256;

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, bool valid) {
    const int n = valid ? 16 : 0;                          // zero-fill rows beyond the matrix
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" :: "r"(dst), "l"(src), "r"(n) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait1() { asm volatile("cp.async.wait_group 1;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait0() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

__device__ __forceinline__ void mma_s4(int (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k64.row.col.s32.s4.s4.s32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};"
                 : "+r"(c[0]), "+r"(c[1]), "+r"(c[2]), "+r"(c[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

template <typename TOut> struct OutCvt;
template <> struct OutCvt<float> { static __device__ __forceinline__ float f(float v) { return v; } };
template <> struct OutCvt<__half> { static __device__ __forceinline__ __half f(float v) { return __float2half_rn(v); } };
template <> struct OutCvt<__nv_bfloat16> {
    static __device__ __forceinline__ __nv_bfloat16 f(float v) { return __float2bfloat16_rn(v); }
};

template <typename TOut>
__global__ void __launch_bounds__(MS_THREADS)
w4a4_gemm_mmasync_kernel(GemmArgs a) {
    __shared__ __align__(16) uint8_t sA[2][MS_TILE];
    __shared__ __align__(16) uint8_t sB[2][MS_TILE];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wm = warp >> 2, wn = warp & 3;               // warp tile: rows 64 wm, columns 32 wn
    const int g = lane >> 2, t = lane & 3;                 // fragment group and thread in group
    const int row0 = blockIdx.y * MS_BM, col0 = blockIdx.x * MS_BN;
    const int KB = a.K / 2;                                // bytes per packed row
    const int steps = a.K / MS_BK;

    // one 16-byte load of each operand per thread and step: row tid / 2, half tid % 2
    const int lr = tid >> 1, lh = tid & 1;
    const bool a_ok = row0 + lr < a.L, b_ok = col0 + lr < a.N;
    const uint8_t* ga = a.Xq + (size_t)(a_ok ? row0 + lr : 0) * KB + 16 * lh;
    const uint8_t* gb = a.Wq + (size_t)(b_ok ? col0 + lr : 0) * KB + 16 * lh;
    const uint32_t da = smem_addr(&sA[0][0]) + lr * MS_ROW + 16 * lh;
    const uint32_t db = smem_addr(&sB[0][0]) + lr * MS_ROW + 16 * lh;
    auto load = [&](int s, int buf) {
        cp_async16(da + buf * MS_TILE, ga + (size_t)s * 32, a_ok);
        cp_async16(db + buf * MS_TILE, gb + (size_t)s * 32, b_ok);
        cp_async_commit();
    };

    int acc[4][4][4];
    #pragma unroll
    for (int i = 0; i < 4; ++i)
        #pragma unroll
        for (int j = 0; j < 4; ++j)
            #pragma unroll
            for (int k = 0; k < 4; ++k) acc[i][j][k] = 0;

    load(0, 0);
    for (int s = 0; s < steps; ++s) {
        const int buf = s & 1;
        if (s + 1 < steps) {
            load(s + 1, buf ^ 1);
            cp_async_wait1();
        } else {
            cp_async_wait0();
        }
        __syncthreads();
        const uint8_t* A = sA[buf];
        const uint8_t* Bm = sB[buf];
        uint32_t af[4][4], bf[4][2];
        #pragma unroll
        for (int i = 0; i < 4; ++i) {                      // rows 64 wm + 16 i + g (+ 8), words t and t + 4
            const uint8_t* r0 = A + (64 * wm + 16 * i + g) * MS_ROW + 4 * t;
            const uint8_t* r1 = r0 + 8 * MS_ROW;
            af[i][0] = *reinterpret_cast<const uint32_t*>(r0);
            af[i][1] = *reinterpret_cast<const uint32_t*>(r1);
            af[i][2] = *reinterpret_cast<const uint32_t*>(r0 + 16);
            af[i][3] = *reinterpret_cast<const uint32_t*>(r1 + 16);
        }
        #pragma unroll
        for (int j = 0; j < 4; ++j) {                      // columns 32 wn + 8 j + g, words t and t + 4
            const uint8_t* c = Bm + (32 * wn + 8 * j + g) * MS_ROW + 4 * t;
            bf[j][0] = *reinterpret_cast<const uint32_t*>(c);
            bf[j][1] = *reinterpret_cast<const uint32_t*>(c + 16);
        }
        #pragma unroll
        for (int i = 0; i < 4; ++i)
            #pragma unroll
            for (int j = 0; j < 4; ++j) mma_s4(acc[i][j], af[i], bf[j][0], bf[j][1]);
        __syncthreads();                                   // the stage may be refilled
    }

    // epilogue: c0, c1 at row g, columns 2 t, 2 t + 1; c2, c3 at row g + 8
    TOut* Y = static_cast<TOut*>(a.Y);
    #pragma unroll
    for (int i = 0; i < 4; ++i) {
        #pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int r = row0 + 64 * wm + 16 * i + g + 8 * h;
            if (r >= a.L) continue;
            const float sa = a.s_a[r];
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                #pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const int n = col0 + 32 * wn + 8 * j + 2 * t + e;
                    if (n >= a.N) continue;
                    const int v = acc[i][j][2 * h + e];
                    float y = __fmul_rn(__fmul_rn((float)v, sa), a.s_w[n]);
                    if (a.bias != nullptr) y = __fadd_rn(y, a.bias[n]);
                    Y[(size_t)r * a.N + n] = OutCvt<TOut>::f(y);
                    if (a.acc_dbg != nullptr) a.acc_dbg[(size_t)r * a.N + n] = v;
                }
            }
        }
    }
}

}  // namespace

cudaError_t launch_w4a4_gemm_mmasync(const GemmArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    const dim3 grid((a.N + MS_BN - 1) / MS_BN, (a.L + MS_BM - 1) / MS_BM);
    switch (a.y_dtype) {
        case STARQ_F16: w4a4_gemm_mmasync_kernel<__half><<<grid, MS_THREADS, 0, stream>>>(a); break;
        case STARQ_BF16: w4a4_gemm_mmasync_kernel<__nv_bfloat16><<<grid, MS_THREADS, 0, stream>>>(a); break;
        case STARQ_F32: w4a4_gemm_mmasync_kernel<float><<<grid, MS_THREADS, 0, stream>>>(a); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

}  // namespace starq
