// Device-side helpers shared by the libstarq kernels (sm_103a only):
// mbarrier and tcgen05 PTX wrappers, bounded waits, shared-memory matrix
// descriptors, and the launcher interface between the C ABI and the kernels.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <cuda_fp16.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include "../../include/starq.h"

namespace starq {

// Bits of the device status word (set with atomicOr, read and cleared by
// starq_check_status).
constexpr unsigned STATUS_TIMEOUT_GEMM = 1u << 0;
constexpr unsigned STATUS_TIMEOUT_FP16_GEMM = 1u << 1;
constexpr unsigned STATUS_TIMEOUT_TEST = 1u << 2;
constexpr unsigned STATUS_TIMEOUT_TAC = 1u << 3;

// Upper bound of any single wait inside a kernel. Kernels of this library
// finish in milliseconds; a wait this long means a broken pipeline, and the
// kernel gives up, records it and returns instead of hanging the GPU.
constexpr unsigned long long WAIT_LIMIT_NS = 2000000000ull;  // 2 s

// ---------------------------------------------------------------------------
// Launchers (host functions in each kernel translation unit). Arguments are
// validated by the C ABI before these are called.
// ---------------------------------------------------------------------------
struct QuantArgs {
    const void* X; int x_dtype; int L; int K;
    const uint8_t* mask; const float* a_m; const float* a_u;
    int hb; int d_sh; int d_m; int d_u;
    int qmax; float post_scale;
    uint8_t* Xq; float* s; float* v_dbg;
    uint8_t* Xe = nullptr;   // optional E4M3 byte copy of the codes [L][K]
    // asymmetric activation quantiser (Eq. 2-4): codes in [0, qmax], zero
    // points out to z [L]; Xe rows are K + 128 long, the last 128 bytes the
    // E4M3 of -z (the zero-point columns of the augmented contraction)
    int asym = 0;
    int32_t* z = nullptr;
    // the caller guarantees that the launch just before this one on the
    // stream neither writes X, mask, a_m, a_u nor reads or writes the
    // outputs, so the rows may start before it completes (programmatic
    // launch; everything earlier has completed by then)
    int independent = 0;
};
cudaError_t launch_sgat_quant(const QuantArgs& a, cudaStream_t stream);
// Two quantisations in one launch when both run the row kernel with one CTA
// per row (the same input type, K <= 4096, hb and code width, symmetric);
// otherwise two launches.
cudaError_t launch_sgat_quant_grouped(const QuantArgs& a, const QuantArgs& b, cudaStream_t stream);

struct GemmArgs {
    const uint8_t* Xq; const float* s_a; const uint8_t* Wq; const float* s_w;
    const float* bias; int L; int N; int K;
    void* Y; int y_dtype; int32_t* acc_dbg;
    unsigned* status;
    const uint8_t* Xe = nullptr;   // optional E4M3 bytes of the activation codes [L][K]
    const uint8_t* We = nullptr;   // optional E4M3 bytes of the weight codes [N][K]
    // The caller guarantees that no kernel still running when this one is
    // launched writes the weights: their first tiles are fetched before
    // the wait for the previous kernel (programmatic launch).
    int weights_ready = 0;
    // Epilogue silu(gate) * up over weight rows interleaved in groups of 16
    // (Xe + We path, 16-bit Y of [L][N / 2]).
    int swiglu = 0;
};
cudaError_t launch_w4a4_gemm(const GemmArgs& a, cudaStream_t stream);
// Two independent products in one persistent TMA pair launch (the same L,
// K and output type; Xe and We given for both; no SwiGLU).
cudaError_t launch_w4a4_gemm_grouped(const GemmArgs& a, const GemmArgs& b, cudaStream_t stream);
// Thread-local cap on the CTA pairs of the TMA pair GEMMs launched from the
// calling thread (0 = none); returns the previous cap.
int set_gemm_pair_limit(int pairs);
// The same product on the warp-level int4 MMA (mma.sync s4), packed operands.
cudaError_t launch_w4a4_gemm_mmasync(const GemmArgs& a, cudaStream_t stream);
// Tile of the calling thread's last TMA pair GEMM launch (BN * 10 + cluster
// size; 0 before the first).
int last_gemm_tile();
// Plain 16-bit GEMM C = A B^T (A = a.Xe [L][K], B = a.We [N][K], both of
// type a.y_dtype, float32 accumulation, C = a.Y), no scales.
cudaError_t launch_fp16_gemm(const GemmArgs& a, cudaStream_t stream);
// Packed int4 codes [rows][K/2] -> E4M3 bytes [rows][K].
cudaError_t launch_unpack_e4m3(const uint8_t* packed, uint8_t* e4m3, size_t rows, int K, cudaStream_t stream);

// Launch attribute that lets a kernel overlap its launch and prologue with
// the tail of the previous kernel in the stream (see grid_dependency_wait).
inline cudaLaunchAttribute pdl_attribute() {
    cudaLaunchAttribute at;
    at.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at.val.programmaticStreamSerializationAllowed = 1;
    return at;
}

struct TacArgs {
    const void* Z; int z_dtype; int L; int C; int g;
    const float* M; const float* d; void* out; int out_dtype;
    unsigned* status = nullptr;   // device status word (tensor-core path)
    const void* Mp = nullptr;     // optional tac_prepare output (tensor-core path)
    // The caller guarantees that no kernel still running when this one is
    // launched writes Mp or d: they are fetched before the wait for the
    // previous kernel (programmatic launch).
    int params_ready = 0;
};
cudaError_t launch_tac(const TacArgs& a, cudaStream_t stream);
// M [C/g][g][g] float32 -> its 16-bit halves (hi = rn(M), lo = rn(M - hi), of
// type z_dtype) in the tensor-core operand layout: per block b, 2 g g 16-bit
// values (hi then lo, each K-major with the 128-byte swizzle).
cudaError_t launch_tac_prepare(const float* M, int C, int g, int z_dtype, void* Mp, cudaStream_t stream);

int num_sms();  // SM count of the current device (cached per device)
// Glue (glue.cu): residual add + RMSNorm, rotary position embedding.
cudaError_t launch_add_rmsnorm(const void* X, const void* R, int dtype, int L, int K, const float* w, float eps,
                               void* h_out, void* Y, cudaStream_t stream);
cudaError_t launch_rope(void* QK, int dtype, int L, int ld, int heads, const int* pos, double theta,
                        cudaStream_t stream);
// Tensor-core rate probe (probe.cu): kind 0..4, `cycles` [ctas] and `errors`
// device buffers; *ctas and *macs_per_cta describe the launch.
cudaError_t launch_probe_mma(int kind, int iters, unsigned long long* cycles, int* errors, unsigned* status,
                             int* ctas, double* macs_per_cta, cudaStream_t stream);
int report_error(int code, const char* msg);  // record msg for starq_last_error(), return code

// sgat_linear with a workspace that the library owns (the device scratch
// array of sgat_linear_noalloc), which the device-memory check skips.
int sgat_linear_scratch(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                        const float* a_u, int hb, int d_sh, int d_m, int d_u, const float* tac_M, const float* tac_d,
                        int tac_g, const void* tac_Mp, const uint8_t* Wq, const uint8_t* We, const float* s_w,
                        const float* bias, int N, int bits, void* Y, int y_dtype, void* scratch, size_t scratch_bytes,
                        void* stream);

// cuTensorMapEncodeTiled from the driver (looked up once, thread-safe), or
// nullptr when the driver does not provide it.
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder();

// A value per device, computed once by `init(dev, &value)` with that device
// current. Several host threads may call get() at once: the first caller for
// a device computes the value under a lock, the others wait for it or read
// the published value; a failed init leaves the entry unset for a retry.
template <typename T>
class DeviceCache {
  public:
    static constexpr int MAX_DEVICES = 64;
    template <typename F>
    cudaError_t get(T* out, F&& init) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e != cudaSuccess) return e;
        if (dev < 0 || dev >= MAX_DEVICES) return cudaErrorInvalidDevice;
        if (!ready_[dev].load(std::memory_order_acquire)) {
            std::lock_guard<std::mutex> lock(mu_);
            if (!ready_[dev].load(std::memory_order_relaxed)) {
                T v{};
                e = init(dev, &v);
                if (e != cudaSuccess) return e;
                val_[dev] = v;
                ready_[dev].store(true, std::memory_order_release);
            }
        }
        *out = val_[dev];
        return cudaSuccess;
    }

  private:
    std::mutex mu_;
    T val_[MAX_DEVICES] = {};
    std::atomic<bool> ready_[MAX_DEVICES] = {};
};

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ unsigned long long globaltimer_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_fence_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("{\n\t.reg .b64 st;\n\tmbarrier.arrive.shared::cta.b64 st, [%0];\n\t}"
                 :: "r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile("{\n\t.reg .pred p;\n\t"
                 "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}"
                 : "=r"(ok) : "r"(bar), "r"(parity) : "memory");
    return ok != 0;
}

// Programmatic dependent launch. A kernel launched with the programmatic
// stream-serialisation attribute may start while the previous kernel of the
// stream is still running; it must call grid_dependency_wait() before its
// first global-memory access (that waits until the previous grid has
// completed and its writes are visible; a no-op without a programmatic
// predecessor). grid_launch_dependents() lets the next such launch begin
// once every CTA of this grid has called it or exited.
__device__ __forceinline__ void grid_dependency_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void grid_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// One lane of a converged warp (the lowest active lane) gets true.
__device__ __forceinline__ bool elect_one() {
    uint32_t pred;
    asm volatile("{\n\t.reg .pred p;\n\t.reg .b32 r;\n\t"
                 "elect.sync r|p, 0xffffffff;\n\t"
                 "selp.u32 %0, 1, 0, p;\n\t}" : "=r"(pred));
    return pred != 0;
}

// Wait for the phase of `bar` with the given parity to complete. Gives up
// (returns false) after limit_ns nanoseconds, or early when *abort is set by
// another role of the same CTA that has already given up.
__device__ __forceinline__ bool mbar_wait_limit(uint32_t bar, uint32_t parity, volatile int* abort,
                                                unsigned long long limit_ns) {
    #pragma unroll 1
    for (int i = 0; i < 256; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = globaltimer_ns();
    #pragma unroll 1
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (globaltimer_ns() - t0 > limit_ns) return false;
    }
}

// The same with the library-wide limit WAIT_LIMIT_NS.
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  volatile int* abort) {
    return mbar_wait_limit(bar, parity, abort, WAIT_LIMIT_NS);
}

// Same, polling every `sleep_ns` nanoseconds: for waits that are not on a
// critical path, so the spinning warp leaves issue slots to its neighbours.
__device__ __forceinline__ bool mbar_wait_bounded_sleepy(uint32_t bar, uint32_t parity, volatile int* abort,
                                                         unsigned sleep_ns) {
    const unsigned long long t0 = globaltimer_ns();
    #pragma unroll 1
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort) return false;
        if (globaltimer_ns() - t0 > WAIT_LIMIT_NS) return false;
        __nanosleep(sleep_ns);
    }
}

// Whole-warp form: every lane waits; the result is the same in every lane.
__device__ __forceinline__ bool mbar_wait_bounded_warp(uint32_t bar, uint32_t parity, volatile int* abort) {
    const bool ok = mbar_wait_bounded(bar, parity, abort);
    return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---- tcgen05 (5th-generation tensor core, tensor memory) -----------------
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                 :: "r"(dst_smem), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;"
                 :: "r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Arrive once on `bar` when every tcgen05 operation issued so far by this
// thread has completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];"
                 :: "r"(bar) : "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, E4M3 x E4M3 -> F32 (kind::f8f6f4).
__device__ __forceinline__ void mma_f8f6f4(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                           uint32_t idesc, uint32_t accumulate) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}"
                 :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
                 : "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, F16/BF16 inputs -> F32 (kind::f16).
__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                        uint32_t idesc, uint32_t accumulate) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
                 :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
                 : "memory");
}

// CTA-pair form (M = 256 across the pair) of the 16-bit MMA.
__device__ __forceinline__ void mma_f16_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                             uint32_t idesc, uint32_t accumulate) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}"
                 :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
                 : "memory");
}

// 32 consecutive 32-bit columns of one TMEM lane per thread (lanes = the
// warp's 32-lane quarter).
__device__ __forceinline__ void tmem_ld_32x32b_x32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
          "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
          "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]),
          "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]),
          "=r"(r[30]), "=r"(r[31])
        : "r"(taddr) : "memory");
}
// 8 consecutive columns.
__device__ __forceinline__ void tmem_ld_32x32b_x8(uint32_t taddr, uint32_t (&r)[8]) {
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr) : "memory");
}
// 16 consecutive columns: the same, in half the registers.
__device__ __forceinline__ void tmem_ld_32x32b_x16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
          "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
          "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr) : "memory");
}
__device__ __forceinline__ void tmem_ld_wait() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}
// Stores of 16 consecutive 32-bit columns of one TMEM lane per thread
// (lanes = the warp's 32-lane quarter), and the wait for them.
__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
                 "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};"
                 :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]),
                    "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
                    "r"(v[15])
                 : "memory");
}
__device__ __forceinline__ void tmem_st_32x32b_x8(uint32_t taddr, const uint32_t (&v)[8]) {
    asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};"
                 :: "r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7])
                 : "memory");
}
__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor for a K-major operand tile stored in the
// 128-byte swizzle layout: rows of 128 bytes, 8-row atoms of 1024 bytes
// (stride-dimension byte offset), 16-byte chunks XOR-ed with the row index
// within the atom. `addr` is the byte address of the tile's first row plus
// the K offset (in bytes, < 128) of the sub-block the MMA reads; the atom
// base must be 1024-byte aligned.
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
    uint64_t d = 0;
    d |= (uint64_t)((addr & 0x3FFFFu) >> 4);          // start address
    d |= (uint64_t)1 << 16;                            // leading byte offset (unused)
    d |= (uint64_t)(1024u >> 4) << 32;                 // stride byte offset
    d |= (uint64_t)1 << 46;                            // descriptor version
    d |= (uint64_t)2 << 61;                            // 128-byte swizzle
    return d;
}

// Byte offset of logical 16-byte chunk `c` (0..7) of row `row` inside a
// 128-byte-swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128_offset(uint32_t row, uint32_t c) {
    return (row >> 3) * 1024u + (row & 7u) * 128u + ((c ^ (row & 7u)) << 4);
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t a, uint32_t b,
                                             uint32_t c, uint32_t d) {
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};"
                 :: "r"(addr), "r"(a), "r"(b), "r"(c), "r"(d) : "memory");
}

__device__ __forceinline__ uint4 ld_global_nc_v4(const void* p) {
    uint4 v;
    asm volatile("ld.global.nc.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
    return v;
}

__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t d;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(sel));
    return d;
}

// ---- clusters and CTA pairs ----------------------------------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// shared::cluster address of the variable at `addr` (a shared::cta address)
// in the CTA of the cluster with rank `rank`.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
    uint32_t d;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(addr), "r"(rank));
    return d;
}
// Arrive on an mbarrier given by its shared::cluster address (any CTA of
// the cluster), with release semantics at cluster scope.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];"
                 :: "r"(cluster_addr) : "memory");
}
// The same without release semantics: for a handoff that orders only
// tcgen05 accesses (completed by tcgen05.wait and ordered by
// tcgen05.fence::before_thread_sync), where no memory write of the arriving
// thread needs to be visible to the waiter.
__device__ __forceinline__ void mbar_arrive_cluster_relaxed(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];"
                 :: "r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
                 :: "r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;"
                 ::: "memory");
}
// 2-D TMA tile load global -> this CTA's shared memory, completion counted
// on `bar` (bytes).
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int x, int y,
                                            uint32_t bar) {
    asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
                 " [%0], [%1, {%2, %3}], [%4];"
                 :: "r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(bar) : "memory");
}
// 2-D TMA tile load into this CTA's shared memory whose completion is
// counted on an mbarrier of either CTA of the pair (shared::cluster
// address `bar`).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void* tmap, int x, int y,
                                                 uint32_t bar) {
    asm volatile("cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.cta_group::2"
                 " [%0], [%1, {%2, %3}], [%4];"
                 :: "r"(dst), "l"(tmap), "r"(x), "r"(y), "r"(bar) : "memory");
}
// Contiguous global -> shared bulk copy (16-byte aligned, size % 16 == 0),
// completion counted on `bar`.
__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 :: "r"(dst), "l"(src), "r"(bytes), "r"(bar) : "memory");
}
// 2-D TMA tile store shared -> global (bulk group of the calling thread).
__device__ __forceinline__ void tma_store_2d(const void* tmap, int x, int y, uint32_t src) {
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];"
                 :: "l"(tmap), "r"(x), "r"(y), "r"(src) : "memory");
}
__device__ __forceinline__ void bulk_commit() {
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}
// Wait until the calling thread's committed bulk stores have read their
// shared-memory sources.
__device__ __forceinline__ void bulk_wait_read0() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// Same, leaving at most the most recent group still reading.
__device__ __forceinline__ void bulk_wait_read1() {
    asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
// Wait until the calling thread's committed bulk stores are complete.
__device__ __forceinline__ void bulk_wait0() {
    asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;"
                 :: "r"(dst_smem), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;"
                 :: "r"(taddr), "r"(ncols) : "memory");
}
// D[tmem of both CTAs] (+)= A[smem, M rows split over the pair] *
// B[smem, N rows split over the pair]^T, E4M3 -> F32; issued by the leader.
__device__ __forceinline__ void mma_f8f6f4_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                                uint32_t idesc, uint32_t accumulate) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}"
                 :: "r"(d_tmem), "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
                 : "memory");
}
// Arrive once on the barrier at shared offset `bar` in every CTA of
// `cta_mask` when the issuing thread's tcgen05 operations have completed.
__device__ __forceinline__ void tc_commit_pair_multicast(uint32_t bar, uint16_t cta_mask) {
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
                 " [%0], %1;" :: "r"(bar), "h"(cta_mask) : "memory");
}

__device__ __forceinline__ uint4 ld_shared_v4(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

// Eight int4 codes (two's complement nibbles, code k in bits 4k..4k+3) to
// eight E4M3 bytes (byte k = code k). Every integer in [-8, 7] is exact in
// E4M3. Per four codes three byte-permutes do the work: one looks the code
// up in the table of non-negative values (a negative code's selector has its
// top bit set, which replicates the zero sign bit of the table byte: 0x00),
// one looks the low three bits up in the table of negative values (selector
// top bits flipped, so non-negative codes yield 0xFF), and one replicates
// each code's sign bit into a byte mask that picks between the two.
__device__ __forceinline__ void int4x8_to_e4m3x8(uint32_t x, uint32_t& lo, uint32_t& hi) {
    // codes 0..7: 0x00 0x38 0x40 0x44 | 0x48 0x4A 0x4C 0x4E
    constexpr uint32_t P0 = 0x44403800u, P1 = 0x4E4C4A48u;
    // codes -8..-1 by their low three bits: 0xD0 0xCE 0xCC 0xCA | 0xC8 0xC4 0xC0 0xB8
    constexpr uint32_t N0 = 0xCACCCED0u, N1 = 0xB8C0C4C8u;
    const uint32_t xs = x << 4;                 // low-nibble sign bits -> byte msb
    const uint32_t xn = x ^ 0x88888888u;
    const uint32_t xh = x >> 16, xnh = xn >> 16;
    // sign masks: byte k = 0xFF iff code k < 0 (sign of code 2j in xs byte j,
    // of code 2j+1 in x byte j)
    const uint32_t mlo = prmt(xs, x, 0xD9C8u);
    const uint32_t mhi = prmt(xs, x, 0xFBEAu);
    lo = prmt(P0, P1, x) | (prmt(N0, N1, xn) & mlo);
    hi = prmt(P0, P1, xh) | (prmt(N0, N1, xnh) & mhi);
}

}  // namespace starq
