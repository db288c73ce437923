// C ABI of libstarq.so (declared in include/starq.h): argument validation,
// error reporting, the device status word, and the composition of the
// kernels into sgat_linear.
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <initializer_list>

#include "common.cuh"
#include "attn.cuh"
#include "tac_calib.cuh"
#include "w8a8.cuh"
#include "asym.cuh"
#include "dense.cuh"

namespace starq {

// Status word written by kernels whose bounded waits run out.
__device__ unsigned g_status_word;

namespace {

thread_local char g_err[512] = "";

int fail(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char* where) {
    return fail(STARQ_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned(const void* p, size_t n) { return (reinterpret_cast<uintptr_t>(p) % n) == 0; }
bool pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }
bool dtype_ok(int t) { return t == STARQ_F16 || t == STARQ_BF16 || t == STARQ_F32; }

unsigned* status_ptr(int* err) {
    static DeviceCache<unsigned*> cache;
    unsigned* p = nullptr;
    const cudaError_t e = cache.get(&p, [](int, unsigned** v) {
        void* a = nullptr;
        const cudaError_t r = cudaGetSymbolAddress(&a, g_status_word);
        *v = static_cast<unsigned*>(a);
        return r;
    });
    if (e != cudaSuccess) { *err = cuda_fail(e, "status word address"); return nullptr; }
    *err = STARQ_OK;
    return p;
}

int check_transform(int K, int hb, int d_sh, int d_m, int d_u, const float* a_m, const float* a_u) {
    if (K < 16 || K % 16 != 0 || K > 20480)
        return fail(STARQ_ERR_SHAPE, "K=%d: need 16 <= K <= 20480 and K %% 16 == 0", K);
    if (!pow2(hb) || hb > 4096 || K % hb != 0)
        return fail(STARQ_ERR_SHAPE, "hb=%d: need a power of two <= 4096 dividing K=%d", hb, K);
    if (d_sh < 0 || d_m < 0 || d_u < 0 || (long)d_sh + d_m + d_u != K)
        return fail(STARQ_ERR_SHAPE, "gate layout (%d, %d, %d) must be >= 0 and sum to K=%d",
                    d_sh, d_m, d_u, K);
    if ((a_m && !aligned(a_m, 16)) || (a_u && !aligned(a_u, 16)))
        return fail(STARQ_ERR_ALIGN, "smoothing vectors must be 16-byte aligned");
    return STARQ_OK;
}

int check_tac(int L, int C, int g, const float* M, const float* d) {
    if (M == nullptr) return fail(STARQ_ERR_ARG, "TAC matrix M is NULL");
    if (!(g == 4 || g == 8 || g == 16 || g == 32 || g == 64 || g == 128))
        return fail(STARQ_ERR_SHAPE, "TAC block g=%d: supported 4, 8, 16, 32, 64, 128", g);
    if (C <= 0 || C % g != 0 || C % 8 != 0)
        return fail(STARQ_ERR_SHAPE, "TAC width C=%d must be a positive multiple of g=%d and 8", C, g);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    if (!aligned(M, 16) || (d && !aligned(d, 16)))
        return fail(STARQ_ERR_ALIGN, "TAC M and d must be 16-byte aligned");
    return STARQ_OK;
}

int check_tac_prepared(const void* Mp, int z_dtype, int g) {
    if (!Mp) return STARQ_OK;
    if ((z_dtype != STARQ_F16 && z_dtype != STARQ_BF16) || (g != 64 && g != 128))
        return fail(STARQ_ERR_ARG, "prepared TAC matrix: 16-bit Z and g = 64 or 128 only");
    if (!aligned(Mp, 16)) return fail(STARQ_ERR_ALIGN, "prepared TAC matrix must be 16-byte aligned");
    return STARQ_OK;
}

// The tac option of sgat_quantize_act and w4a4_gemm: parameters for a
// [L][C] tensor of element type dtype (its scratch buffer included).
int check_tac_option(const char* who, const starq_tac* t, int L, int C, int dtype) {
    int rc = check_tac(L, C, t->g, t->M, t->d);
    if (rc) return rc;
    if ((rc = check_tac_prepared(t->Mp, dtype, t->g))) return rc;
    if (L > 0 && !t->scratch) return fail(STARQ_ERR_ARG, "%s: tac->scratch is NULL", who);
    if (L > 0 && !aligned(t->scratch, 16)) return fail(STARQ_ERR_ALIGN, "%s: tac->scratch must be 16-byte aligned", who);
    return STARQ_OK;
}

int check_gemm(const uint8_t* Xq, const uint8_t* Xe, const float* s_a, const uint8_t* Wq, const uint8_t* We,
               const float* s_w, const float* bias, int L, int N, int K, void* Y, int y_dtype) {
    if ((!Wq && !We) || !s_w) return fail(STARQ_ERR_ARG, "w4a4_gemm: NULL Wq/We or s_w");
    if (L > 0 && !Wq && !Xe) return fail(STARQ_ERR_ARG, "w4a4_gemm: We without Xe needs Wq");
    if (L > 0 && ((!Xq && !Xe) || !s_a || !Y)) return fail(STARQ_ERR_ARG, "w4a4_gemm: NULL Xq/Xe, s_a or Y");
    if (!dtype_ok(y_dtype)) return fail(STARQ_ERR_ARG, "w4a4_gemm: unknown output dtype %d", y_dtype);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    if (N < 32 || N % 32 != 0) return fail(STARQ_ERR_SHAPE, "N=%d: need N >= 32, N %% 32 == 0", N);
    if (K < 128 || K % 128 != 0 || K > 65536)
        return fail(STARQ_ERR_SHAPE, "K=%d: need 128 <= K <= 65536 and K %% 128 == 0", K);
    if (L == 0) return STARQ_OK;  // nothing is read or written
    if (!aligned(Xq, 16) || !aligned(Xe, 16) || !aligned(Wq, 16) || !aligned(We, 16) || !aligned(Y, 16) ||
        !aligned(s_w, 16) || (bias && !aligned(bias, 16)) || !aligned(s_a, 4))
        return fail(STARQ_ERR_ALIGN, "w4a4_gemm: Xq, Xe, Wq, We, Y, s_w, bias must be 16-byte aligned");
    return STARQ_OK;
}

constexpr size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Operands that the kernels reach through TMA tensor maps must be device
// memory of the current device: a tensor map describes this GPU's own
// memory. Every non-null pointer is checked with cudaPointerGetAttributes,
// except while `stream` is capturing a CUDA graph (the eager calls before a
// capture are checked; a capture records the same pointers).
int check_local(const char* who, cudaStream_t stream, std::initializer_list<const void*> ptrs) {
    cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(stream, &cap) != cudaSuccess) {
        cudaGetLastError();
        cap = cudaStreamCaptureStatusNone;
    }
    if (cap != cudaStreamCaptureStatusNone) return STARQ_OK;
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    for (const void* p : ptrs) {
        if (p == nullptr) continue;
        cudaPointerAttributes at;
        e = cudaPointerGetAttributes(&at, p);
        if (e != cudaSuccess) {
            cudaGetLastError();
            return fail(STARQ_ERR_ARG, "%s: pointer %p is not CUDA memory", who, p);
        }
        if (at.type != cudaMemoryTypeDevice || at.device != dev)
            return fail(STARQ_ERR_ARG, "%s: pointer %p is not device memory of the current device %d "
                        "(memory type %d, device %d)", who, p, dev, (int)at.type, at.device);
    }
    return STARQ_OK;
}

// The dense-basis transform of `rows` rows into V (float16): the scaled
// rows fl16(fl32(x * a_s)) into Xs, then V = Xs P on the 16-bit GEMM
// (B operand Pt = P^T).
cudaError_t dense_transform(const void* X, int x_dtype, int rows, int K, const uint8_t* mask, const float* a_m,
                            const float* a_u, const void* Pt, __half* Xs, __half* V, unsigned* st, cudaStream_t s) {
    cudaError_t e = launch_scale_rows_f16(X, x_dtype, rows, K, mask, a_m, a_u, Xs, s);
    if (e != cudaSuccess) return e;
    GemmArgs g{nullptr, nullptr, nullptr, nullptr, nullptr, rows, K, K, V, STARQ_F16, nullptr, st,
               reinterpret_cast<const uint8_t*>(Xs), static_cast<const uint8_t*>(Pt)};
    return launch_fp16_gemm(g, s);
}

int check_dense(int K, const void* Pt) {
    if (!Pt) return fail(STARQ_ERR_ARG, "dense basis: NULL Pt");
    if (K < 128 || K % 128 != 0 || K > 16384)
        return fail(STARQ_ERR_SHAPE, "dense basis: K=%d: need 128 <= K <= 16384, K %% 128 == 0", K);
    if (!aligned(Pt, 16)) return fail(STARQ_ERR_ALIGN, "dense basis: Pt must be 16-byte aligned");
    return STARQ_OK;
}

int check_w8a8(const uint8_t* Xe, const float* s_a, const uint8_t* We, const float* s_w, const float* bias, int L,
               int N, int K, void* Y, int y_dtype) {
    if (!We || !s_w) return fail(STARQ_ERR_ARG, "w8a8_gemm: NULL We or s_w");
    if (L > 0 && (!Xe || !s_a || !Y)) return fail(STARQ_ERR_ARG, "w8a8_gemm: NULL Xe, s_a or Y");
    if (!dtype_ok(y_dtype)) return fail(STARQ_ERR_ARG, "w8a8_gemm: unknown output dtype %d", y_dtype);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    if (N < 128 || N % 128 != 0) return fail(STARQ_ERR_SHAPE, "w8a8_gemm: N=%d: need N >= 128, N %% 128 == 0", N);
    if (K < 128 || K % 128 != 0 || K > 65536)
        return fail(STARQ_ERR_SHAPE, "w8a8_gemm: K=%d: need 128 <= K <= 65536 and K %% 128 == 0", K);
    if (L == 0) return STARQ_OK;
    if (!aligned(Xe, 16) || !aligned(We, 16) || !aligned(Y, 16) || !aligned(s_w, 16) || (bias && !aligned(bias, 16)) ||
        !aligned(s_a, 4))
        return fail(STARQ_ERR_ALIGN, "w8a8_gemm: Xe, We, Y, s_w, bias must be 16-byte aligned");
    return STARQ_OK;
}

}  // namespace

int report_error(int code, const char* msg) { return fail(code, "%s", msg); }

namespace {
// Failure-detection self-test: one thread waits on an mbarrier that nothing
// ever arrives on, through the same bounded wait as every pipeline wait of
// the library (with a short limit), gives up, records STATUS_TIMEOUT_TEST in
// the status word and returns. Nothing faults and the context stays usable.
__global__ void selftest_wait_timeout_kernel(unsigned* status, unsigned long long limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort;
    if (threadIdx.x == 0) {
        abort = 0;
        mbar_init(smem_addr(&bar), 1);       // expects one arrival, which never comes
        mbar_fence_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !mbar_wait_limit(smem_addr(&bar), 0, &abort, limit_ns))
        atomicOr(status, STATUS_TIMEOUT_TEST);
}
}  // namespace

int num_sms() {
    static DeviceCache<int> cache;
    int n = 1;
    if (cache.get(&n, [](int dev, int* v) {
            int c = 0;
            const cudaError_t r = cudaDeviceGetAttribute(&c, cudaDevAttrMultiProcessorCount, dev);
            *v = c > 0 ? c : 1;
            return r;
        }) != cudaSuccess)
        return 1;
    return n;
}

PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
    static const PFN_cuTensorMapEncodeTiled_v12000 fn = []() -> PFN_cuTensorMapEncodeTiled_v12000 {
        cudaDriverEntryPointQueryResult q;
        void* f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
                cudaSuccess || q != cudaDriverEntryPointSuccess)
            return nullptr;
        return reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    }();
    return fn;
}

}  // namespace starq

using namespace starq;

extern "C" {

int starq_version(void) { return 100; }

int starq_last_gemm_tile(void) { return last_gemm_tile(); }

const char* starq_last_error(void) { return g_err; }

int starq_check_status(void* stream) {
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    unsigned v = 0, zero = 0;
    e = cudaMemcpyFromSymbol(&v, g_status_word, sizeof(v));
    if (e != cudaSuccess) return cuda_fail(e, "read status word");
    if (v != 0) {
        e = cudaMemcpyToSymbol(g_status_word, &zero, sizeof(zero));
        if (e != cudaSuccess) return cuda_fail(e, "clear status word");
        return fail(STARQ_ERR_TIMEOUT, "a kernel gave up a bounded wait (status bits 0x%x)", v);
    }
    return STARQ_OK;
}

int starq_selftest_wait_timeout(unsigned limit_us, void* stream) {
    if (limit_us < 1 || limit_us > 100000)
        return fail(STARQ_ERR_ARG, "starq_selftest_wait_timeout: limit_us=%u outside [1, 100000]", limit_us);
    int rc = STARQ_OK;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    selftest_wait_timeout_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(st, 1000ull * limit_us);
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "starq_selftest_wait_timeout launch");
    return STARQ_OK;
}

int glue_add_rmsnorm(const void* X, const void* R, int dtype, int L, int K, const float* w, float eps, void* h_out,
                     void* Y, void* stream) {
    if (dtype != STARQ_F16 && dtype != STARQ_BF16) return fail(STARQ_ERR_ARG, "glue_add_rmsnorm: dtype must be F16 or BF16");
    if (L < 0 || K < 8 || K % 8 != 0 || K > 20480)
        return fail(STARQ_ERR_SHAPE, "glue_add_rmsnorm: L=%d, K=%d: need L >= 0, 8 <= K <= 20480, K %% 8 == 0", L, K);
    if (L == 0) return STARQ_OK;
    if (!X || (Y && !w) || (!Y && !h_out)) return fail(STARQ_ERR_ARG, "glue_add_rmsnorm: NULL X, w, or no output");
    if (h_out && !R) return fail(STARQ_ERR_ARG, "glue_add_rmsnorm: h_out needs the residual R");
    if (!(eps >= 0.f)) return fail(STARQ_ERR_ARG, "glue_add_rmsnorm: eps must be >= 0");
    if (!aligned(X, 16) || (R && !aligned(R, 16)) || (w && !aligned(w, 16)) || (h_out && !aligned(h_out, 16)) ||
        (Y && !aligned(Y, 16)))
        return fail(STARQ_ERR_ALIGN, "glue_add_rmsnorm: X, R, w, h_out, Y must be 16-byte aligned");
    const cudaError_t e = launch_add_rmsnorm(X, R, dtype, L, K, w, eps, h_out, Y, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "glue_add_rmsnorm launch");
    return STARQ_OK;
}

int glue_rope(void* QK, int dtype, int L, int ld, int heads, const int32_t* pos, double theta, void* stream) {
    if (dtype != STARQ_F16 && dtype != STARQ_BF16) return fail(STARQ_ERR_ARG, "glue_rope: dtype must be F16 or BF16");
    if (L < 0 || heads < 1 || ld < 128 * heads)
        return fail(STARQ_ERR_SHAPE, "glue_rope: L=%d, heads=%d, ld=%d: need ld >= 128 heads", L, heads, ld);
    if (!(theta > 1.0)) return fail(STARQ_ERR_ARG, "glue_rope: theta must be > 1");
    if (L == 0) return STARQ_OK;
    if (!QK || !pos) return fail(STARQ_ERR_ARG, "glue_rope: NULL QK or pos");
    const cudaError_t e = launch_rope(QK, dtype, L, ld, heads, pos, theta, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "glue_rope launch");
    return STARQ_OK;
}

int starq_probe_mma(int kind, int iters, unsigned long long* cycles, int* errors, int* ctas, double* macs_per_cta,
                    void* stream) {
    if (kind < 0 || kind > 4) return fail(STARQ_ERR_ARG, "starq_probe_mma: kind=%d outside 0..4", kind);
    if (iters < 1 || iters > 2048) return fail(STARQ_ERR_ARG, "starq_probe_mma: iters=%d outside 1..2048", iters);
    if (!cycles || !errors || !ctas || !macs_per_cta) return fail(STARQ_ERR_ARG, "starq_probe_mma: NULL pointer");
    int rc = check_local("starq_probe_mma", static_cast<cudaStream_t>(stream), {cycles, errors});
    if (rc) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    const cudaError_t e = launch_probe_mma(kind, iters, cycles, errors, st, ctas, macs_per_cta,
                                           static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "starq_probe_mma launch");
    return STARQ_OK;
}

int sgat_quantize_act(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                      const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                      const starq_tac* tac, int bits, uint8_t* Xq, float* s_a, uint8_t* Xe, float* v_dbg,
                      void* stream) {
    if (L > 0 && (!X || (!Xq && !Xe) || !s_a)) return fail(STARQ_ERR_ARG, "sgat_quantize_act: NULL X, s_a, or both Xq and Xe");
    if (!dtype_ok(x_dtype)) return fail(STARQ_ERR_ARG, "sgat_quantize_act: unknown dtype %d", x_dtype);
    if (bits != 4 && bits != 8) return fail(STARQ_ERR_BITS, "bits=%d: the GPU path implements 4- and 8-bit codes", bits);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    int rc = check_transform(K, hb, d_sh, d_m, d_u, a_m, a_u);
    if (rc) return rc;
    if (L == 0) return STARQ_OK;
    if (!aligned(X, 16) || !aligned(Xq, 8) || (v_dbg && !aligned(v_dbg, 16)) || (Xe && !aligned(Xe, 16)))
        return fail(STARQ_ERR_ALIGN, "sgat_quantize_act: X (16 B), Xq (8 B), Xe (16 B), v_dbg (16 B) alignment");
    const void* src = X;
    cudaError_t e;
    if (tac) {                       // TAC(X) into the scratch buffer, then quantise that
        if ((rc = check_tac_option("sgat_quantize_act", tac, L, K, x_dtype))) return rc;
        if ((rc = check_local("sgat_quantize_act", static_cast<cudaStream_t>(stream), {X, tac->scratch}))) return rc;
        unsigned* st = status_ptr(&rc);
        if (!st) return rc;
        TacArgs t{X, x_dtype, L, K, tac->g, tac->M, tac->d, tac->scratch, x_dtype, st, tac->Mp};
        if ((e = launch_tac(t, static_cast<cudaStream_t>(stream))) != cudaSuccess)
            return cuda_fail(e, "sgat_quantize_act: TAC launch");
        src = tac->scratch;
    }
    QuantArgs a{src, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, bits == 8 ? 127 : 7, 1.f, Xq, s_a, v_dbg, Xe};
    e = launch_sgat_quant(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "sgat_quantize_act launch");
    return STARQ_OK;
}

int sgat_quantize_act_grouped(const starq_quant_io* p0, const starq_quant_io* p1, int x_dtype, int L, int K,
                              int hb, int bits, void* stream) {
    if (!p0 || !p1) return fail(STARQ_ERR_ARG, "sgat_quantize_act_grouped: NULL problem");
    if (!dtype_ok(x_dtype)) return fail(STARQ_ERR_ARG, "sgat_quantize_act_grouped: unknown dtype %d", x_dtype);
    if (bits != 4 && bits != 8) return fail(STARQ_ERR_BITS, "bits=%d: the GPU path implements 4- and 8-bit codes", bits);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    for (const starq_quant_io* p : {p0, p1}) {
        if (L > 0 && (!p->X || (!p->Xq && !p->Xe) || !p->s_a))
            return fail(STARQ_ERR_ARG, "sgat_quantize_act_grouped: NULL X, s_a, or both Xq and Xe");
        int rc = check_transform(K, hb, p->d_sh, p->d_m, p->d_u, p->a_m, p->a_u);
        if (rc) return rc;
        if (L > 0 && (!aligned(p->X, 16) || !aligned(p->Xq, 8) || (p->Xe && !aligned(p->Xe, 16))))
            return fail(STARQ_ERR_ALIGN, "sgat_quantize_act_grouped: X (16 B), Xq (8 B), Xe (16 B) alignment");
    }
    if (L == 0) return STARQ_OK;
    const int qmax = bits == 8 ? 127 : 7;
    QuantArgs a{p0->X, x_dtype, L, K, p0->mask, p0->a_m, p0->a_u, hb, p0->d_sh, p0->d_m, p0->d_u, qmax, 1.f,
                p0->Xq, p0->s_a, nullptr, p0->Xe};
    QuantArgs b{p1->X, x_dtype, L, K, p1->mask, p1->a_m, p1->a_u, hb, p1->d_sh, p1->d_m, p1->d_u, qmax, 1.f,
                p1->Xq, p1->s_a, nullptr, p1->Xe};
    a.independent = p0->independent != 0;
    b.independent = p1->independent != 0;
    const cudaError_t e = launch_sgat_quant_grouped(a, b, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "sgat_quantize_act_grouped launch");
    return STARQ_OK;
}

int sgat_prepare_weight(const void* W, int w_dtype, int N, int K, const float* inv_a_w, int hb,
                        int bits, uint8_t* Wq, float* s_w, void* stream) {
    if (N > 0 && (!W || !Wq || !s_w)) return fail(STARQ_ERR_ARG, "sgat_prepare_weight: NULL W, Wq or s_w");
    if (!dtype_ok(w_dtype)) return fail(STARQ_ERR_ARG, "sgat_prepare_weight: unknown dtype %d", w_dtype);
    if (bits != 4 && bits != 8) return fail(STARQ_ERR_BITS, "bits=%d: the GPU path implements 4- and 8-bit codes", bits);
    if (N < 0) return fail(STARQ_ERR_SHAPE, "N=%d < 0", N);
    int rc = check_transform(K, hb, K, 0, 0, nullptr, inv_a_w);
    if (rc) return rc;
    if (N == 0) return STARQ_OK;
    if (!aligned(W, 16) || !aligned(Wq, 8))
        return fail(STARQ_ERR_ALIGN, "sgat_prepare_weight: W (16 B), Wq (8 B) alignment");
    QuantArgs a{W, w_dtype, N, K, nullptr, nullptr, inv_a_w, hb, K, 0, 0, bits == 8 ? 127 : 7, 1.f / (float)hb,
                Wq, s_w, nullptr};
    cudaError_t e = launch_sgat_quant(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "sgat_prepare_weight launch");
    return STARQ_OK;
}

int w4_unpack_e4m3(const uint8_t* Wq, int N, int K, uint8_t* We, void* stream) {
    if (N > 0 && (!Wq || !We)) return fail(STARQ_ERR_ARG, "w4_unpack_e4m3: NULL Wq or We");
    if (N < 0 || K < 32 || K % 32 != 0) return fail(STARQ_ERR_SHAPE, "w4_unpack_e4m3: N=%d K=%d (K %% 32 == 0)", N, K);
    if (N == 0) return STARQ_OK;
    if (!aligned(Wq, 16) || !aligned(We, 16)) return fail(STARQ_ERR_ALIGN, "w4_unpack_e4m3: Wq, We alignment");
    cudaError_t e = launch_unpack_e4m3(Wq, We, (size_t)N, K, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w4_unpack_e4m3 launch");
    return STARQ_OK;
}

int w4a4_gemm(const uint8_t* Xq, const uint8_t* Xe, const float* s_a, const uint8_t* Wq, const uint8_t* We,
              const float* s_w, const float* bias, int L, int N, int K, void* Y, int y_dtype,
              const starq_tac* out_tac, int32_t* acc_dbg, void* stream) {
    int rc = check_gemm(Xq, Xe, s_a, Wq, We, s_w, bias, L, N, K, Y, y_dtype);
    if (rc) return rc;
    if (acc_dbg && !aligned(acc_dbg, 16)) return fail(STARQ_ERR_ALIGN, "acc_dbg must be 16-byte aligned");
    if (out_tac && (rc = check_tac_option("w4a4_gemm", out_tac, L, N, y_dtype))) return rc;
    void* dst = out_tac ? out_tac->scratch : Y;    // the dequantised output before TAC
    if (L > 0 && (rc = check_local("w4a4_gemm", static_cast<cudaStream_t>(stream),
                                   {Xe, Xe ? We : nullptr, Xe ? Wq : nullptr, Y, dst})))
        return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    GemmArgs a{Xq, s_a, Wq, s_w, bias, L, N, K, dst, y_dtype, acc_dbg, st, Xe, Xe ? We : nullptr};
    cudaError_t e = launch_w4a4_gemm(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w4a4_gemm launch");
    if (out_tac && L > 0) {
        TacArgs t{dst, y_dtype, L, N, out_tac->g, out_tac->M, out_tac->d, Y, y_dtype, st, out_tac->Mp};
        if ((e = launch_tac(t, static_cast<cudaStream_t>(stream))) != cudaSuccess)
            return cuda_fail(e, "w4a4_gemm: TAC launch");
    }
    return STARQ_OK;
}

int w4a4_gemm_grouped(const uint8_t* Xe0, const float* s_a0, const uint8_t* We0, const float* s_w0,
                      const float* bias0, int N0, void* Y0, const uint8_t* Xe1, const float* s_a1,
                      const uint8_t* We1, const float* s_w1, const float* bias1, int N1, void* Y1, int L, int K,
                      int y_dtype, int32_t* acc_dbg0, int32_t* acc_dbg1, int flags, void* stream) {
    if (!We0 || !We1) return fail(STARQ_ERR_ARG, "w4a4_gemm_grouped: NULL We0 or We1");
    if (flags & ~STARQ_GEMM_WEIGHTS_READY) return fail(STARQ_ERR_ARG, "w4a4_gemm_grouped: unknown flags %d", flags);
    if (L > 0 && (!Xe0 || !Xe1)) return fail(STARQ_ERR_ARG, "w4a4_gemm_grouped: NULL Xe0 or Xe1");
    int rc = check_gemm(nullptr, Xe0, s_a0, nullptr, We0, s_w0, bias0, L, N0, K, Y0, y_dtype);
    if (rc) return rc;
    if ((rc = check_gemm(nullptr, Xe1, s_a1, nullptr, We1, s_w1, bias1, L, N1, K, Y1, y_dtype))) return rc;
    if ((acc_dbg0 && !aligned(acc_dbg0, 16)) || (acc_dbg1 && !aligned(acc_dbg1, 16)))
        return fail(STARQ_ERR_ALIGN, "w4a4_gemm_grouped: acc_dbg must be 16-byte aligned");
    if (L == 0) return STARQ_OK;
    if ((rc = check_local("w4a4_gemm_grouped", static_cast<cudaStream_t>(stream), {Xe0, We0, Y0, Xe1, We1, Y1})))
        return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    GemmArgs a{nullptr, s_a0, nullptr, s_w0, bias0, L, N0, K, Y0, y_dtype, acc_dbg0, st, Xe0, We0};
    GemmArgs b{nullptr, s_a1, nullptr, s_w1, bias1, L, N1, K, Y1, y_dtype, acc_dbg1, st, Xe1, We1};
    a.weights_ready = b.weights_ready = (flags & STARQ_GEMM_WEIGHTS_READY) ? 1 : 0;
    cudaError_t e = launch_w4a4_gemm_grouped(a, b, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w4a4_gemm_grouped launch");
    return STARQ_OK;
}

int starq_set_gemm_pair_limit(int pairs) {
    if (pairs < 0) return fail(STARQ_ERR_ARG, "starq_set_gemm_pair_limit: pairs=%d < 0", pairs);
    return set_gemm_pair_limit(pairs);
}

int w4a4_gemm_mma_sync(const uint8_t* Xq, const float* s_a, const uint8_t* Wq, const float* s_w,
                       const float* bias, int L, int N, int K, void* Y, int y_dtype, int32_t* acc_dbg,
                       void* stream) {
    if (L > 0 && (!Xq || !s_a || !Y)) return fail(STARQ_ERR_ARG, "w4a4_gemm_mma_sync: NULL Xq, s_a or Y");
    if (!Wq || !s_w) return fail(STARQ_ERR_ARG, "w4a4_gemm_mma_sync: NULL Wq or s_w");
    if (!dtype_ok(y_dtype)) return fail(STARQ_ERR_ARG, "w4a4_gemm_mma_sync: unknown output dtype %d", y_dtype);
    if (L < 0 || N < 1 || K < 128 || K % 128 != 0 || K > 65536)
        return fail(STARQ_ERR_SHAPE, "w4a4_gemm_mma_sync: L=%d N=%d K=%d (N >= 1, K %% 128 == 0, 128 <= K <= 65536)",
                    L, N, K);
    if (L == 0) return STARQ_OK;
    if (!aligned(Xq, 16) || !aligned(Wq, 16))
        return fail(STARQ_ERR_ALIGN, "w4a4_gemm_mma_sync: Xq and Wq must be 16-byte aligned");
    int rc = check_local("w4a4_gemm_mma_sync", static_cast<cudaStream_t>(stream), {Xq, Wq, Y});
    if (rc) return rc;
    GemmArgs a{Xq, s_a, Wq, s_w, bias, L, N, K, Y, y_dtype, acc_dbg, nullptr};
    cudaError_t e = launch_w4a4_gemm_mmasync(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w4a4_gemm_mma_sync launch");
    return STARQ_OK;
}

int sgat_quantize_act_asym(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                           const float* a_u, int hb, int d_sh, int d_m, int d_u, uint8_t* Xq, float* s_a,
                           int32_t* z_a, uint8_t* Xe, void* stream) {
    if (L > 0 && (!X || !Xq || !s_a || !z_a)) return fail(STARQ_ERR_ARG, "sgat_quantize_act_asym: NULL X, Xq, s_a or z_a");
    if (!dtype_ok(x_dtype)) return fail(STARQ_ERR_ARG, "sgat_quantize_act_asym: unknown dtype %d", x_dtype);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    int rc = check_transform(K, hb, d_sh, d_m, d_u, a_m, a_u);
    if (rc) return rc;
    if (Xe && (K % 128 != 0 || K > ASYM_MAX_K))
        return fail(STARQ_ERR_SHAPE, "sgat_quantize_act_asym: K=%d: Xe needs K %% 128 == 0 and K <= %d", K, ASYM_MAX_K);
    if (L == 0) return STARQ_OK;
    if (!aligned(X, 16) || !aligned(Xq, 8) || !aligned(z_a, 4) || (Xe && !aligned(Xe, 16)))
        return fail(STARQ_ERR_ALIGN, "sgat_quantize_act_asym: X (16 B), Xq (8 B), z_a (4 B), Xe (16 B) alignment");
    QuantArgs a{X, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, 15, 1.f, Xq, s_a, nullptr, Xe};
    a.asym = 1;
    a.z = z_a;
    cudaError_t e = launch_sgat_quant(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "sgat_quantize_act_asym launch");
    return STARQ_OK;
}

int w4_zero_point_columns(const uint8_t* Wq, int N, int K, uint8_t* We, void* stream) {
    if (N > 0 && (!Wq || !We)) return fail(STARQ_ERR_ARG, "w4_zero_point_columns: NULL Wq or We");
    if (N < 0 || K < 128 || K % 128 != 0 || K > ASYM_MAX_K)
        return fail(STARQ_ERR_SHAPE, "w4_zero_point_columns: N=%d K=%d (K %% 128 == 0, K <= %d)", N, K, ASYM_MAX_K);
    if (N == 0) return STARQ_OK;
    if (!aligned(Wq, 16) || !aligned(We, 16)) return fail(STARQ_ERR_ALIGN, "w4_zero_point_columns: Wq, We alignment");
    cudaError_t e = launch_zero_point_columns(Wq, We, N, K, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w4_zero_point_columns launch");
    return STARQ_OK;
}

size_t sgat_linear_asym_workspace_size(int L, int K) {
    if (L < 0 || K < 0) return 0;
    return align256((size_t)L * K / 2) + 2 * align256((size_t)L * 4) + align256((size_t)L * (K + 128));
}

int sgat_linear_asym(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                     const float* a_u, int hb, int d_sh, int d_m, int d_u, const uint8_t* We, const float* s_w,
                     const float* bias, int N, void* Y, int y_dtype, void* workspace, size_t workspace_bytes,
                     void* stream) {
    if (!We || !s_w) return fail(STARQ_ERR_ARG, "sgat_linear_asym: NULL We or s_w");
    if (L > 0 && (!X || !Y || !workspace)) return fail(STARQ_ERR_ARG, "sgat_linear_asym: NULL X, Y or workspace");
    if (!dtype_ok(x_dtype) || !dtype_ok(y_dtype)) return fail(STARQ_ERR_ARG, "sgat_linear_asym: unknown dtype");
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    int rc = check_transform(K, hb, d_sh, d_m, d_u, a_m, a_u);
    if (rc) return rc;
    if (K % 128 != 0 || K > ASYM_MAX_K)
        return fail(STARQ_ERR_SHAPE, "sgat_linear_asym: K=%d: need K %% 128 == 0 and K <= %d", K, ASYM_MAX_K);
    if (L == 0) return STARQ_OK;
    const size_t need = sgat_linear_asym_workspace_size(L, K);
    if (workspace_bytes < need) return fail(STARQ_ERR_SHAPE, "workspace %zu bytes < %zu needed", workspace_bytes, need);
    if (!aligned(workspace, 256) || !aligned(X, 16)) return fail(STARQ_ERR_ALIGN, "sgat_linear_asym alignment");
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    uint8_t* Xq = ws;
    float* s_a = reinterpret_cast<float*>(ws + align256((size_t)L * K / 2));
    int32_t* z_a = reinterpret_cast<int32_t*>(ws + align256((size_t)L * K / 2) + align256((size_t)L * 4));
    uint8_t* Xe = ws + align256((size_t)L * K / 2) + 2 * align256((size_t)L * 4);
    const int K2 = K + 128;                       // the augmented contraction
    rc = check_gemm(nullptr, Xe, s_a, nullptr, We, s_w, bias, L, N, K2, Y, y_dtype);
    if (rc) return rc;
    if ((rc = check_local("sgat_linear_asym", static_cast<cudaStream_t>(stream), {workspace, We, Y}))) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    QuantArgs q{X, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, 15, 1.f, Xq, s_a, nullptr, Xe};
    q.asym = 1;
    q.z = z_a;
    cudaError_t e;
    if ((e = launch_sgat_quant(q, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear_asym: quant launch");
    GemmArgs g{nullptr, s_a, nullptr, s_w, bias, L, N, K2, Y, y_dtype, nullptr, st, Xe, We};
    g.weights_ready = 1;
    if ((e = launch_w4a4_gemm(g, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear_asym: gemm launch");
    return STARQ_OK;
}

size_t sgat_dense_workspace_size(int rows, int K) {
    if (rows < 0 || K < 0) return 0;
    return 2 * align256((size_t)rows * K * 2);
}

int sgat_quantize_act_dense(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                            const float* a_u, const void* Pt, int d_sh, int d_m, int d_u, uint8_t* Xq, float* s_a,
                            uint8_t* Xe, void* workspace, size_t workspace_bytes, void* stream) {
    if (L > 0 && (!X || !Xq || !s_a || !workspace)) return fail(STARQ_ERR_ARG, "sgat_quantize_act_dense: NULL argument");
    if (!dtype_ok(x_dtype)) return fail(STARQ_ERR_ARG, "sgat_quantize_act_dense: unknown dtype %d", x_dtype);
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    int rc = check_dense(K, Pt);
    if (rc) return rc;
    if ((rc = check_transform(K, 1, d_sh, d_m, d_u, a_m, a_u))) return rc;
    if (L == 0) return STARQ_OK;
    if (workspace_bytes < sgat_dense_workspace_size(L, K))
        return fail(STARQ_ERR_SHAPE, "workspace %zu bytes < %zu", workspace_bytes, sgat_dense_workspace_size(L, K));
    if (!aligned(X, 16) || !aligned(Xq, 8) || (Xe && !aligned(Xe, 16)) || !aligned(workspace, 256))
        return fail(STARQ_ERR_ALIGN, "sgat_quantize_act_dense: X, Xe (16 B), Xq (8 B), workspace (256 B) alignment");
    if ((rc = check_local("sgat_quantize_act_dense", static_cast<cudaStream_t>(stream), {workspace, Pt}))) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    __half* Xs = static_cast<__half*>(workspace);
    __half* V = reinterpret_cast<__half*>(static_cast<uint8_t*>(workspace) + align256((size_t)L * K * 2));
    cudaError_t e = dense_transform(X, x_dtype, L, K, mask, a_m, a_u, Pt, Xs, V, st, s);
    if (e != cudaSuccess) return cuda_fail(e, "sgat_quantize_act_dense: transform launch");
    QuantArgs q{V, STARQ_F16, L, K, mask, nullptr, nullptr, 1, d_sh, d_m, d_u, 7, 1.f, Xq, s_a, nullptr, Xe};
    if ((e = launch_sgat_quant(q, s)) != cudaSuccess) return cuda_fail(e, "sgat_quantize_act_dense: quant launch");
    return STARQ_OK;
}

int sgat_prepare_weight_dense(const void* W, int w_dtype, int N, int K, const float* inv_a_w, const void* Pt,
                              uint8_t* Wq, float* s_w, void* workspace, size_t workspace_bytes, void* stream) {
    if (N > 0 && (!W || !Wq || !s_w || !workspace)) return fail(STARQ_ERR_ARG, "sgat_prepare_weight_dense: NULL argument");
    if (!dtype_ok(w_dtype)) return fail(STARQ_ERR_ARG, "sgat_prepare_weight_dense: unknown dtype %d", w_dtype);
    if (N < 0) return fail(STARQ_ERR_SHAPE, "N=%d < 0", N);
    int rc = check_dense(K, Pt);
    if (rc) return rc;
    if ((rc = check_transform(K, 1, K, 0, 0, nullptr, inv_a_w))) return rc;
    if (N == 0) return STARQ_OK;
    if (workspace_bytes < sgat_dense_workspace_size(N, K))
        return fail(STARQ_ERR_SHAPE, "workspace %zu bytes < %zu", workspace_bytes, sgat_dense_workspace_size(N, K));
    if (!aligned(W, 16) || !aligned(Wq, 8) || !aligned(workspace, 256))
        return fail(STARQ_ERR_ALIGN, "sgat_prepare_weight_dense: W (16 B), Wq (8 B), workspace (256 B) alignment");
    if ((rc = check_local("sgat_prepare_weight_dense", static_cast<cudaStream_t>(stream), {workspace, Pt}))) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    __half* Ws = static_cast<__half*>(workspace);
    __half* Wf = reinterpret_cast<__half*>(static_cast<uint8_t*>(workspace) + align256((size_t)N * K * 2));
    cudaError_t e = dense_transform(W, w_dtype, N, K, nullptr, nullptr, inv_a_w, Pt, Ws, Wf, st, s);
    if (e != cudaSuccess) return cuda_fail(e, "sgat_prepare_weight_dense: transform launch");
    QuantArgs q{Wf, STARQ_F16, N, K, nullptr, nullptr, nullptr, 1, K, 0, 0, 7, 1.f, Wq, s_w, nullptr};
    if ((e = launch_sgat_quant(q, s)) != cudaSuccess) return cuda_fail(e, "sgat_prepare_weight_dense: quant launch");
    return STARQ_OK;
}

size_t sgat_linear_dense_workspace_size(int L, int K) {
    if (L < 0 || K < 0) return 0;
    return sgat_dense_workspace_size(L, K) + align256((size_t)L * K / 2) + align256((size_t)L * 4) +
           align256((size_t)L * K);
}

int sgat_linear_dense(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                      const float* a_u, const void* Pt, int d_sh, int d_m, int d_u, const uint8_t* Wq,
                      const uint8_t* We, const float* s_w, const float* bias, int N, void* Y, int y_dtype,
                      void* workspace, size_t workspace_bytes, void* stream) {
    if (L > 0 && (!X || !Y || !workspace)) return fail(STARQ_ERR_ARG, "sgat_linear_dense: NULL X, Y or workspace");
    if (!dtype_ok(x_dtype) || !dtype_ok(y_dtype)) return fail(STARQ_ERR_ARG, "sgat_linear_dense: unknown dtype");
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    int rc = check_dense(K, Pt);
    if (rc) return rc;
    if ((rc = check_transform(K, 1, d_sh, d_m, d_u, a_m, a_u))) return rc;
    if (L == 0) return STARQ_OK;
    const size_t need = sgat_linear_dense_workspace_size(L, K);
    if (workspace_bytes < need) return fail(STARQ_ERR_SHAPE, "workspace %zu bytes < %zu needed", workspace_bytes, need);
    if (!aligned(workspace, 256) || !aligned(X, 16)) return fail(STARQ_ERR_ALIGN, "sgat_linear_dense alignment");
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    __half* Xs = reinterpret_cast<__half*>(ws);
    __half* V = reinterpret_cast<__half*>(ws + align256((size_t)L * K * 2));
    uint8_t* Xq = ws + sgat_dense_workspace_size(L, K);
    float* s_a = reinterpret_cast<float*>(Xq + align256((size_t)L * K / 2));
    uint8_t* Xe = Xq + align256((size_t)L * K / 2) + align256((size_t)L * 4);
    if ((rc = check_gemm(Xq, Xe, s_a, Wq, We, s_w, bias, L, N, K, Y, y_dtype))) return rc;
    if ((rc = check_local("sgat_linear_dense", static_cast<cudaStream_t>(stream), {workspace, Pt, Wq, We, Y}))) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = dense_transform(X, x_dtype, L, K, mask, a_m, a_u, Pt, Xs, V, st, s);
    if (e != cudaSuccess) return cuda_fail(e, "sgat_linear_dense: transform launch");
    QuantArgs q{V, STARQ_F16, L, K, mask, nullptr, nullptr, 1, d_sh, d_m, d_u, 7, 1.f, nullptr, s_a, nullptr, Xe};
    if ((e = launch_sgat_quant(q, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear_dense: quant launch");
    GemmArgs g{nullptr, s_a, Wq, s_w, bias, L, N, K, Y, y_dtype, nullptr, st, Xe, We};   // Xe: no packed codes read
    g.weights_ready = 1;
    if ((e = launch_w4a4_gemm(g, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear_dense: gemm launch");
    return STARQ_OK;
}

int w8_codes_f16(const uint8_t* Wq, int N, int K, uint8_t* We, void* stream) {
    if (N > 0 && (!Wq || !We)) return fail(STARQ_ERR_ARG, "w8_codes_f16: NULL Wq or We");
    if (N < 0 || K < 128 || K % 128 != 0) return fail(STARQ_ERR_SHAPE, "w8_codes_f16: N=%d K=%d (K %% 128 == 0)", N, K);
    if (N == 0) return STARQ_OK;
    if (!aligned(Wq, 16) || !aligned(We, 16)) return fail(STARQ_ERR_ALIGN, "w8_codes_f16: Wq, We alignment");
    cudaError_t e = launch_w8_codes_f16(Wq, We, (size_t)N, K, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w8_codes_f16 launch");
    return STARQ_OK;
}

int w8a8_gemm(const uint8_t* Xe, const float* s_a, const uint8_t* We, const float* s_w, const float* bias, int L,
              int N, int K, void* Y, int y_dtype, int32_t* acc_dbg, void* stream) {
    int rc = check_w8a8(Xe, s_a, We, s_w, bias, L, N, K, Y, y_dtype);
    if (rc) return rc;
    if (L == 0) return STARQ_OK;
    if (acc_dbg && !aligned(acc_dbg, 16)) return fail(STARQ_ERR_ALIGN, "acc_dbg must be 16-byte aligned");
    if ((rc = check_local("w8a8_gemm", static_cast<cudaStream_t>(stream), {Xe, We}))) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    GemmArgs a{nullptr, s_a, nullptr, s_w, bias, L, N, K, Y, y_dtype, acc_dbg, st, Xe, We};
    cudaError_t e = launch_w8a8_gemm(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "w8a8_gemm launch");
    return STARQ_OK;
}

int fp16_gemm_ref(const void* A, const void* B, int dtype, int M, int N, int K, void* C, void* stream) {
    if (M > 0 && (!A || !B || !C)) return fail(STARQ_ERR_ARG, "fp16_gemm_ref: NULL A, B or C");
    if (dtype != STARQ_F16 && dtype != STARQ_BF16) return fail(STARQ_ERR_ARG, "fp16_gemm_ref: dtype must be F16 or BF16");
    if (M < 0) return fail(STARQ_ERR_SHAPE, "M=%d < 0", M);
    if (N < 32 || N % 32 != 0) return fail(STARQ_ERR_SHAPE, "fp16_gemm_ref: N=%d: need N >= 32, N %% 32 == 0", N);
    if (K < 64 || K % 64 != 0) return fail(STARQ_ERR_SHAPE, "fp16_gemm_ref: K=%d: need K >= 64, K %% 64 == 0", K);
    if (M == 0) return STARQ_OK;
    if (!aligned(A, 16) || !aligned(B, 16) || !aligned(C, 16))
        return fail(STARQ_ERR_ALIGN, "fp16_gemm_ref: A, B, C must be 16-byte aligned");
    int rc = check_local("fp16_gemm_ref", static_cast<cudaStream_t>(stream), {A, B, C});
    if (rc) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    GemmArgs a{nullptr, nullptr, nullptr, nullptr, nullptr, M, N, K, C, dtype, nullptr, st,
               static_cast<const uint8_t*>(A), static_cast<const uint8_t*>(B)};
    cudaError_t e = launch_fp16_gemm(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "fp16_gemm_ref launch");
    return STARQ_OK;
}

int tac_prepare(const float* M, int C, int g, int z_dtype, void* Mp, void* stream) {
    if (C > 0 && (!M || !Mp)) return fail(STARQ_ERR_ARG, "tac_prepare: NULL M or Mp");
    if (z_dtype != STARQ_F16 && z_dtype != STARQ_BF16)
        return fail(STARQ_ERR_ARG, "tac_prepare: z_dtype must be F16 or BF16 (the tensor-core path)");
    if (g != 64 && g != 128) return fail(STARQ_ERR_SHAPE, "tac_prepare: g=%d: the tensor-core path takes 64 or 128", g);
    if (C < 0 || C % g != 0) return fail(STARQ_ERR_SHAPE, "tac_prepare: C=%d must be a multiple of g=%d", C, g);
    if (C == 0) return STARQ_OK;
    if (!aligned(M, 16) || !aligned(Mp, 16)) return fail(STARQ_ERR_ALIGN, "tac_prepare: M, Mp alignment");
    cudaError_t e = launch_tac_prepare(M, C, g, z_dtype, Mp, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tac_prepare launch");
    return STARQ_OK;
}


int tac_apply(const void* Z, int z_dtype, int L, int C, int g, const float* M, const float* d, const void* Mp,
              void* out, int out_dtype, void* stream) {
    if (L > 0 && (!Z || !out)) return fail(STARQ_ERR_ARG, "tac_apply: NULL Z or out");
    if (!dtype_ok(z_dtype) || !dtype_ok(out_dtype)) return fail(STARQ_ERR_ARG, "tac_apply: unknown dtype");
    int rc = check_tac(L, C, g, M, d);
    if (rc) return rc;
    if ((rc = check_tac_prepared(Mp, z_dtype, g))) return rc;
    if (L == 0) return STARQ_OK;
    if (!aligned(Z, 16) || !aligned(out, 16)) return fail(STARQ_ERR_ALIGN, "tac_apply: Z, out alignment");
    if ((rc = check_local("tac_apply", static_cast<cudaStream_t>(stream), {Z, out}))) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    TacArgs a{Z, z_dtype, L, C, g, M, d, out, out_dtype, st, Mp};
    cudaError_t e = launch_tac(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tac_apply launch");
    return STARQ_OK;
}

size_t attention_pv_tac_workspace_size(int L, int Hkv) {
    if (L <= 0 || Hkv <= 0) return 0;
    return attn_workspace_bytes(L, Hkv);
}

int attention_pv_tac_gqa(const void* Q, const void* K, const void* V, int ld, int L, int H, int Hkv, int dtype,
                         const void* Mp, const float* d, void* Z, uint8_t* dbg_codes, float* dbg_l, int32_t* dbg_acc,
                         void* workspace, size_t workspace_bytes, void* stream) {
    if (!Q || !K || !V || !Mp || !Z || !workspace) return fail(STARQ_ERR_ARG, "attention_pv_tac: NULL pointer");
    if (dtype != STARQ_F16 && dtype != STARQ_BF16)
        return fail(STARQ_ERR_ARG, "attention_pv_tac: dtype must be F16 or BF16");
    if (H < 1 || Hkv < 1 || H % Hkv != 0)
        return fail(STARQ_ERR_SHAPE, "attention_pv_tac: H=%d, Hkv=%d: need H a positive multiple of Hkv", H, Hkv);
    if (L < ATTN_TILE || L % ATTN_TILE != 0 || L > 8192)
        return fail(STARQ_ERR_SHAPE, "attention_pv_tac: L=%d: need 128 <= L <= 8192, L %% 128 == 0", L);
    if (ld < ATTN_D * H || ld % 8 != 0)
        return fail(STARQ_ERR_SHAPE, "attention_pv_tac: ld=%d: need ld >= 128 H and ld %% 8 == 0", ld);
    const size_t need = attention_pv_tac_workspace_size(L, Hkv);
    if (workspace_bytes < need) return fail(STARQ_ERR_SHAPE, "attention_pv_tac: workspace %zu bytes < %zu", workspace_bytes, need);
    if (!aligned(Q, 16) || !aligned(K, 16) || !aligned(V, 16) || !aligned(Mp, 16) || !aligned(Z, 16) ||
        (d && !aligned(d, 16)) || !aligned(workspace, 256))
        return fail(STARQ_ERR_ALIGN, "attention_pv_tac: Q, K, V, Mp, Z, d 16-byte and workspace 256-byte alignment");
    int rc = check_local("attention_pv_tac", static_cast<cudaStream_t>(stream), {Q, K, V, Z, workspace});
    if (rc) return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    AttnArgs a{Q, K, V, ld, L, H, Mp, d, Z, reinterpret_cast<uint16_t*>(ws),
               reinterpret_cast<float*>(ws + ((size_t)ATTN_D * Hkv * L * 2 + 255) / 256 * 256),
               dbg_codes, dbg_l, dbg_acc, st, Hkv, dtype};
    cudaError_t e = launch_attention_pv_tac(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "attention_pv_tac launch");
    return STARQ_OK;
}

int attention_pv_tac(const void* Q, const void* K, const void* V, int ld, int L, int H, const void* Mp,
                     const float* d, void* Z, uint8_t* dbg_codes, float* dbg_l, int32_t* dbg_acc, void* workspace,
                     size_t workspace_bytes, void* stream) {
    return attention_pv_tac_gqa(Q, K, V, ld, L, H, H, STARQ_F16, Mp, d, Z, dbg_codes, dbg_l, dbg_acc, workspace,
                                workspace_bytes, stream);
}

size_t tac_calibrate_workspace_size(int C, int g) {
    if (C <= 0 || g <= 0 || C % g != 0) return 0;
    return tac_calib_workspace_doubles(C, g) * sizeof(double);
}

int tac_calibrate(const void* Z_fp, const void* Z_q, int z_dtype, int N, int C, int g, double rho, double eps,
                  double eta, double alpha, float* M, float* d, void* workspace, size_t workspace_bytes,
                  void* stream) {
    if (!Z_fp || !Z_q || !M || !d || !workspace) return fail(STARQ_ERR_ARG, "tac_calibrate: NULL pointer");
    if (!dtype_ok(z_dtype)) return fail(STARQ_ERR_ARG, "tac_calibrate: unknown dtype %d", z_dtype);
    if (!(g == 4 || g == 8 || g == 16 || g == 32 || g == 64 || g == 128))
        return fail(STARQ_ERR_SHAPE, "tac_calibrate: g=%d: supported 4, 8, 16, 32, 64, 128", g);
    if (C <= 0 || C % g != 0) return fail(STARQ_ERR_SHAPE, "tac_calibrate: C=%d must be a positive multiple of g=%d", C, g);
    if (N < 1) return fail(STARQ_ERR_SHAPE, "tac_calibrate: N=%d: at least one token", N);
    if (!(rho >= 0.0) || !(eps > 0.0) || !(eta >= 0.0 && eta <= 1.0) || !(alpha >= 0.0 && alpha <= 1.0))
        return fail(STARQ_ERR_ARG, "tac_calibrate: need rho >= 0, eps > 0, eta and alpha in [0, 1]");
    const size_t need = tac_calibrate_workspace_size(C, g);
    if (workspace_bytes < need) return fail(STARQ_ERR_SHAPE, "tac_calibrate: workspace %zu bytes < %zu", workspace_bytes, need);
    if (!aligned(Z_fp, 16) || !aligned(Z_q, 16) || !aligned(M, 16) || !aligned(d, 16) || !aligned(workspace, 256))
        return fail(STARQ_ERR_ALIGN, "tac_calibrate: Z_fp, Z_q, M, d 16-byte and workspace 256-byte alignment");
    int rc = STARQ_OK;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    CalArgs a{Z_fp, Z_q, z_dtype, N, C, g, rho, eps, eta, alpha, M, d, static_cast<double*>(workspace), st};
    cudaError_t e = launch_tac_calibrate(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "tac_calibrate launch");
    return STARQ_OK;
}

size_t sgat_linear_workspace_size_bits(int L, int K, int with_tac, int bits) {
    if (L < 0 || K < 0 || (bits != 4 && bits != 8)) return 0;
    // codes (packed nibbles or bytes), s_a, the GEMM operand (E4M3 codes or
    // 8-bit codes as fp16), TAC output
    const size_t q = bits == 8 ? (size_t)L * K : (size_t)L * K / 2;
    const size_t e = bits == 8 ? (size_t)L * K * 2 : (size_t)L * K;
    size_t n = align256(q) + align256((size_t)L * 4) + align256(e);
    if (with_tac) n += align256((size_t)L * K * 4);
    return n;
}

size_t sgat_linear_workspace_size(int L, int K, int with_tac) {
    return sgat_linear_workspace_size_bits(L, K, with_tac, 4);
}

}  // extern "C"

namespace {
int sgat_linear_impl(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                     const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                     const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                     const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias, int N, int bits,
                     void* Y, int y_dtype, void* workspace, size_t workspace_bytes, void* stream, int swiglu,
                     bool ws_owned) {
    if ((!Wq && !We) || !s_w) return fail(STARQ_ERR_ARG, "sgat_linear: NULL Wq/We or s_w");
    if (L > 0 && (!X || !Y || !workspace)) return fail(STARQ_ERR_ARG, "sgat_linear: NULL X, Y or workspace");
    if (!dtype_ok(x_dtype) || !dtype_ok(y_dtype)) return fail(STARQ_ERR_ARG, "sgat_linear: unknown dtype");
    if (bits != 4 && bits != 8) return fail(STARQ_ERR_BITS, "bits=%d: the GPU path implements 4- and 8-bit codes", bits);
    if (bits == 8 && swiglu) return fail(STARQ_ERR_BITS, "sgat_linear_swiglu: 4-bit codes only");
    if (L < 0) return fail(STARQ_ERR_SHAPE, "L=%d < 0", L);
    int rc = check_transform(K, hb, d_sh, d_m, d_u, a_m, a_u);
    if (rc) return rc;
    if (tac_M && (rc = check_tac(L, K, tac_g, tac_M, tac_d))) return rc;
    if (tac_M && (rc = check_tac_prepared(tac_Mp, x_dtype, tac_g))) return rc;
    if (L == 0) return STARQ_OK;
    const size_t need = sgat_linear_workspace_size_bits(L, K, tac_M != nullptr, bits);
    if (workspace_bytes < need)
        return fail(STARQ_ERR_SHAPE, "workspace %zu bytes < %zu needed", workspace_bytes, need);
    if (!aligned(workspace, 256) || !aligned(X, 16)) return fail(STARQ_ERR_ALIGN, "sgat_linear alignment");
    const size_t qbytes = bits == 8 ? (size_t)L * K : (size_t)L * K / 2;
    const size_t ebytes = bits == 8 ? (size_t)L * K * 2 : (size_t)L * K;
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    uint8_t* Xq = ws;
    float* s_a = reinterpret_cast<float*>(ws + align256(qbytes));
    uint8_t* Xe = ws + align256(qbytes) + align256((size_t)L * 4);
    // TAC output in the input's type (the region has room for float32)
    void* zt = tac_M ? static_cast<void*>(Xe + align256(ebytes)) : nullptr;
    rc = bits == 8 ? check_w8a8(Xe, s_a, We, s_w, bias, L, N, K, Y, y_dtype)
                   : check_gemm(Xq, Xe, s_a, Wq, We, s_w, bias, L, N, K, Y, y_dtype);
    if (rc) return rc;
    // the scratch of sgat_linear_noalloc is the library's own device array
    if ((rc = check_local("sgat_linear", static_cast<cudaStream_t>(stream),
                          {X, ws_owned ? nullptr : workspace, We ? We : Wq, Y})))
        return rc;
    unsigned* st = status_ptr(&rc);
    if (!st) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const void* qin = X;
    int qin_dtype = x_dtype;
    cudaError_t e;
    if (tac_M) {
        TacArgs t{X, x_dtype, L, K, tac_g, tac_M, tac_d, zt, x_dtype, st, tac_Mp};
        t.params_ready = 1;      // layer parameters: see the header's note on programmatic launch
        if ((e = launch_tac(t, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear: tac launch");
        qin = zt;
        qin_dtype = x_dtype;
    }
    // every GEMM path below reads the E4M3 form, so the packed codes are not written
    QuantArgs q{qin, qin_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, bits == 8 ? 127 : 7, 1.f, nullptr, s_a, nullptr, Xe};
    if ((e = launch_sgat_quant(q, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear: quant launch");
    if (bits == 8) {
        GemmArgs g8{nullptr, s_a, nullptr, s_w, bias, L, N, K, Y, y_dtype, nullptr, st, Xe, We};
        g8.weights_ready = 1;    // the predecessor is the quantiser, which does not write the weights
        if ((e = launch_w8a8_gemm(g8, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear: w8a8 gemm launch");
        return STARQ_OK;
    }
    GemmArgs g{nullptr, s_a, Wq, s_w, bias, L, N, K, Y, y_dtype, nullptr, st, Xe, We};   // Xe: no packed codes read
    // the GEMM's predecessor is the quantiser launched above, which waits for
    // everything before it and does not write the weights
    g.weights_ready = 1;
    g.swiglu = swiglu;
    if ((e = launch_w4a4_gemm(g, s)) != cudaSuccess) return cuda_fail(e, "sgat_linear: gemm launch");
    return STARQ_OK;
}
}  // namespace

namespace starq {
int sgat_linear_scratch(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                        const float* a_u, int hb, int d_sh, int d_m, int d_u, const float* tac_M, const float* tac_d,
                        int tac_g, const void* tac_Mp, const uint8_t* Wq, const uint8_t* We, const float* s_w,
                        const float* bias, int N, int bits, void* Y, int y_dtype, void* scratch, size_t scratch_bytes,
                        void* stream) {
    return sgat_linear_impl(X, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, tac_M, tac_d, tac_g, tac_Mp, Wq,
                            We, s_w, bias, N, bits, Y, y_dtype, scratch, scratch_bytes, stream, 0, true);
}
}  // namespace starq

extern "C" {

int sgat_linear(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias, int N, int bits,
                void* Y, int y_dtype, void* workspace, size_t workspace_bytes, void* stream) {
    return sgat_linear_impl(X, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, tac_M, tac_d, tac_g, tac_Mp, Wq,
                            We, s_w, bias, N, bits, Y, y_dtype, workspace, workspace_bytes, stream, 0, false);
}

int sgat_linear_swiglu(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                       const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                       const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                       const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias, int N, int bits,
                       void* H, int h_dtype, void* workspace, size_t workspace_bytes, void* stream) {
    if (!We) return fail(STARQ_ERR_ARG, "sgat_linear_swiglu: needs the E4M3 weights We");
    if (h_dtype != STARQ_F16 && h_dtype != STARQ_BF16)
        return fail(STARQ_ERR_ARG, "sgat_linear_swiglu: output dtype must be F16 or BF16");
    if (N < 32 || N % 32 != 0)
        return fail(STARQ_ERR_SHAPE, "sgat_linear_swiglu: N=%d: gate and up rows interleaved by 16, N %% 32 == 0", N);
    return sgat_linear_impl(X, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, tac_M, tac_d, tac_g, tac_Mp, Wq,
                            We, s_w, bias, N, bits, H, h_dtype, workspace, workspace_bytes, stream, 1, false);
}

}  // extern "C"
