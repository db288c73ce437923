/*
 * starq.h -- C ABI of libstarq.so, the GB300 (sm_103a) hot path of the
 * STaR-Quant quantised denoising step: the SGAT-transformed W4A4 linear and
 * Temporal Attention Compensation (TAC).
 *
 * Conventions for every entry point:
 *   - All array arguments are DEVICE pointers owned by the caller. The library
 *     never allocates, frees or keeps a pointer past the call. Operands that
 *     the kernels read or write through TMA tensor maps must be memory of
 *     the current device (cudaSetDevice); calls that build tensor maps check
 *     this with cudaPointerGetAttributes (outside stream capture) and return
 *     STARQ_ERR_ARG for host, managed or another device's memory.
 *   - Host-side state (per-device kernel attributes, occupancy and
 *     address caches) is initialised once per device under a lock, so the
 *     entry points may be called from several host threads at once.
 *   - Work is enqueued asynchronously on `stream` (a cudaStream_t passed as
 *     void*; NULL = the legacy default stream). Arguments are validated on
 *     the host before anything is launched; a call that returns an error
 *     launched nothing.
 *   - Return value: STARQ_OK (0) or a negative STARQ_ERR_* code; the
 *     message of the last error on the calling thread is returned by
 *     starq_last_error().
 *   - Matrices are row-major and dense (row stride = number of columns).
 *   - L = 0 (no tokens) is a valid no-op; pointers to arrays with L rows may
 *     then be NULL.
 *   - Packed int4: a [rows][K] code matrix is stored as uint8 [rows][K/2];
 *     code k lives in byte k/2, even k in the low nibble, odd k in the high
 *     nibble, each nibble in two's complement. Codes lie in [-7, 7].
 *   - Mask: uint8 per token, 1 = masked (state m), 0 = unmasked (state u).
 */
#ifndef STARQ_H
#define STARQ_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Element types of activations, weights and outputs. */
enum starq_dtype { STARQ_F16 = 0, STARQ_BF16 = 1, STARQ_F32 = 2 };

/*
 * TAC parameters for the tac option of sgat_quantize_act and w4a4_gemm
 * (Sec. 3.3 Eq. 17: z_b <- M_b z_b + d_b on every block of g channels; the
 * same arithmetic as tac_apply). All pointers are device memory the caller
 * owns.
 *   g        block size: 4, 8, 16, 32, 64 or 128; the channel count is a
 *            multiple of g.
 *   M, d     [C/g][g][g] and [C/g][g] float32, 16-byte aligned (d NULL =
 *            zeros).
 *   Mp       tac_prepare output for the tensor being compensated (its
 *            element type, this C and g), or NULL (see tac_apply).
 *   scratch  [L][C] buffer, 16-byte aligned, of the compensated tensor's
 *            element type: sgat_quantize_act writes the compensated input
 *            there and quantises it; w4a4_gemm writes the uncompensated
 *            output there and compensates it into Y. It must not overlap
 *            the call's other buffers.
 */
typedef struct {
    int g;
    const float* M;
    const float* d;
    const void* Mp;
    void* scratch;
} starq_tac;

/* Return codes. */
enum starq_status {
    STARQ_OK = 0,
    STARQ_ERR_ARG = -1,      /* null pointer or unknown enum value            */
    STARQ_ERR_SHAPE = -2,    /* size outside the supported set (see each call) */
    STARQ_ERR_ALIGN = -3,    /* pointer not aligned as the call requires       */
    STARQ_ERR_BITS = -4,     /* bit-width other than 4 on the GPU path         */
    STARQ_ERR_CUDA = -5,     /* a CUDA runtime call or launch failed           */
    STARQ_ERR_TIMEOUT = -6   /* a kernel gave up a bounded wait (see status)   */
};

/* Library version (major * 10000 + minor * 100 + patch). */
int starq_version(void);

/* Message of the last error returned on the calling thread ("" if none). */
const char* starq_last_error(void);

/*
 * Synchronise `stream`, then read and clear the device status word that the
 * kernels set when a bounded wait inside them runs out. Returns STARQ_OK,
 * STARQ_ERR_TIMEOUT (the kernel returned early; its outputs are undefined)
 * or STARQ_ERR_CUDA.
 *
 * Scope: there is ONE status word per device, shared by every stream and
 * host thread that launches this library's kernels on it. The call waits
 * for `stream` only, then reads and clears the whole word: a timeout of a
 * kernel on another stream of the same device is reported (and cleared) by
 * whichever call reads the word first, and a timeout on another stream that
 * is still running when the word is read shows up in a later call. A caller
 * that uses several streams should synchronise all of them before calling
 * this, and treat a timeout as a failure of every kernel since its last
 * check on that device.
 */
int starq_check_status(void* stream);

/*
 * starq_selftest_wait_timeout -- failure-detection self-test (the paper has
 * no counterpart). Launches one kernel whose single thread waits on an
 * mbarrier that nothing arrives on, through the library's bounded wait,
 * with a limit of limit_us microseconds (1 .. 100000). The wait runs out,
 * the kernel sets the status bit 0x4 (self-test timeout) and returns: no
 * fault, no hang, and the context stays usable. The next
 * starq_check_status on the device then returns STARQ_ERR_TIMEOUT with the
 * bit in its message and clears the word. Returns STARQ_OK once launched,
 * STARQ_ERR_ARG for a limit outside the range, STARQ_ERR_CUDA if the launch
 * fails.
 */
int starq_selftest_wait_timeout(unsigned limit_us, void* stream);

/*
 * starq_probe_mma -- rate probe of the tensor-core instruction kinds, the
 * measured denominators of the GEMM rooflines (the paper has no
 * counterpart; sm_103a has no integer tcgen05 MMA, so the W4A4 path runs on
 * the FP8 kind and its peak has to be measured, not looked up).
 *
 * Every CTA issues `iters` rounds of back-to-back MMAs on operands resident
 * on chip, waits (bounded) for them, writes its cycle count to cycles[cta]
 * and adds the number of accumulators that differ from the exact expected
 * value to *errors. The caller times the launch with events on `stream`
 * and computes 2 * macs_per_cta * ctas / time.
 *   kind 0  tcgen05.mma cta_group::1 kind::f8f6f4, E4M3 x E4M3 -> F32,
 *           M 128 N 256 K 32 per instruction, one CTA per SM; operands all
 *           E4M3(7), so every accumulator must equal 49 * 128 * iters
 *           exactly (integer sums below 2^24 through the FP8 path).
 *   kind 1  the same on CTA pairs (cta_group::2, M 256 over the pair), the
 *           form w4a4_gemm issues.
 *   kind 2  tcgen05.mma cta_group::1 kind::f16, bf16 operands 1.0,
 *           M 128 N 256 K 16; accumulators 64 * iters.
 *   kind 3  mma.sync m16n8k32 s8.s8.s32 (warp-level integer MMA), four CTAs
 *           per SM of four warps, eight independent accumulator chains per
 *           warp; accumulators 32 * iters.
 *   kind 4  mma.sync m16n8k64 s4.s4.s32, likewise; accumulators 64 * iters.
 *   iters   1 .. 2048.
 *   cycles  device u64 [4 * SM count] (room for every kind), out.
 *   errors  device int32, zeroed by the caller; mismatch count added.
 *   ctas, macs_per_cta  host outputs: CTAs launched, multiply-adds per CTA.
 */
int starq_probe_mma(int kind, int iters, unsigned long long* cycles, int* errors, int* ctas,
                    double* macs_per_cta, void* stream);

/*
 * sgat_quantize_act -- state-guided activation transform + per-token A4
 * quantisation (Sec. 3.2 Eq. 7-11 and Eq. 13's Q_a; Sec. 3.1 Eq. 2-3).
 *
 * For every token i with state s = mask[i]:
 *   v = ((X[i] * a_s) H_hb) G_s        (Phi_s of Eq. 11; H_hb is the
 *                                        unnormalised block-diagonal Sylvester
 *                                        Hadamard, fast transform in float32)
 *   s_a[i] = amax / 7,  r = 7 / amax,  q = clamp(rne(v * r), -7, 7)
 * Tokens are processed in place of the paper's split + scatter: each row
 * picks its own transform, which gives the same rows in token order.
 *
 *   X       [L][K] activations, element type x_dtype (F16, BF16 or F32),
 *           16-byte aligned.
 *   mask    [L] uint8 or NULL (NULL = every token unmasked).
 *   a_m,a_u [K] float32 per-state diagonal smoothing, 16-byte aligned, or
 *           NULL (= ones).
 *   hb      Hadamard block: power of two, 1 <= hb <= 4096, K % hb == 0
 *           (hb = 1 is the identity).
 *   d_sh,d_m,d_u  gate layout over transformed coordinates (Eq. 8-9):
 *           [0, d_sh) shared, [d_sh, d_sh + d_m) masked-only, the rest
 *           unmasked-only; each >= 0 and d_sh + d_m + d_u == K.
 *   bits    4, or 8 for the W8A8 setting (Tab. 5): the same quantiser with
 *           127 in place of 7.
 *   Xq      codes out, 8-byte aligned: bits 4: [L][K/2] packed int4 (low
 *           nibble = even k); bits 8: [L][K] int8. May be NULL when Xe is
 *           given (then only the GEMM operand form is written).
 *   s_a     [L] float32 per-token scales out (0 for an all-zero row).
 *   Xe      the GEMM operand out, 16-byte aligned, or NULL. bits 4: [L][K]
 *           the codes as E4M3 bytes (the form w4a4_gemm streams by TMA).
 *           bits 8: [L][K] the codes as fp16 numbers (exact for |c| <=
 *           127; the operand of w8a8_gemm).
 *   v_dbg   [L][K] float32 transformed activations out (before rounding),
 *           16-byte aligned, or NULL.
 *   tac     NULL, or TAC on the input first (the attention output before
 *           the output projection, Sec. 3.3): tac->scratch [L][K] of x_dtype
 *           receives TAC(X), and the transform and quantisation above read
 *           it in place of X. Two kernels (TAC on the tensor cores for
 *           16-bit X and g = 64 or 128, then the quantiser): a token's
 *           transform needs all K compensated channels, every one of the
 *           K / g blocks of M.
 * Shapes: L >= 0, 16 <= K <= 20480, K % 16 == 0.
 */
int sgat_quantize_act(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                      const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                      const starq_tac* tac, int bits, uint8_t* Xq, float* s_a, uint8_t* Xe, float* v_dbg,
                      void* stream);

/*
 * sgat_quantize_act_grouped -- two independent state-guided quantisations
 * of sgat_quantize_act's definition (Sec. 3.2 Eq. 7-11 and Eq. 2) in one
 * launch, e.g. the QKV projection's input and the O projection's
 * TAC-compensated input of one step. p0 and p1 each name an input X
 * [L][K] of x_dtype, its mask, smoothing vectors, gate layout and outputs
 * (Xq, s_a and optionally Xe), with the meanings of sgat_quantize_act; K,
 * hb, L, x_dtype and bits are shared. The results are bit-identical to two
 * sgat_quantize_act calls (no TAC option: apply tac_apply first). Symmetric
 * codes with K <= 4096 run as one kernel with one CTA per row of either
 * problem; other shapes run as two launches. Errors as sgat_quantize_act.
 */
typedef struct {
    const void* X;
    const uint8_t* mask;
    const float* a_m;
    const float* a_u;
    int d_sh, d_m, d_u;
    uint8_t* Xq;
    float* s_a;
    uint8_t* Xe;
    int independent;   /* 1: the caller guarantees that the launch just before this
                          call on the stream neither writes X, mask, a_m, a_u nor reads
                          or writes Xq, s_a, Xe; this problem's rows may then start
                          while that launch finishes (programmatic launch). 0: wait. */
} starq_quant_io;
int sgat_quantize_act_grouped(const starq_quant_io* p0, const starq_quant_io* p1, int x_dtype, int L, int K,
                              int hb, int bits, void* stream);

/*
 * sgat_prepare_weight -- the unified static weight transform, quantised once
 * (Sec. 3.2 Eq. 12; App. B W_f = Q_w(P^T W^T)), per-output-channel symmetric.
 *
 * For every output channel n:
 *   w = ((W[n] * inv_a_w) H_hb) / hb   (float32, fast transform)
 *   s_w[n] = amax / 7,  Wq[n] = clamp(rne(w * 7 / amax), -7, 7)
 *
 *   W       [N][K] weights, element type w_dtype (F16, BF16 or F32), 16-byte
 *           aligned.
 *   inv_a_w [K] float32 weight-side inverse smoothing or NULL (= ones).
 *   Wq      codes out: bits 4: [N][K/2] packed int4; bits 8: [N][K] int8.
 *   s_w     [N] float32 out.
 * Shapes and hb as for sgat_quantize_act; bits 4 or 8 (127 in place of 7).
 */
int sgat_prepare_weight(const void* W, int w_dtype, int N, int K, const float* inv_a_w, int hb,
                        int bits, uint8_t* Wq, float* s_w, void* stream);

/*
 * w4_unpack_e4m3 -- the prepared weight codes in the byte form the tensor
 * cores read: each int4 code q of Wq becomes the E4M3 byte of the value q
 * (exact: every integer of [-8, 8] is an E4M3 number). Run once per weight
 * after sgat_prepare_weight and keep We with Wq and s_w; w4a4_gemm and
 * sgat_linear then stream both operands by TMA without converting them.
 * (The paper has no counterpart: its int4 codes are unchanged, only their
 * storage for this GPU's FP8 tensor-core kind.)
 *
 *   Wq [N][K/2] packed int4 (low nibble = even k), 16-byte aligned.
 *   We [N][K] out, 16-byte aligned, caller-owned (N*K bytes).
 * Shapes: N >= 0, K >= 32 with K % 32 == 0.
 */
int w4_unpack_e4m3(const uint8_t* Wq, int N, int K, uint8_t* We, void* stream);

/*
 * w8_codes_f16 -- 8-bit weight codes in the form w8a8_gemm reads: each code
 * c of Wq [N][K] (int8) as the fp16 number c (exact for |c| <= 127),
 * We [N][K] fp16. Run once per weight after sgat_prepare_weight with
 * bits = 8.
 *   Wq, We 16-byte aligned; We caller-owned (2 N K bytes).
 * Shapes: N >= 0, K >= 128 with K % 128 == 0.
 */
int w8_codes_f16(const uint8_t* Wq, int N, int K, uint8_t* We, void* stream);

/*
 * w8a8_gemm -- the integer projection and its dequantisation at 8 bits (the
 * W8A8 setting of Tab. 5; Sec. 3.2 Eq. 13, Sec. 3.1 Eq. 3):
 *
 *   acc[i][n] = sum_k q_a[i][k] * q_w[n][k]            (exact integer)
 *   Y[i][n]   = (float)acc * s_a[i] * s_w[n] (+ bias[n]) rounded to y_dtype
 *               (float32 products in that order, then one rounding).
 *
 *   Xe [L][K] activation codes as fp16 (sgat_quantize_act, bits 8), We [N][K]
 *      weight codes as fp16 (w8_codes_f16), 16-byte aligned (2 K bytes a
 *      row each).
 *   One 16-bit tensor-core product (tcgen05 kind::f16, CTA pairs) on the
 *   codes, accumulated in float32 in runs of 512 K (each run an integer of
 *   magnitude at most 512 * 127^2 < 2^23, so exact); the epilogue adds the
 *   runs in int32.
 *   s_a [L], s_w [N] float32; bias [N] float32 or NULL.
 *   Y  [L][N] out, y_dtype F16, BF16 or F32, 16-byte aligned.
 *   acc_dbg [L][N] int32 out (the exact accumulators) or NULL.
 * Shapes: L >= 0, N >= 128 with N % 128 == 0, 128 <= K <= 65536 with
 * K % 128 == 0 (|acc| <= 127^2 K < 2^31).
 */
int w8a8_gemm(const uint8_t* Xe, const float* s_a, const uint8_t* We, const float* s_w, const float* bias, int L,
              int N, int K, void* Y, int y_dtype, int32_t* acc_dbg, void* stream);

/*
 * Asymmetric activation quantisation (Eq. 2-4) with symmetric per-channel
 * weights, through the 4-bit GEMM.
 *
 * sgat_quantize_act_asym -- sgat_quantize_act with the asymmetric 4-bit
 * quantiser per token: X_min = min(min v, 0), X_max = max(max v, 0) (zero
 * is inside the range), s = (X_max - X_min) / 15, r = 15 / (X_max - X_min),
 * z = rne(-X_min r) in [0, 15], q = clamp(rne(v r) + z, 0, 15), all in
 * float32; an all-zero row gets s = 0, z = 0, codes 0. X_hat = s (q - z).
 *   Xq  [L][K/2] packed unsigned nibbles out (low nibble = even k).
 *   s_a [L] float32 out, z_a [L] int32 out.
 *   Xe  [L][K + 128] out or NULL: the codes as E4M3 bytes, then 128 bytes
 *       of E4M3(-z) (the zero-point columns); K % 128 == 0 and K <= 7680.
 * Other arguments as for sgat_quantize_act.
 *
 * w4_zero_point_columns -- symmetric 4-bit weight codes Wq [N][K/2] (from
 * sgat_prepare_weight) to We [N][K + 128]: the codes as E4M3 bytes, then
 * 128 E4M3 values whose sum is exactly sum_k q_w[n][k]. With the
 * activations' zero-point columns, the GEMM over K + 128 computes
 * sum_k (q_a - z) q_w exactly. K % 128 == 0, K <= 7680 (128 E4M3 values of
 * at most 448 hold |sum| <= 7 K).
 *
 * sgat_linear_asym -- the fused linear with asymmetric activation codes:
 *   Y = (float)acc * s_a[i] * s_w[n] (+ bias), acc = sum_k (q_a - z_a) q_w,
 * i.e. sgat_quantize_act_asym then w4a4_gemm(Xe, We, K + 128). workspace:
 * sgat_linear_asym_workspace_size(L, K) bytes, 256-byte aligned, laid out
 * as [Xq L*K/2][s_a 4L][z_a 4L][Xe L*(K+128)], each part padded to 256.
 * N >= 32 with N % 32 == 0.
 */
int sgat_quantize_act_asym(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                           const float* a_u, int hb, int d_sh, int d_m, int d_u, uint8_t* Xq, float* s_a,
                           int32_t* z_a, uint8_t* Xe, void* stream);
int w4_zero_point_columns(const uint8_t* Wq, int N, int K, uint8_t* We, void* stream);
size_t sgat_linear_asym_workspace_size(int L, int K);

/*
 * Dense orthogonal basis (the learned P of App. B; W_f = Q_w(P^T W^T)) in
 * place of the block Hadamard transform. The transform X^s P is a 16-bit
 * GEMM: its operands are the scaled rows fl16(fl32(x * a_s)) and P, both
 * float16, accumulated in float32 on the tensor cores, and the result is
 * stored as float16. The gate and the symmetric 4-bit quantiser (hb = 1)
 * then run on it.
 *
 *   Pt [K][K] float16: the basis transposed (row j holds column j of P),
 *      16-byte aligned. P must be orthogonal: the weight side then uses the
 *      same matrix (w_f = w P, the row form of P^T W^T).
 *   Shapes: 128 <= K <= 16384 with K % 128 == 0.
 *
 * sgat_quantize_act_dense -- Q_a(X^s P G_s) per token: Xq [L][K/2] packed
 *   int4, s_a [L], Xe [L][K] E4M3 or NULL, as for sgat_quantize_act.
 *   workspace: sgat_dense_workspace_size(L, K) bytes, 256-byte aligned; it
 *   holds [scaled rows fp16 L*K][V = X^s P fp16 L*K], each padded to 256.
 * sgat_prepare_weight_dense -- Wq [N][K/2], s_w [N] from the rows
 *   fl16(fl16(w * inv_a_w) P); workspace sgat_dense_workspace_size(N, K).
 * sgat_linear_dense -- the fused linear: sgat_quantize_act_dense then
 *   w4a4_gemm (Wq/We from sgat_prepare_weight_dense and w4_unpack_e4m3).
 *   workspace: sgat_linear_dense_workspace_size(L, K) bytes: the dense
 *   workspace, then [Xq][s_a][Xe] as in sgat_linear.
 */
size_t sgat_dense_workspace_size(int rows, int K);
int sgat_quantize_act_dense(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                            const float* a_u, const void* Pt, int d_sh, int d_m, int d_u, uint8_t* Xq, float* s_a,
                            uint8_t* Xe, void* workspace, size_t workspace_bytes, void* stream);
int sgat_prepare_weight_dense(const void* W, int w_dtype, int N, int K, const float* inv_a_w, const void* Pt,
                              uint8_t* Wq, float* s_w, void* workspace, size_t workspace_bytes, void* stream);
size_t sgat_linear_dense_workspace_size(int L, int K);
int sgat_linear_dense(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                      const float* a_u, const void* Pt, int d_sh, int d_m, int d_u, const uint8_t* Wq,
                      const uint8_t* We, const float* s_w, const float* bias, int N, void* Y, int y_dtype,
                      void* workspace, size_t workspace_bytes, void* stream);
int sgat_linear_asym(const void* X, int x_dtype, int L, int K, const uint8_t* mask, const float* a_m,
                     const float* a_u, int hb, int d_sh, int d_m, int d_u, const uint8_t* We, const float* s_w,
                     const float* bias, int N, void* Y, int y_dtype, void* workspace, size_t workspace_bytes,
                     void* stream);

/*
 * w4a4_gemm -- the shared-weight integer projection and its dequantisation
 * (Sec. 3.2 Eq. 13, Sec. 3.1 Eq. 5 and Eq. 3).
 *
 *   acc[i][n] = sum_k q_a[i][k] * q_w[n][k]            (exact integer)
 *   Y[i][n]   = (float)acc * s_a[i] * s_w[n] (+ bias[n]) rounded to y_dtype
 *               (float32 products in that order, then one rounding).
 *
 *   Xq [L][K/2], Wq [N][K/2] packed int4, 16-byte aligned.
 *   Xe [L][K] the activation codes as E4M3 bytes (sgat_quantize_act's Xe
 *      output), 16-byte aligned, or NULL (then Xq is read).
 *   We [N][K] the weight codes as E4M3 bytes (w4_unpack_e4m3), 16-byte
 *      aligned, or NULL (then Wq is read). Used only together with Xe.
 *   Kernels: Xe and We: TMA streams both operands to CTA pairs (tcgen05
 *   cta_group::2, FP8 kind, float32 accumulators that hold the integer sums
 *   exactly); Xe only: the pairs convert the packed weights on the fly;
 *   neither: one CTA per tile converts both.
 *   s_a [L], s_w [N] float32; bias [N] float32 or NULL.
 *   Y  [L][N] out, y_dtype F16, BF16 or F32, 16-byte aligned.
 *   acc_dbg [L][N] int32 out (the exact accumulators) or NULL.
 *   out_tac NULL, or TAC on the output (C = N): the dequantised output goes
 *      to out_tac->scratch [L][N] of y_dtype, and Y = TAC(scratch) (a
 *      second kernel; the quantised softmax-value product has its TAC
 *      fused into its epilogue, attention_pv_tac).
 * Shapes: L >= 0, N >= 32 with N % 32 == 0, K >= 128 with K % 128 == 0,
 * K <= 65536 (so |acc| <= 49 K < 2^22).
 */
int w4a4_gemm(const uint8_t* Xq, const uint8_t* Xe, const float* s_a, const uint8_t* Wq,
              const uint8_t* We, const float* s_w, const float* bias, int L, int N, int K, void* Y,
              int y_dtype, const starq_tac* out_tac, int32_t* acc_dbg, void* stream);

/*
 * w4a4_gemm_grouped -- two independent W4A4 products of w4a4_gemm's
 * definition (Sec. 3.2 Eq. 13, Sec. 3.1 Eq. 3 and Eq. 5) in one launch:
 * Y0 = dequant(Xe0 We0^T) and Y1 = dequant(Xe1 We1^T), with the same L, K
 * and output type (e.g. the QKV projection of X and the O projection of the
 * compensated attention output, which share their token count and width).
 * The output tiles of problem 1 follow those of problem 0 in one persistent
 * stream of CTA-pair tiles, so a short problem's pipeline fill and drain
 * hide behind the other's tiles. Each output is bit-identical to a
 * w4a4_gemm call with Xe and We.
 *
 *   Xe0 [L][K], Xe1 [L][K]: E4M3 activation codes; We0 [N0][K], We1 [N1][K]:
 *      E4M3 weight codes (w4_unpack_e4m3); all 16-byte aligned, device
 *      memory of the current device (the caller owns every buffer).
 *   s_a0, s_a1 [L], s_w0 [N0], s_w1 [N1] float32; bias0, bias1 or NULL.
 *   Y0 [L][N0], Y1 [L][N1] of y_dtype (F16, BF16 or F32), 16-byte aligned.
 *   acc_dbg0, acc_dbg1: the exact int32 accumulators, or NULL.
 *   flags: 0, or STARQ_GEMM_WEIGHTS_READY: the caller guarantees that the
 *      launch just before this call on the stream does not write We0 or
 *      We1, so the first weight tiles are fetched while it finishes
 *      (programmatic launch); other bits are an error (STARQ_ERR_ARG).
 * Shapes and errors as w4a4_gemm for each problem (N0, N1 >= 32 and
 * multiples of 32; 128 <= K <= 65536, K % 128 == 0); L == 0 does nothing.
 */
#define STARQ_GEMM_WEIGHTS_READY 1
int w4a4_gemm_grouped(const uint8_t* Xe0, const float* s_a0, const uint8_t* We0, const float* s_w0,
                      const float* bias0, int N0, void* Y0, const uint8_t* Xe1, const float* s_a1,
                      const uint8_t* We1, const float* s_w1, const float* bias1, int N1, void* Y1, int L, int K,
                      int y_dtype, int32_t* acc_dbg0, int32_t* acc_dbg1, int flags, void* stream);

/*
 * starq_set_gemm_pair_limit -- at most `pairs` CTA pairs (two SMs each) for
 * the W4A4 and 16-bit TMA pair GEMMs launched afterwards from the calling
 * thread (w4a4_gemm with Xe and We, the sgat_linear family, fp16_gemm_ref);
 * 0 removes the cap. Returns the previous cap (>= 0), or STARQ_ERR_ARG for
 * pairs < 0. The cap is part of the launch, so a CUDA graph captured under
 * it keeps it. Use: a GEMM that runs beside other kernels (two branches of
 * one step) leaves them the remaining SMs; the results do not depend on it.
 */
int starq_set_gemm_pair_limit(int pairs);

/*
 * w4a4_gemm_mma_sync -- the same integer projection and dequantisation as
 * w4a4_gemm (Sec. 3.2 Eq. 13, Eq. 5, Eq. 3) on the warp-level integer MMA
 * (mma.sync m16n8k64 s4.s4.s32, the only int4 tensor-core instruction of
 * sm_103a), with native int32 accumulators: the comparison point for the
 * FP8-kind path that w4a4_gemm takes (starq_probe_mma kinds 1 and 4 give
 * the two instructions' rates).
 *
 *   Xq [L][K/2], Wq [N][K/2] packed int4 (low nibble = even k), 16-byte
 *   aligned; s_a [L], s_w [N] float32; bias [N] float32 or NULL; Y [L][N]
 *   out, y_dtype F16, BF16 or F32; acc_dbg [L][N] int32 out or NULL.
 *   Y[i][n] = fl(fl((float)acc s_a[i]) s_w[n]) (+ bias[n]), one rounding to
 *   y_dtype, as w4a4_gemm.
 * Shapes: L >= 0, N >= 1, K >= 128 with K % 128 == 0, K <= 65536.
 */
int w4a4_gemm_mma_sync(const uint8_t* Xq, const float* s_a, const uint8_t* Wq, const float* s_w,
                       const float* bias, int L, int N, int K, void* Y, int y_dtype, int32_t* acc_dbg,
                       void* stream);

/*
 * Tile of the last Xe + We (or fp16_gemm_ref) launch on the calling thread,
 * as BN * 10 + cluster size: 2562 (256-channel pair tiles) or 2242
 * (224-channel pair tiles); a cluster is one CTA pair, and each CTA loads
 * its own operand rows. 0 before the first. The launcher estimates each
 * shape's time as ceil(tiles / resident pairs) rounds of a stage cost bound
 * by shared-memory traffic and takes the cheaper. A diagnostic for tests
 * and tuning; the results do not depend on it.
 */
int starq_last_gemm_tile(void);

/*
 * fp16_gemm_ref -- the 16-bit baseline of the projections: C = A B^T with
 * float32 accumulation and one rounding to the element type. It is the
 * unquantised model's linear layer that Sec. 4.4 measures its speed-up
 * against; here it serves only as that denominator (the same CTA-pair
 * tcgen05 kernel structure as w4a4_gemm, kind::f16, no cuBLAS).
 *
 *   A [M][K], B [N][K] row-major, C [M][N] out; all of element type dtype
 *   (F16 or BF16), 16-byte aligned.
 * Shapes: M >= 0, N >= 32 with N % 32 == 0, K >= 64 with K % 64 == 0.
 */
int fp16_gemm_ref(const void* A, const void* B, int dtype, int M, int N, int K, void* C, void* stream);

/*
 * tac_prepare -- the TAC matrices in the form the tensor-core TAC reads
 * (the paper has no counterpart: a storage form, like w4_unpack_e4m3).
 * Every block M_b is split into two 16-bit matrices of Z's type,
 * hi = rn(M_b) and lo = rn(M_b - hi) (Z hi^T + Z lo^T reproduces Z M_b^T
 * with float32 accumulation to about 2^-22 relative), laid out K-major with
 * the 128-byte swizzle. Run once per set of TAC parameters; pass the result
 * as Mp to tac_apply / sgat_linear, which then copy it instead of splitting
 * M in every CTA.
 *
 *   M  [C/g][g][g] float32, 16-byte aligned.
 *   Mp out, 4*C*g bytes, 16-byte aligned, caller-owned.
 *   z_dtype: F16 or BF16, the type of the Z it will be applied to.
 * Shapes: g in {64, 128}, C % g == 0.
 */
int tac_prepare(const float* M, int C, int g, int z_dtype, void* Mp, void* stream);

/*
 * tac_apply -- block-wise affine compensation of the quantised attention
 * output before the output projection (Sec. 3.3 Eq. 17; App. C row-major
 * form Z_b M_b^T + 1 d_b^T).
 *
 *   out[i][b*g + r] = sum_j M[b][r][j] * Z[i][b*g + j] + d[b][r]
 *
 *   Z   [L][C] element type z_dtype (F16, BF16 or F32), 16-byte aligned.
 *   M   [C/g][g][g] float32 (row r = output channel r of block b); d [C/g][g]
 *       float32 (NULL = zeros). Both 16-byte aligned.
 *   Mp  tac_prepare(M, C, g, z_dtype) output or NULL; only with 16-bit Z and
 *       g = 64 or 128 (the tensor-core path), which otherwise splits M in
 *       every CTA.
 *   out [L][C] element type out_dtype (F16, BF16 or F32), 16-byte aligned;
 *       must not overlap Z.
 * Shapes: L >= 0, g in {4, 8, 16, 32, 64, 128}, C % g == 0, C % 8 == 0.
 */
int tac_apply(const void* Z, int z_dtype, int L, int C, int g, const float* M, const float* d,
              const void* Mp, void* out, int out_dtype, void* stream);

/*
 * attention_pv_tac -- the quantised softmax-value product of an attention
 * layer with TAC fused into its dequantisation epilogue (Sec. 3.3: Z_hat is
 * the quantised counterpart of Softmax(Q K^T / sqrt(d_h)) V, compensated
 * block-wise before the output projection; App. C places TAC right after
 * the softmax-value multiplication).
 *
 * The paper fixes neither the bit widths nor the granularity of that
 * multiplication. The readings:
 *   P per query row, unsigned 8-bit: c_ij = rne(255 exp(s_ij - m_i)), scale
 *     1 / (255 l_i), with s = q . k / sqrt(128), m_i = max_j s_ij and
 *     l_i = sum_j exp(s_ij - m_i). The row's largest probability maps to 255;
 *   V per channel, signed 4-bit: the activation quantiser along each column
 *     (t_c = amax_c / 7, v_jc = rne(V_jc fl(7 / amax_c)));
 *   Z_hat_ic = fl(fl(acc_ic fl(1 / fl(255 l_i))) t_c), acc_ic = sum_j c_ij v_jc
 *     exact (float32 tensor-core accumulation of integers below 2^24);
 *   Z = Z_hat_h M_h^T + d_h per head h: the head's 128 channels are one TAC
 *     block (Eq. 17 with g = 128).
 *
 *   Q, K, V fp16 [L][ld]: head h is columns 128 h .. 128 h + 127 (e.g. the
 *     three slices of the QKV projection's output, ld = 3 * 128 H).
 *   Mp: tac_prepare(M, 128 H, 128, F16) output; d [H][128] float32 or NULL.
 *   Z out fp16 [L][128 H], the TAC-compensated attention output.
 *   dbg_codes NULL or uint8 [H][L][L] (P codes), dbg_l NULL or float32 [H][L]
 *     (row sums l), dbg_acc NULL or int32 [H][L][128] (the exact sums): for
 *     tests.
 *   workspace: attention_pv_tac_workspace_size(L, H) bytes, 256-byte aligned
 *     (V codes transposed and the channel scales; the size takes the number
 *     of key/value heads, which is H here).
 * Shapes: head dimension 128, H >= 1, 128 <= L <= 8192 with L % 128 == 0,
 * ld >= 128 H with ld % 8 == 0; all pointers 16-byte aligned.
 * Kernels: a V quantiser (per-channel scales and transposed codes) and one
 * tcgen05 kernel with a CTA per (128-query tile, head): two passes of
 * Q K^T over 128-key chunks (row maxima, then probabilities, codes and sums
 * with P V^T accumulated one chunk behind), then the dequantisation and TAC
 * epilogue. Every CTA loads its own K / V tiles by TMA. The call is
 * asynchronous on `stream`; a wait that gives up inside the kernel is
 * reported by starq_check_status.
 */
size_t attention_pv_tac_workspace_size(int L, int Hkv);
int attention_pv_tac(const void* Q, const void* K, const void* V, int ld, int L, int H, const void* Mp,
                     const float* d, void* Z, uint8_t* dbg_codes, float* dbg_l, int32_t* dbg_acc,
                     void* workspace, size_t workspace_bytes, void* stream);

/*
 * attention_pv_tac_gqa -- attention_pv_tac with grouped-query attention and
 * a choice of element type (the Dream-7B / Qwen2.5 block: 28 query heads
 * over 4 key/value heads, bf16). Query head h reads key/value head
 * h / (H / Hkv): K and V hold Hkv heads (columns 128 k .. 128 k + 127 of
 * head k), Q and Z hold H heads. V is quantised per channel of the Hkv
 * heads, so the query heads of a group share one set of V codes and scales.
 *   dtype  STARQ_F16 or STARQ_BF16: the type of Q, K, V and Z. Q K^T runs in
 *          that type; the P and V codes are integers (exact in fp16); the
 *          TAC product runs on fp16 halves of Z_hat (scaled per head by an
 *          exact power of two into fp16's range) against M's fp16 halves,
 *          so Mp = tac_prepare(M, 128 H, 128, STARQ_F16) for either dtype.
 *   workspace  attention_pv_tac_workspace_size(L, Hkv) bytes.
 *   Other arguments, shapes and outputs as attention_pv_tac; H % Hkv == 0.
 * attention_pv_tac is this call with Hkv = H and dtype = STARQ_F16.
 */
int attention_pv_tac_gqa(const void* Q, const void* K, const void* V, int ld, int L, int H, int Hkv, int dtype,
                         const void* Mp, const float* d, void* Z, uint8_t* dbg_codes, float* dbg_l,
                         int32_t* dbg_acc, void* workspace, size_t workspace_bytes, void* stream);

/*
 * tac_calibrate -- the closed-form TAC parameters (App. C, "Block-wise
 * statistics" through "Bias estimation"), on the GPU in float64.
 *
 *   For every block b of g channels, from the N paired calibration tokens:
 *     mu_b, Sigma_b = population mean and covariance of Z_fp and of Z_q;
 *     lambda_b = rho * max(Tr(Sigma^Q_b) / g, eps);
 *     M_b = (Sigma^FP_b)^(1/2) (Sigma^Q_b + lambda_b I)^(-1/2), each power
 *           Q diag(max(lambda_i, 1e-12)^p) Q^T of a symmetric
 *           eigendecomposition;
 *     singular values of M_b replaced by (1 - eta) sigma_i + eta mean(sigma);
 *     M_b <- (1 - alpha) M_b + alpha I;  d_b = mu^FP_b - M_b mu^Q_b.
 *   The paper's defaults: rho = 3e-4, eps = 1e-8, eta = 0.15, alpha = 0.55.
 *
 *   Z_fp, Z_q [N][C] of element type z_dtype (F16, BF16 or F32), the full-
 *     precision and quantised attention outputs of the same N tokens,
 *     16-byte aligned.
 *   M out [C/g][g][g] float32 (row r = output channel r of block b), d out
 *     [C/g][g] float32: tac_apply's parameter layout. 16-byte aligned.
 *   workspace: tac_calibrate_workspace_size(C, g) bytes of device memory,
 *     256-byte aligned, caller-owned; its contents do not matter.
 * Shapes: N >= 1, g in {4, 8, 16, 32, 64, 128}, C % g == 0.
 * Kernels: a token reduction (fp64 sums and second moments per block) and
 * one CTA per block for the matrix functions (parallel cyclic Jacobi) and
 * the SVD of M (one-sided Jacobi on the same schedule).
 */
size_t tac_calibrate_workspace_size(int C, int g);
int tac_calibrate(const void* Z_fp, const void* Z_q, int z_dtype, int N, int C, int g, double rho, double eps,
                  double eta, double alpha, float* M, float* d, void* workspace, size_t workspace_bytes,
                  void* stream);

/*
 * sgat_linear -- the fused SGAT W4A4 linear of one quantised layer: optional
 * TAC on the input (Eq. 17), the state-guided transform and A4 quantisation
 * (Eq. 11), and the shared-weight integer GEMM with its dequantisation
 * epilogue (Eq. 13). Equivalent to tac_apply (to float32) ->
 * sgat_quantize_act -> w4a4_gemm, with the intermediates in `workspace`.
 *
 *   tac_M, tac_d, tac_g, tac_Mp: TAC parameters as for tac_apply (tac_Mp =
 *   tac_prepare output or NULL), or tac_M = NULL for no TAC. Wq/s_w come
 *   from sgat_prepare_weight, We (optional, NULL = convert Wq on the fly)
 *   from w4_unpack_e4m3. Other arguments as in the calls above.
 *   K % 128 == 0.
 *   workspace: device buffer of at least sgat_linear_workspace_size(L, K,
 *   tac_M != NULL) bytes (bits 4) or sgat_linear_workspace_size_bits(L, K,
 *   tac_M != NULL, bits), 256-byte aligned, owned by the caller. On return
 *   it holds the intermediates, laid out as [a region of L*K/2 bytes (bits
 *   4) or L*K (bits 8), padded to 256, left unwritten: the GEMM reads the
 *   codes in their operand form only][s_a: 4*L bytes, padded to 256][GEMM
 *   operand Xe, the codes: L*K E4M3 bytes (bits 4) or L*K fp16 (bits 8),
 *   padded to 256][TAC output: L*K values of x_dtype (room for float32),
 *   only with TAC]. The TAC output is rounded to x_dtype once, as the
 *   unquantised model stores attention outputs, and the quantiser reads it.
 *   bits 8 (the W8A8 setting): Wq may be NULL; We is the w8_codes_f16
 *   output and the GEMM is w8a8_gemm's; N % 128 == 0.
 *
 *   Programmatic launch: the kernels of sgat_linear may start while the
 *   previous kernel of the stream is still running (CUDA programmatic
 *   dependent launch) and read the layer's parameters (Wq/We, s_w, bias,
 *   tac_M, tac_d, tac_Mp) before waiting for it; the inputs and the
 *   workspace are read only after it has completed. Parameters must
 *   therefore not be written by a kernel that lets its dependents start
 *   early; no kernel of this library does, and the preparation calls
 *   (sgat_prepare_weight, w4_unpack_e4m3, tac_prepare) never let them.
 */
size_t sgat_linear_workspace_size(int L, int K, int with_tac);
size_t sgat_linear_workspace_size_bits(int L, int K, int with_tac, int bits);
int sgat_linear(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias, int N,
                int bits, void* Y, int y_dtype, void* workspace, size_t workspace_bytes, void* stream);

/*
 * sgat_linear_swiglu -- sgat_linear for the gate and up projections of a
 * SwiGLU MLP, with the activation fused into the GEMM's epilogue. Gate and
 * up share one quantised input (Sec. 3.2: every quantised linear, the MLP's
 * included, runs through the SGAT transform). The activation is the MLP's
 * own, silu(gate) * up, not part of the paper's method.
 *
 *   Wq, We, s_w, bias: the 2F output channels with gate and up rows
 *     interleaved in groups of 16: rows 32 k .. 32 k + 15 are gate channels
 *     16 k .. 16 k + 15, rows 32 k + 16 .. 32 k + 31 the matching up
 *     channels. Prepare them from the weight rows in that order.
 *   N = 2F, N % 32 == 0; We is required.
 *   H [L][F] out, h_dtype F16 or BF16:
 *     H[i][f] = silu(y_gate) * y_up rounded once to h_dtype, y = the float32
 *     dequantised outputs, silu(x) = x / (1 + exp(-x)).
 * Other arguments and the workspace are exactly sgat_linear's.
 */
int sgat_linear_swiglu(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                       const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                       const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                       const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias, int N,
                       int bits, void* H, int h_dtype, void* workspace, size_t workspace_bytes, void* stream);

/*
 * sgat_linear_noalloc -- sgat_linear for callers that cannot allocate device
 * memory. (The paper has no counterpart: this is a deployment convenience.)
 *
 * Some callers may not call cudaMalloc at all: a serving runtime that plans
 * all device memory at start-up and owns the pool, a plugin or custom-op
 * interface that passes an operator only its inputs and outputs, or a
 * latency-critical path where cudaMalloc's implicit device synchronisation
 * is not acceptable. They cannot supply sgat_linear's workspace. This entry
 * point instead keeps the intermediates in a fixed scratch array of
 * STARQ_NOALLOC_SCRATCH_BYTES bytes inside the library's device image
 * (every GPU that loads the library holds it until the process exits), and
 * allocates nothing: no cudaMalloc, no cudaFree, no allocating library call.
 * The caller still passes all inputs and outputs; arguments and results are
 * exactly those of sgat_linear without `workspace` / `workspace_bytes`.
 *
 *   - Limit: sgat_linear_workspace_size_bits(L, K, tac_M != NULL, bits)
 *     must not exceed STARQ_NOALLOC_SCRATCH_BYTES (32 MiB). At K = 4096 a
 *     4-bit call with TAC needs 22,532 bytes per token (1024 tokens:
 *     23,072,768 bytes), so up to 1489 tokens fit; without TAC 6,148 bytes
 *     per token. 8-bit calls need more (K + 4 + 2K, plus 4K with TAC, bytes
 *     per token) and reach the limit at fewer tokens (1170 at K = 4096 with
 *     TAC). Larger calls return STARQ_ERR_SHAPE with a message and launch
 *     nothing.
 *   - The first call on each device looks up the scratch array's device
 *     address (cudaGetSymbolAddress, with that device current) and caches
 *     it; make that first call before any stream capture on that device.
 *     The cached address is stale after cudaDeviceReset on that device: do
 *     not call this entry point there again in the same process.
 *   - All calls on a device share the one array, which keeps the last call's
 *     contents. Nothing in it needs to start at zero: every byte a call reads
 *     back was written earlier in the same call. Calls whose work overlaps on
 *     the GPU (concurrent streams, or several host threads) race on the
 *     array and corrupt each other's results: serialise them.
 */
#define STARQ_NOALLOC_SCRATCH_BYTES (32u << 20)
int sgat_linear_noalloc(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                        const float* a_m, const float* a_u, int hb, int d_sh, int d_m, int d_u,
                        const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                        const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias,
                        int N, int bits, void* Y, int y_dtype, void* stream);

/*
 * Glue of the quantised transformer blocks (not part of the paper's method:
 * Sec. 3 quantises the linears and the softmax-value product; the block
 * runs these element-wise passes between them, on this GPU like the rest).
 *
 * glue_add_rmsnorm -- residual add and RMSNorm of rows of K values:
 *   h = fl_T(X + R)                     (R = NULL: h = X)
 *   Y = fl_T(fl32(h * inv) * w),  inv = 1 / sqrt(mean_k(h^2) + eps)
 * with the sum of squares, mean and reciprocal square root in float32.
 *   X, R, h_out, Y  [L][K] of element type dtype (F16 or BF16), 16-byte
 *   aligned; R, h_out and Y may be NULL (h_out needs R; at least one of
 *   h_out, Y). h_out may be X or R (in place).
 *   w  [K] float32 gain (needed with Y).
 * Shapes: L >= 0, 8 <= K <= 20480, K % 8 == 0.
 *
 * glue_rope -- rotary position embedding, in place, on the first `heads`
 * heads of 128 channels of each row of QK [L][ld] (the query and key heads
 * of a fused QKV output): for i < 64 the pair (x_i, x_{i+64}) of a head is
 * rotated by the angle pos[token] * f_i, f_i = theta^(-2 i / 128) (float64,
 * rounded to float32), as (x_i c - x_{i+64} s, x_{i+64} c + x_i s) in
 * float32 with one rounding to dtype (the rotate-half form of the LLaMA and
 * Qwen2 families). pos: int32 [L] device array; theta > 1 (1e6 for Qwen2.5).
 * Shapes: L >= 0, heads >= 1, ld >= 128 heads.
 */
int glue_add_rmsnorm(const void* X, const void* R, int dtype, int L, int K, const float* w, float eps,
                     void* h_out, void* Y, void* stream);
int glue_rope(void* QK, int dtype, int L, int ld, int heads, const int32_t* pos, double theta, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* STARQ_H */
