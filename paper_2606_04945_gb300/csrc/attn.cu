// The quantised softmax-value product of an attention layer with TAC fused
// into its dequantisation epilogue (Sec. 3.3: Z_hat, the quantised
// counterpart of Softmax(Q K^T / sqrt(d_h)) V, compensated block-wise before
// the output projection; App. C, TAC inserted right after the
// softmax-value multiplication).
//
// The paper fixes neither the bit widths nor the granularity of the
// quantised softmax-value multiplication. Readings (stated with the C ABI):
//   P: unsigned 8-bit per query row. The row's largest probability 1 / l_i
//      maps to 255, so the code of p_ij is c_ij = rne(255 exp(s_ij - m_i))
//      and its scale 1 / (255 l_i).
//   V: signed 4-bit per channel, the activation quantiser along each column
//      (t_c = amax_c / 7, v_jc = rne(V_jc fl(7 / amax_c))).
//   Z_hat_ic = fl(fl(acc_ic * fl(1 / fl(255 l_i))) * t_c), with
//   acc_ic = sum_j c_ij v_jc exact (|acc| <= 255 * 7 * L < 2^24 in float32).
//   TAC: Z = Z_hat_h M_h^T + d_h per head (the head's 128 channels are one
//   block).
// Grouped-query attention: H query heads share Hkv key/value heads (H a
// multiple of Hkv); query head h reads key/value head h / (H / Hkv), whose
// V channels carry one set of codes and scales for the whole group.
// Element type T of Q, K, V and Z: fp16 or bf16. Q K^T runs in T; the P and
// V codes are integers held as fp16 (exact either way). The TAC product
// always runs on fp16 halves (Z_hat and M split into hi + lo, 2^-22
// relative): before the split Z_hat is scaled by an exact power of two
// 2^-k chosen per head from its largest V scale, so that its bound
// 16 * 7 max_c t_c lands in [2^13, 2^14) (inside fp16's range, with its
// full precision), and the TAC accumulator is scaled back by 2^k.
//
// attn_vquant_kernel   V codes per channel, written as fp16 values into
//                      Vt [128 H][L] (keys contiguous: the K-major B
//                      operand of P V^T), and the channel scales t.
// attn_pv_tac_kernel   persistent CTAs (at most one per SM) looping over the
//                      (128-query tile, head) items, each loading its own
//                      K / V tiles by TMA. 16 softmax / epilogue warps (a
//                      TMEM lane quarter times 32 of the 128 columns each),
//                      a TMA warp and one MMA warp, which issues every MMA
//                      (tcgen05 kind::f16 on one CTA, M = N = 128, K = 16)
//                      with the A operand (Q, P, Z_hat) in tensor memory and
//                      B (K, V, M) in shared memory.
//   prologue  the softmax warps copy the Q tile (loaded by TMA) into TMEM.
//   pass 1  S = Q K^T chunk by chunk (128 keys, two TMEM buffers); each
//           thread keeps the running maximum of its row's part of S.
//   pass 2  S again; each thread turns its 32 scores into
//           e = exp2(s c - m c), c = log2(e) / sqrt(d) (one fma, ex2.approx),
//           adds them to l (four partial sums) and writes the codes
//           rne(255 e), rounded exactly by a float32 bias whose low bits
//           are fp16 1024 + code, as fp16 over the S columns it has read.
//           The MMA warp then accumulates P V^T (exact integers) and
//           computes the scores two chunks ahead into the same buffer.
//   epilogue  Z_hat from the accumulator, split into fp16 hi + lo (Z_hat =
//           hi + lo to ~2^-22), written to TMEM as the A operands of the
//           TAC product Z_hi M_hi^T + Z_hi M_lo^T + Z_lo M_hi^T with M's
//           prepared halves (tac_prepare); + d; rounded to the I/O type and
//           stored by TMA (stores straight from registers, 64 bytes per
//           thread and row, measured slower).
// Shared memory holds only operand tiles and the output boxes: a ring of
// six 32 KB tiles streams each item's Q tile, pass-1 K chunks, pass-2 K and
// V chunks, M's two halves and then the slot of its output boxes, in the
// order they are used, running on into the next item.
// TMEM (512 columns): two S / P buffers, the P V^T accumulator (then the
// TAC accumulator), Q, and Z_hat's halves (see the column map below). The
// tensor pipe keeps almost no queue of issued MMAs, so it runs dry
// whenever the issuing thread is busy elsewhere (its waits and bookkeeping,
// slowed by the softmax warps that share its scheduler): the MMA warp
// therefore waits once per pass-2 chunk, on all of the chunk's barriers at
// once, and then issues its P V^T and the Q K^T two chunks ahead back to
// back. Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <type_traits>

#include "attn.cuh"
#include "common.cuh"

namespace starq {
namespace {

constexpr unsigned STATUS_TIMEOUT_ATTN = 1u << 4;
constexpr int ATT_SOFTMAX_WARPS = 16;           // 4 TMEM lane quarters x 4 column parts of 32
constexpr int ATT_SOFTMAX_THREADS = ATT_SOFTMAX_WARPS * 32;
constexpr int ATT_TMA_WARP = ATT_SOFTMAX_WARPS, ATT_MMA_WARP = ATT_SOFTMAX_WARPS + 1;
constexpr int ATT_THREADS = ATT_SOFTMAX_THREADS + 64;
constexpr int TILE_BYTES = ATTN_TILE * ATTN_D * 2;            // 128 x 128 fp16, two 128-byte-swizzled atoms
constexpr int ATOM_BYTES = TILE_BYTES / 2;
constexpr int ATT_SLOTS = 6;                                  // the ring of K / V tiles
constexpr int ATT_TILES_BYTES = ATT_SLOTS * TILE_BYTES;
// TMEM columns: S in two buffers of 128, the P V^T accumulator O and Q
// (16-bit, two per column). P overwrites the S it came from: the warp that
// read S columns [32 p, 32 p + 32) writes their 32 codes to columns
// [32 p, 32 p + 16), so no other warp's scores are touched and no wait is
// needed; the next Q K^T into that buffer is issued after the P V^T that
// reads P, and the MMAs of one thread run in issue order. After the passes
// the TAC accumulator takes the P V^T accumulator's columns (read out by
// then), Z_hat's high half the last 64 columns and its low half the upper
// half of the second S buffer. The first S buffer and the lower half of the
// second stay free, so the next item's Q K^T can follow the TAC product at
// once (the MMAs of one thread run in issue order, so it cannot overwrite
// Z_lo before the TAC product has read it).
constexpr uint32_t TM_S = 0, TM_O = 256, TM_Q = 384;
constexpr uint32_t TM_TAC = TM_O, TM_ZHI = 448, TM_ZLO = 192;

struct AttSm {
    uint64_t q_full, full[ATT_SLOTS], empty[ATT_SLOTS], s_full[2], s_empty[2];
    uint64_t pv_done, z_full, tac_done;
    uint32_t tmem_base;
    int abort;
    alignas(16) float xm[4][ATTN_TILE];            // row maxima / sums of the four column parts
    alignas(16) float tv[ATTN_D], dv[ATTN_D];      // the head's V channel scales and TAC offsets
};
constexpr size_t ATT_SMEM = ATT_TILES_BYTES + 1024 + sizeof(AttSm);

// log2(e) / sqrt(128): S (unscaled Q K^T) to base-2 exponents
constexpr float EXP_SCALE = (float)(1.4426950408889634 / 11.313708498984761);
// 1.5 * 2^23 + 0x6400: fma(255, e, ROUND_BIAS) rounds 255 e to the nearest
// integer n (the spacing of float32 there is 1; the bias is even, so ties
// go to even n) and leaves 0x6400 + n, the fp16 bits of 1024 + n, in the
// low half of the result's bits
constexpr float ROUND_BIAS = 12608512.f;

// 2^x by the PTX approximation (relative error about 2^-22; subnormal
// results flush to zero, where the code is 0 anyway)
// Two independent IEEE float32 operations on a register pair (the f32x2
// forms): each lane rounds exactly as the scalar fma / add would, with half
// the issue slots.
__device__ __forceinline__ float2 fma2_rn(float2 a, float2 b, float2 c) {
    float2 d;
    asm("{\n\t.reg .b64 A, B, C, D;\n\t"
        "mov.b64 A, {%2, %3};\n\tmov.b64 B, {%4, %5};\n\tmov.b64 C, {%6, %7};\n\t"
        "fma.rn.f32x2 D, A, B, C;\n\tmov.b64 {%0, %1}, D;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}
__device__ __forceinline__ float2 add2_rn(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 A, B, D;\n\t"
        "mov.b64 A, {%2, %3};\n\tmov.b64 B, {%4, %5};\n\t"
        "add.rn.f32x2 D, A, B;\n\tmov.b64 {%0, %1}, D;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// D (+)= A B^T, f16 inputs, f32 accumulate, A (128 rows, K-major: a row per
// TMEM lane, two elements per 32-bit column) in tensor memory, B in shared
// memory.
__device__ __forceinline__ void mma_f16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
    asm volatile("{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
                 "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}"
                 :: "r"(d_tmem), "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate) : "memory");
}


// Both phases complete (warp-uniform result). The two first queries are
// issued back to back, so their latencies overlap.
__device__ __forceinline__ bool mbar_wait2_bounded_warp(uint32_t b0, uint32_t p0, uint32_t b1, uint32_t p1,
                                                        volatile int* abort) {
    const bool d0 = mbar_try_wait(b0, p0);
    const bool d1 = mbar_try_wait(b1, p1);
    bool ok = true;
    if (!(d0 && d1)) ok = (d0 || mbar_wait_bounded(b0, p0, abort)) && (d1 || mbar_wait_bounded(b1, p1, abort));
    return __all_sync(0xffffffffu, ok);
}

// Three phases complete, the first queries back to back as above.
__device__ __forceinline__ bool mbar_wait3_bounded_warp(uint32_t b0, uint32_t p0, uint32_t b1, uint32_t p1, uint32_t b2,
                                                        uint32_t p2, volatile int* abort) {
    const bool d0 = mbar_try_wait(b0, p0);
    const bool d1 = mbar_try_wait(b1, p1);
    const bool d2 = mbar_try_wait(b2, p2);
    bool ok = true;
    if (!(d0 && d1 && d2))
        ok = (d0 || mbar_wait_bounded(b0, p0, abort)) && (d1 || mbar_wait_bounded(b1, p1, abort)) &&
             (d2 || mbar_wait_bounded(b2, p2, abort));
    return __all_sync(0xffffffffu, ok);
}

__device__ __forceinline__ float2 to_float2(__half2 h) { return __half22float2(h); }
__device__ __forceinline__ float2 to_float2(__nv_bfloat162 h) { return __bfloat1622float2(h); }

// Two floats -> T2 bits (round to nearest even), and a float rounded to T
// and back.
__device__ __forceinline__ uint32_t pack2(__half, float x, float y) {
    const __half2 v = __floats2half2_rn(x, y);
    return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ uint32_t pack2(__nv_bfloat16, float x, float y) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(x, y);
    return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ uint16_t bits_rn(__half, float x) { return __half_as_ushort(__float2half_rn(x)); }
__device__ __forceinline__ uint16_t bits_rn(__nv_bfloat16, float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }
__device__ __forceinline__ float from_bits(__half, uint16_t b) { return __half2float(__ushort_as_half(b)); }
__device__ __forceinline__ float from_bits(__nv_bfloat16, uint16_t b) { return __bfloat162float(__ushort_as_bfloat16(b)); }

__device__ __forceinline__ void named_sync_softmax() {
    asm volatile("bar.sync 1, %0;" :: "r"(ATT_SOFTMAX_THREADS) : "memory");
}

// One CTA per 16 channels: two threads per key row, each holding 8
// channels (16 bytes), 128 rows per sweep. Pass 1 takes the channel maxima,
// pass 2 (from L2) the codes, transposed through shared memory in tiles of
// 512 keys and written as 16-byte rows of Vt.
constexpr int VQ_CH = 16, VQ_KEYS = 512;

template <typename T>
__global__ void __launch_bounds__(256) attn_vquant_kernel(AttnArgs a) {
    using T2 = typename std::conditional<std::is_same<T, __half>::value, __half2, __nv_bfloat162>::type;
    __shared__ float red[8][VQ_CH];
    __shared__ float rcp[VQ_CH];
    __shared__ __align__(16) uint16_t tile[VQ_CH][VQ_KEYS + 8];
    const int c0 = blockIdx.x * VQ_CH;
    const int tid = threadIdx.x, hv = tid & 1, rr = tid >> 1, warp = tid >> 5, lane = tid & 31;
    const T* col = static_cast<const T*>(a.V) + c0 + 8 * hv;
    auto load = [&](int r) {
        return r < a.L ? __ldg(reinterpret_cast<const uint4*>(col + (size_t)r * a.ld)) : make_uint4(0u, 0u, 0u, 0u);
    };
    float m[8];
    #pragma unroll
    for (int k = 0; k < 8; ++k) m[k] = 0.f;
    for (int r0 = 0; r0 < a.L; r0 += VQ_KEYS) {
        uint4 v[4];
        #pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = load(r0 + rr + 128 * u);
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            const T2* p = reinterpret_cast<const T2*>(&v[u]);
            #pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 f = to_float2(p[k]);
                m[2 * k] = fmaxf(m[2 * k], fabsf(f.x));
                m[2 * k + 1] = fmaxf(m[2 * k + 1], fabsf(f.y));
            }
        }
    }
    // lanes of equal parity hold the same channels
    #pragma unroll
    for (int k = 0; k < 8; ++k)
        #pragma unroll
        for (int o = 2; o < 32; o <<= 1) m[k] = fmaxf(m[k], __shfl_xor_sync(0xffffffffu, m[k], o));
    if (lane < 2) {
        #pragma unroll
        for (int k = 0; k < 8; ++k) red[warp][8 * lane + k] = m[k];
    }
    __syncthreads();
    if (tid < VQ_CH) {
        float mm = 0.f;
        #pragma unroll
        for (int w = 0; w < 8; ++w) mm = fmaxf(mm, red[w][tid]);
        const bool nz = mm > 0.f;
        a.t[c0 + tid] = nz ? __fdiv_rn(mm, 7.f) : 0.f;
        rcp[tid] = nz ? __fdiv_rn(7.f, mm) : 0.f;
    }
    __syncthreads();
    float rc[8];
    #pragma unroll
    for (int k = 0; k < 8; ++k) rc[k] = rcp[8 * hv + k];
    for (int r0 = 0; r0 < a.L; r0 += VQ_KEYS) {
        uint4 v[4];
        #pragma unroll
        for (int u = 0; u < 4; ++u) v[u] = load(r0 + rr + 128 * u);
        #pragma unroll
        for (int u = 0; u < 4; ++u) {
            const T2* p = reinterpret_cast<const T2*>(&v[u]);
            #pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float2 f = to_float2(p[k]);
                tile[8 * hv + 2 * k][rr + 128 * u] = __half_as_ushort(__float2half_rn(rintf(__fmul_rn(f.x, rc[2 * k]))));
                tile[8 * hv + 2 * k + 1][rr + 128 * u] =
                    __half_as_ushort(__float2half_rn(rintf(__fmul_rn(f.y, rc[2 * k + 1]))));
            }
        }
        __syncthreads();
        const int segs = min(VQ_KEYS, a.L - r0) / 8;          // L is a multiple of 128
        for (int i = tid; i < VQ_CH * segs; i += 256) {
            const int c = i / segs, sg = i - c * segs;
            *reinterpret_cast<uint4*>(a.Vt + (size_t)(c0 + c) * a.L + r0 + 8 * sg) =
                *reinterpret_cast<const uint4*>(&tile[c][8 * sg]);
        }
        __syncthreads();
    }
}

// Persistent: a CTA takes the work items w = blockIdx.x + i gridDim.x (i =
// 0, 1, ...) of the nq H items (query tile w mod nq of head w / nq), so the
// CTAs running at one time share heads and their K / V tiles in L2. Every
// role loops over the same items, and every barrier's phase runs on across
// items.
//
// The ring's entries of item i are E = 3 nk + 4 in number, global index
// G = i E + 1 + u: u = -1 the item's Q tile (the softmax warps copy it into
// TMEM; the MMA warp gives the slot back once they have), u = 0 .. nk-1 the
// K chunks of pass 1, u = nk + 2j, nk + 2j + 1 chunk j's K and V for pass 2,
// u = 3 nk and 3 nk + 1 M's halves (one bulk copy each), u = 3 nk + 2 the
// output boxes (the TMA warp hands the free slot to the softmax warps with
// a plain arrive on its full barrier; they give it back after their stores
// have read it). Entry G uses slot G mod 6 for the (G / 6)-th time. So the
// next item's Q and K chunks stream in while this item's epilogue runs.
//
// TMEM across items: the next item's Q is written as soon as this item's
// P V^T has completed (its columns are then dead), before Z_hat, and the
// MMA warp issues the next item's first Q K^T right after this item's TAC
// product (see the column map above).
template <typename T>
__global__ void __launch_bounds__(ATT_THREADS, 1)
attn_pv_tac_kernel(AttnArgs a, const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_z) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    AttSm* sh = reinterpret_cast<AttSm*>(smem_raw + (base - raw) + ATT_TILES_BYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk = a.L / ATTN_TILE;                          // key chunks = query tiles of a head
    const int items = nk * a.H;
    const int my_items = blockIdx.x < (unsigned)items ? (items - 1 - (int)blockIdx.x) / (int)gridDim.x + 1 : 0;
    const int group = a.H / a.Hkv;
    volatile int* abort = &sh->abort;
    // (the lambdas capture by value: a local captured by reference lives in
    // memory and is reloaded after every asm with a memory clobber)
    auto B = [](const uint64_t& bar) { return smem_addr(&bar); };
    const int E = 3 * nk + 4;                                // ring entries per item
    // (entry indices stay below 2^31: at most 64 key chunks per head and
    // a few thousand items per CTA; 32-bit division by a constant is cheap)
    auto slot = [=](int g) { return base + ((uint32_t)g % ATT_SLOTS) * TILE_BYTES; };
    auto full_bar = [=](int g) { return B(sh->full[(uint32_t)g % ATT_SLOTS]); };
    auto empty_bar = [=](int g) { return B(sh->empty[(uint32_t)g % ATT_SLOTS]); };
    auto use_parity = [](int g) { return ((uint32_t)g / ATT_SLOTS) & 1u; };
    auto item_q0 = [=](int i) { return ((int)blockIdx.x + i * (int)gridDim.x) % nk * ATTN_TILE; };
    auto item_h = [=](int i) { return ((int)blockIdx.x + i * (int)gridDim.x) / nk; };
    // S buffer of Q K^T number it of item i (pass 1: it = 0 .. nk-1; pass
    // 2: it = nk + j; the two buffers alternate within each pass) and the
    // number of that buffer's earlier uses, counted over all items
    const int u0 = (nk + 1) / 2, u1 = nk / 2;                // uses of buffer 0 / 1 per pass
    auto sbuf = [=](int i, int it, int& b, int& n) {
        const int j = it < nk ? it : it - nk;
        b = j & 1;
        const int per = b == 0 ? u0 : u1;
        n = (j >> 1) + (it < nk ? 0 : per) + i * 2 * per;
    };

    if (threadIdx.x == 0) {
        mbar_init(B(sh->q_full), ATT_SOFTMAX_WARPS);
        for (int k = 0; k < ATT_SLOTS; ++k) {
            mbar_init(B(sh->full[k]), 1);
            mbar_init(B(sh->empty[k]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(B(sh->s_full[b]), 1);
            mbar_init(B(sh->s_empty[b]), ATT_SOFTMAX_WARPS);
        }
        mbar_init(B(sh->pv_done), 1);
        mbar_init(B(sh->z_full), ATT_SOFTMAX_WARPS);
        mbar_init(B(sh->tac_done), 1);
        sh->abort = 0;
        mbar_fence_init();
    }
    if (warp == ATT_MMA_WARP) {
        tmem_alloc(smem_addr(&sh->tmem_base), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sh->tmem_base;

    if (warp == ATT_TMA_WARP) {
        bool ok = true;
        for (int i = 0; i < my_items && ok; ++i) {
            const int h = item_h(i), hk = h / group;
            for (int ue = 0; ue < E && ok; ++ue) {
                const int g = i * E + ue;
                const int u = ue - 1;                            // -1: Q; from 0 the entries below
                if (!mbar_wait_bounded_warp(empty_bar(g), use_parity(g) ^ 1u, abort)) { ok = false; break; }
                const uint32_t dst = slot(g), fb = full_bar(g);
                if (elect_one()) {
                    if (u < 0) {                                 // the item's Q tile, as A of Q K^T
                        mbar_arrive_expect_tx(fb, TILE_BYTES);
                        tma_load_2d(dst, &tm_q, h * ATTN_D, item_q0(i), fb);
                        tma_load_2d(dst + ATOM_BYTES, &tm_q, h * ATTN_D + 64, item_q0(i), fb);
                    } else if (u < 3 * nk) {
                        mbar_arrive_expect_tx(fb, TILE_BYTES);
                        const int w = u - nk;
                        const void* tm = (w < 0 || (w & 1) == 0) ? (const void*)&tm_k : (const void*)&tm_v;
                        int x, y;
                        if (w < 0 || (w & 1) == 0) {             // K chunk: keys are the rows
                            x = hk * ATTN_D;
                            y = (w < 0 ? u : w >> 1) * ATTN_TILE;
                        } else {                                 // V chunk: channels are the rows
                            x = (w >> 1) * ATTN_TILE;
                            y = hk * ATTN_D;
                        }
                        tma_load_2d(dst, tm, x, y, fb);
                        tma_load_2d(dst + ATOM_BYTES, tm, x + 64, y, fb);
                    } else if (u < 3 * nk + 2) {                 // M_hi, M_lo of head h
                        const uint8_t* mp = static_cast<const uint8_t*>(a.Mp) +
                                            ((size_t)h * 2 + (size_t)(u - 3 * nk)) * TILE_BYTES;
                        mbar_arrive_expect_tx(fb, TILE_BYTES);
                        bulk_load(dst, mp, TILE_BYTES, fb);
                    } else {                                     // the output boxes' slot
                        mbar_arrive(fb);
                    }
                }
                __syncwarp();
            }
        }
        // every slot's last use has been given back, so no commit or arrive
        // lands after this CTA has exited
        const int G = my_items * E;
        for (int g = G - ATT_SLOTS; g < G && ok; ++g)
            if (g >= 0) ok = mbar_wait_bounded_warp(empty_bar(g), use_parity(g), abort);
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_ATTN); }
    } else if (warp == ATT_MMA_WARP) {
        // f32 D, N = 128 (bits 17..22), M = 128 (bits 24..28); A and B fp16
        // (P V^T: integer codes; TAC: fp16 halves) or of type T (Q K^T; bf16
        // sets the A and B format fields, bits 7..9 and 10..12)
        constexpr uint32_t IDESC_F16 = (1u << 4) | ((uint32_t)(ATTN_TILE >> 3) << 17) | ((uint32_t)(ATTN_TILE >> 4) << 24);
        constexpr uint32_t IDESC_T = IDESC_F16 | (std::is_same<T, __nv_bfloat16>::value ? ((1u << 7) | (1u << 10)) : 0u);
        // D (+)= A B^T over K = 128: A from TMEM at a_col (8 columns per K
        // step; for P, K steps 2p and 2p + 1 sit at 32 p and 32 p + 8), B
        // the K-major tile at bt (issued by the elected lane)
        auto mma_tile = [=](uint32_t d, uint32_t a_col, uint32_t bt, bool acc0, bool p_layout, uint32_t idesc) {
            // K step offsets added to the descriptor's start-address field
            // (addresses below 2^18, so the field never carries)
            const uint64_t bd = smem_desc_sw128(bt);
            const uint32_t ta = tmem + a_col;
            #pragma unroll
            for (int ks = 0; ks < ATTN_D / 16; ++ks) {
                const uint32_t koff = (uint32_t)(ks >> 2) * ATOM_BYTES + (uint32_t)(ks & 3) * 32;
                const uint32_t ac = p_layout ? 32u * (uint32_t)(ks >> 1) + 8u * (uint32_t)(ks & 1) : 8u * (uint32_t)ks;
                mma_f16_ts(d, ta + ac, bd + (uint64_t)(koff >> 4), idesc, (acc0 || ks > 0) ? 1u : 0u);
            }
        };
        bool ok = true;
        int tac_commits = 0;
        tc_fence_after();
        for (int i = 0; i < my_items && ok; ++i) {
            const int gq = i * E, g0 = gq + 1;
            // Q in TMEM: its ring slot is free again
            ok = mbar_wait_bounded_warp(B(sh->q_full), (uint32_t)(i & 1), abort);
            if (ok && elect_one()) mbar_arrive(empty_bar(gq));
            __syncwarp();
            // Q K^T number it, once its K tile has landed and the softmax
            // warps have read the S buffer's previous scores (s_empty)
            auto qk = [=](int it) -> bool {
                const int g = g0 + (it < nk ? it : nk + 2 * (it - nk));
                int b, n;
                sbuf(i, it, b, n);
                if (!mbar_wait2_bounded_warp(full_bar(g), use_parity(g), B(sh->s_empty[b]), (uint32_t)(n & 1) ^ 1u,
                                             abort))
                    return false;
                tc_fence_after();
                if (elect_one()) {
                    mma_tile(tmem + TM_S + b * ATTN_TILE, TM_Q, slot(g), false, false, IDESC_T);
                    tc_commit(empty_bar(g));
                    tc_commit(B(sh->s_full[b]));
                }
                __syncwarp();
                return true;
            };
            // Pass 2, one wait per chunk: P V^T of chunk j once its P is in
            // place over S(j) (the softmax warps arrive on the buffer's
            // s_empty after writing it) and its V tile has landed, then
            // Q K^T of chunk j + 2 into the same buffer once its K tile has
            // landed. Every wait of the issuing thread lets the tensor pipe
            // run dry, so the two products go out back to back behind a
            // single wait.
            auto step2 = [=](int j) -> bool {
                const int gv = g0 + nk + 2 * j + 1, gk = gv + 3;
                const bool more = j + 2 < nk;
                int b, n;
                sbuf(i, nk + j, b, n);
                if (!(more ? mbar_wait3_bounded_warp(B(sh->s_empty[b]), (uint32_t)(n & 1), full_bar(gv), use_parity(gv),
                                                     full_bar(gk), use_parity(gk), abort)
                           : mbar_wait2_bounded_warp(B(sh->s_empty[b]), (uint32_t)(n & 1), full_bar(gv), use_parity(gv),
                                                     abort)))
                    return false;
                tc_fence_after();
                if (elect_one()) {
                    mma_tile(tmem + TM_O, TM_S + b * ATTN_TILE, slot(gv), j > 0, true, IDESC_F16);
                    tc_commit(empty_bar(gv));
                    if (more) {
                        mma_tile(tmem + TM_S + b * ATTN_TILE, TM_Q, slot(gk), false, false, IDESC_T);
                        tc_commit(empty_bar(gk));
                        tc_commit(B(sh->s_full[b]));
                    }
                }
                __syncwarp();
                return true;
            };
            tc_fence_after();
            for (int it = 0; it < nk + 2 && it < 2 * nk && ok; ++it) ok = qk(it);   // pass 1, then two chunks ahead
            for (int j = 0; j < nk && ok; ++j) ok = step2(j);
            if (elect_one()) tc_commit(B(sh->pv_done));
            __syncwarp();
            const int gm = g0 + 3 * nk;               // M_hi; M_lo at gm + 1
            ok = ok && mbar_wait2_bounded_warp(B(sh->z_full), (uint32_t)(i & 1), full_bar(gm), use_parity(gm), abort) &&
                 mbar_wait_bounded_warp(full_bar(gm + 1), use_parity(gm + 1), abort);
            tc_fence_after();
            if (elect_one()) {
                if (ok) {
                    mma_tile(tmem + TM_TAC, TM_ZHI, slot(gm), false, false, IDESC_F16);       // Z_hi M_hi^T
                    mma_tile(tmem + TM_TAC, TM_ZHI, slot(gm + 1), true, false, IDESC_F16);    // + Z_hi M_lo^T
                    mma_tile(tmem + TM_TAC, TM_ZLO, slot(gm), true, false, IDESC_F16);        // + Z_lo M_hi^T
                    tc_commit(empty_bar(gm));
                    tc_commit(empty_bar(gm + 1));
                }
                tc_commit(B(sh->tac_done));
            }
            __syncwarp();
            ++tac_commits;
        }
        if (tac_commits > 0 && lane == 0) {
            // every MMA of this thread has completed before TMEM is released
            volatile int never = 0;
            if (!mbar_wait_bounded(B(sh->tac_done), (uint32_t)((tac_commits - 1) & 1), &never)) ok = false;
        }
        __syncwarp();
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_ATTN); }
    } else {
        const int quarter = warp & 3, part = warp >> 2, col = part * 32;
        const int row = quarter * 32 + lane;                // query within the tile (TMEM lane)
        const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
        bool ok = true;
        uint32_t r[32];
        // the query row's 32 channels of this part, from item i's Q tile in
        // its ring slot (two 64-channel halves of 128-byte rows, the 16-byte
        // chunks of row r XOR-ed with r mod 8), into TMEM (A of Q K^T)
        auto put_q = [=](int i) -> bool {
            const int gq = i * E;
            if (!mbar_wait_bounded_warp(full_bar(gq), use_parity(gq), abort)) return false;
            const uint32_t src = slot(gq) + (uint32_t)(part >> 1) * ATOM_BYTES + (uint32_t)row * 128u;
            uint32_t qv[16];
            #pragma unroll
            for (int k = 0; k < 4; ++k) {
                const uint4 w = ld_shared_v4(src + ((uint32_t)(((part & 1) * 4 + k) ^ (row & 7)) << 4));
                qv[4 * k] = w.x;
                qv[4 * k + 1] = w.y;
                qv[4 * k + 2] = w.z;
                qv[4 * k + 3] = w.w;
            }
            tmem_st_32x32b_x16(tl + TM_Q + part * 16, qv);
            tmem_st_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(sh->q_full));
            return true;
        };
        if (my_items > 0) ok = put_q(0);
        // Every softmax warp runs every item and every named barrier; after a
        // failed wait it only skips the work.
        for (int i = 0; i < my_items; ++i) {
            const int q0 = item_q0(i), h = item_h(i), hk = h / group;
            const int g0 = i * E + 1;
            const uint32_t ip = (uint32_t)(i & 1);
            if (threadIdx.x >= ATTN_D && threadIdx.x < 2 * ATTN_D) {
                const int c = threadIdx.x - ATTN_D;
                sh->dv[c] = a.d != nullptr ? a.d[h * ATTN_D + c] : 0.f;
            }
            // pass 1: row maxima
            float mx = -INFINITY;
            for (int it = 0; it < nk && ok; ++it) {
                int b, n;
                sbuf(i, it, b, n);
                if (!mbar_wait_bounded_warp(B(sh->s_full[b]), (uint32_t)(n & 1), abort)) { ok = false; break; }
                tc_fence_after();
                tmem_ld_32x32b_x32(tl + TM_S + b * ATTN_TILE + col, r);
                tmem_ld_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(B(sh->s_empty[b]));
                #pragma unroll
                for (int k = 0; k < 32; ++k) mx = fmaxf(mx, __uint_as_float(r[k]));
            }
            if (threadIdx.x < ATTN_D) sh->tv[threadIdx.x] = a.t[hk * ATTN_D + threadIdx.x];  // V channel scales
            sh->xm[part][row] = mx;
            named_sync_softmax();
            mx = fmaxf(fmaxf(sh->xm[0][row], sh->xm[1][row]), fmaxf(sh->xm[2][row], sh->xm[3][row]));
            named_sync_softmax();
            // pass 2: probabilities, their codes and the row sums
            // partial row sums, four independent chains held as two pairs:
            // (l0, l2) and (l1, l3), l0 + l1 over even-k scores, l2 + l3 odd
            float2 lpa = make_float2(0.f, 0.f), lpb = make_float2(0.f, 0.f);
            // the exponent as one fma: s c - m c differs from (s - m) c by an
            // ulp of m c at most, ~1e-6 in e at |m| <= 100 (the codes' rounding
            // decisions move only within 3e-4 of a half-integer)
            const float mxc = __fmul_rn(mx, EXP_SCALE);
            for (int j = 0; j < nk && ok; ++j) {
                int b, n;
                sbuf(i, nk + j, b, n);
                if (!mbar_wait_bounded_warp(B(sh->s_full[b]), (uint32_t)(n & 1), abort)) { ok = false; break; }
                tc_fence_after();
                tmem_ld_32x32b_x32(tl + TM_S + b * ATTN_TILE + col, r);
                tmem_ld_wait();
                // e = 2^((s - m) log2(e) / sqrt(d)); the code n = rne(255 e) in
                // one rounding: the low halves of fma(255, e, ROUND_BIAS) are the
                // fp16 values 1024 + n of two codes, and 1024 is subtracted
                // exactly in fp16
                uint32_t packed[16];
                const __half2 minus1024 = __float2half2_rn(-1024.f);
                const float2 c2 = make_float2(EXP_SCALE, EXP_SCALE), nm2 = make_float2(-mxc, -mxc);
                const float2 q2 = make_float2(255.f, 255.f), bias2 = make_float2(ROUND_BIAS, ROUND_BIAS);
                #pragma unroll
                for (int k = 0; k < 32; k += 2) {
                    const float2 t = fma2_rn(make_float2(__uint_as_float(r[k]), __uint_as_float(r[k + 1])), c2, nm2);
                    const float2 e = make_float2(ex2_approx(t.x), ex2_approx(t.y));
                    if ((k >> 1) & 1) lpb = add2_rn(lpb, e);
                    else lpa = add2_rn(lpa, e);
                    const float2 u = fma2_rn(e, q2, bias2);
                    const uint32_t biased = prmt(__float_as_uint(u.x), __float_as_uint(u.y), 0x5410u);   // {1024 + n0, 1024 + n1}
                    const __half2 hc = __hadd2(*reinterpret_cast<const __half2*>(&biased), minus1024);
                    packed[k / 2] = *reinterpret_cast<const uint32_t*>(&hc);
                }
                if (a.dbg_codes != nullptr) {
                    uint8_t* dc = a.dbg_codes + ((size_t)h * a.L + q0 + row) * a.L + j * ATTN_TILE + col;
                    #pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        dc[2 * k] = (uint8_t)__half2float(__ushort_as_half((uint16_t)(packed[k] & 0xFFFFu)));
                        dc[2 * k + 1] = (uint8_t)__half2float(__ushort_as_half((uint16_t)(packed[k] >> 16)));
                    }
                }
                // P over the S columns this warp has read
                tmem_st_32x32b_x16(tl + TM_S + b * ATTN_TILE + col, packed);
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(B(sh->s_empty[b]));
            }
            sh->xm[part][row] = (lpa.x + lpb.x) + (lpa.y + lpb.y);
            named_sync_softmax();
            const float l = (sh->xm[0][row] + sh->xm[1][row]) + (sh->xm[2][row] + sh->xm[3][row]);
            const float sp = __fdiv_rn(1.f, __fmul_rn(255.f, l));
            // the head's power-of-two TAC scale: |Z_hat| <= 16 * 7 max_c t_c (the
            // codes of a row sum to at most twice 255 l), brought into [2^13, 2^14)
            float tmax = 0.f;
            #pragma unroll
            for (int c = lane; c < ATTN_D; c += 32) tmax = fmaxf(tmax, sh->tv[c]);
            #pragma unroll
            for (int m = 16; m > 0; m >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, m));
            const int zk = tmax > 0.f ? ilogbf(112.f * tmax) - 13 : 0;
            const float zscale = ldexpf(1.f, -zk), zunscale = ldexpf(1.f, zk);
            if (a.dbg_l != nullptr && part == 0) a.dbg_l[(size_t)h * a.L + q0 + row] = l;
            // every MMA reading Q has completed (pv_done), so the next item's
            // Q goes in first, for its Q K^T right after this item's TAC
            // product
            ok = ok && mbar_wait_bounded_warp(B(sh->pv_done), ip, abort);
            if (ok && i + 1 < my_items) ok = put_q(i + 1);
            // epilogue 1: Z_hat = (acc sp) t as fp16 hi + lo, the A operands of
            // the TAC product, into TMEM
            if (ok) {
                tc_fence_after();
                tmem_ld_32x32b_x32(tl + TM_O + col, r);
                tmem_ld_wait();
                if (a.dbg_acc != nullptr) {
                    int32_t* da = a.dbg_acc + ((size_t)h * a.L + q0 + row) * ATTN_D + col;
                    #pragma unroll
                    for (int k = 0; k < 32; ++k) da[k] = __float2int_rn(__uint_as_float(r[k]));
                }
                uint32_t hi[16], lo[16];
                #pragma unroll
                for (int k = 0; k < 32; k += 4) {
                    const float4 t4 = *reinterpret_cast<const float4*>(&sh->tv[col + k]);
                    const float tk[4] = {t4.x, t4.y, t4.z, t4.w};
                    #pragma unroll
                    for (int u = 0; u < 4; u += 2) {
                        const float z0 = __fmul_rn(__fmul_rn(__fmul_rn(__uint_as_float(r[k + u]), sp), tk[u]), zscale);
                        const float z1 = __fmul_rn(__fmul_rn(__fmul_rn(__uint_as_float(r[k + u + 1]), sp), tk[u + 1]), zscale);
                        const __half2 zh = __floats2half2_rn(z0, z1);
                        const float2 zb = __half22float2(zh);
                        const __half2 zl = __floats2half2_rn(__fsub_rn(z0, zb.x), __fsub_rn(z1, zb.y));
                        hi[(k + u) / 2] = *reinterpret_cast<const uint32_t*>(&zh);
                        lo[(k + u) / 2] = *reinterpret_cast<const uint32_t*>(&zl);
                    }
                }
                tmem_st_32x32b_x16(tl + TM_ZHI + part * 16, hi);
                tmem_st_32x32b_x16(tl + TM_ZLO + part * 16, lo);
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(B(sh->z_full));
            }
            // epilogue 2: + d, rounded to T, TMA store from the ring slot of
            // entry 3 nk + 2
            const int go = g0 + 3 * nk + 2;
            ok = ok && mbar_wait2_bounded_warp(B(sh->tac_done), ip, full_bar(go), use_parity(go), abort);
            if (ok) {
                tc_fence_after();
                tmem_ld_32x32b_x32(tl + TM_TAC + col, r);
                tmem_ld_wait();
                const uint32_t box = slot(go) + (uint32_t)warp * 2048;
                const bool add_d = a.d != nullptr;
                #pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const float4 d0 = *reinterpret_cast<const float4*>(&sh->dv[col + 8 * g]);
                    const float4 d1 = *reinterpret_cast<const float4*>(&sh->dv[col + 8 * g + 4]);
                    const float dk[8] = {d0.x, d0.y, d0.z, d0.w, d1.x, d1.y, d1.z, d1.w};
                    uint32_t w[4];
                    #pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int k = 8 * g + 2 * u;
                        float y0 = __fmul_rn(__uint_as_float(r[k]), zunscale), y1 = __fmul_rn(__uint_as_float(r[k + 1]), zunscale);
                        if (add_d) {
                            y0 = __fadd_rn(y0, dk[2 * u]);
                            y1 = __fadd_rn(y1, dk[2 * u + 1]);
                        }
                        w[u] = pack2(T(), y0, y1);
                    }
                    st_shared_v4(box + lane * 64 + 16 * (g ^ ((lane >> 1) & 3)), w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tm_z, h * ATTN_D + col, q0 + quarter * 32, box);
                    bulk_commit();
                    bulk_wait_read0();           // the box has been read; the write completes with the grid
                }
                __syncwarp();
            }
            // item boundary: every box of this slot has been read, and dv, tv
            // and xm are free for the next item
            named_sync_softmax();
            if (ok && threadIdx.x == 0) mbar_arrive(empty_bar(go));
        }
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_ATTN); }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == ATT_MMA_WARP) tmem_dealloc(tmem, 512);
}

bool encode_2d(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint64_t row_elems,
               uint32_t box_rows, uint32_t box_cols, CUtensorMapSwizzle swz,
               CUtensorMapDataType type = CU_TENSOR_MAP_DATA_TYPE_FLOAT16) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {row_elems * 2};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, type, 2, const_cast<void*>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

template <typename T>
cudaError_t launch_pv_tac(const AttnArgs& a, cudaStream_t stream) {
    const int C = ATTN_D * a.H, Ckv = ATTN_D * a.Hkv;
    const CUtensorMapDataType io = std::is_same<T, __half>::value ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                                                   : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
    CUtensorMap tq, tk, tv, tz;
    if (!encode_2d(&tq, a.Q, (uint64_t)a.L, (uint64_t)C, (uint64_t)a.ld, ATTN_TILE, 64, CU_TENSOR_MAP_SWIZZLE_128B, io) ||
        !encode_2d(&tk, a.K, (uint64_t)a.L, (uint64_t)Ckv, (uint64_t)a.ld, ATTN_TILE, 64, CU_TENSOR_MAP_SWIZZLE_128B, io) ||
        !encode_2d(&tv, a.Vt, (uint64_t)Ckv, (uint64_t)a.L, (uint64_t)a.L, ATTN_D, 64, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_2d(&tz, a.Z, (uint64_t)a.L, (uint64_t)C, (uint64_t)C, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B, io))
        return cudaErrorInvalidValue;
    static DeviceCache<int> attr;
    int done = 0;
    cudaError_t e = attr.get(&done, [](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(attn_pv_tac_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ATT_SMEM);
    });
    if (e != cudaSuccess) return e;
    attn_vquant_kernel<T><<<Ckv / VQ_CH, 256, 0, stream>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // persistent CTAs, one per SM at most, each with the same number of
    // items (the last CTAs one fewer)
    const int items = a.L / ATTN_TILE * a.H;
    const int per_cta = (items + num_sms() - 1) / num_sms();
    const int grid = (items + per_cta - 1) / per_cta;
    attn_pv_tac_kernel<T><<<grid, ATT_THREADS, ATT_SMEM, stream>>>(a, tq, tk, tv, tz);
    return cudaGetLastError();
}

cudaError_t launch_attention_pv_tac(const AttnArgs& a, cudaStream_t stream) {
    return a.dtype == STARQ_BF16 ? launch_pv_tac<__nv_bfloat16>(a, stream) : launch_pv_tac<__half>(a, stream);
}

}  // namespace starq
