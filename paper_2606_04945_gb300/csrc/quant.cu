// SGAT activation transform + per-row symmetric int4 quantisation.
//
// Per row (a token for Q_a, an output channel for Q_w); Sec. 3.2 Eq. 11 with
// P = diag(a_s) H_hb, Sec. 3.1 Eq. 2:
//   v = fl32(x * a_s)                      state picked by the row's mask bit
//   v = v H_hb                             fast Walsh-Hadamard transform
//   v = v * gate_s                          binary subspace gate (Eq. 9)
//   v = fl32(v * post_scale)               1/hb on the weight side (Eq. 12)
//   amax = max |v|; s = amax / qmax; r = qmax / amax; q = rne(v * r)
// The transform is the butterfly network of the fast Walsh-Hadamard
// transform in stage order h = 1, 2, 4, ..., hb/2, each butterfly
// (a, b) -> (a + b, a - b) in float32 round-to-nearest; every float operation
// is an explicit round-to-nearest intrinsic, so nothing is contracted into an
// FMA and the values match the reference network bit for bit. With qmax = 7
// no clamp is needed: |fl(v * r)| <= 7 (1 + 2^-24)^2 < 7.5 (likewise 127.5
// for qmax = 127).
//
// Storage by code width. qmax <= 7 (4-bit): Xq packs two codes per byte and
// Xe holds each code as an E4M3 byte [rows][K]. qmax = 127 (8-bit, the W8A8
// setting of Tab. 5): Xq holds one code per byte (two's complement) and Xe
// [rows][K] each code as an fp16 number (exact: |c| <= 127), the operand of
// the 8-bit GEMM.
//
// Asymmetric mode (a.asym, Eq. 2-4, activations): per row X_max = max(max v,
// 0) and -X_min = max(max -v, 0); s = fl(fl(X_max - X_min) / qmax), r =
// fl(qmax / fl(X_max - X_min)), z = rne(fl(-X_min r)) in [0, qmax], codes
// clamp(rne(fl(v r)) + z, 0, qmax) (qmax = 15: unsigned nibbles in Xq, E4M3
// bytes in Xe, whose rows are K + 128 long and end in 128 bytes of E4M3(-z):
// with weight rows ending in E4M3 values that sum to sum_k q_w, the 4-bit
// GEMM over K + 128 then gives sum_k (q_a - z) q_w exactly).
//
// Work split: a warp owns a chunk of C = 32 E consecutive elements of a row
// (C = 1024 when hb >= 1024, else C = 512 holding 512 / hb Hadamard blocks).
// In layout A lane l holds elements E l .. E l + E - 1, so stages h < E are
// butterflies between registers of one thread. One transpose through shared
// memory (layout B: lane l holds elements l + 32 i) makes the stages
// 32 <= h < C register-local too; a transpose back gives each lane E
// contiguous values again. Stages h >= C (hb = 2048, 4096) pair chunks held
// by different warps of the row and exchange through shared memory.
//
// A row takes min(K / C, 8) warps, each keeping up to NC chunks in
// registers; short rows share a CTA of 8 warps. amax is reduced across a
// row's warps through shared memory.
#include "common.cuh"

namespace starq {
namespace {

template <typename T> struct In;
template <> struct In<__half> {
    template <int E>
    static __device__ __forceinline__ void load(const __half* p, float (&v)[E]) {
        const uint4* q = reinterpret_cast<const uint4*>(p);
        #pragma unroll
        for (int u = 0; u < E / 8; ++u) {
            uint4 w = __ldg(q + u);
            const __half2* h = reinterpret_cast<const __half2*>(&w);
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                float2 f = __half22float2(h[j]);
                v[8 * u + 2 * j] = f.x;
                v[8 * u + 2 * j + 1] = f.y;
            }
        }
    }
};
template <> struct In<__nv_bfloat16> {
    template <int E>
    static __device__ __forceinline__ void load(const __nv_bfloat16* p, float (&v)[E]) {
        const uint4* q = reinterpret_cast<const uint4*>(p);
        #pragma unroll
        for (int u = 0; u < E / 8; ++u) {
            uint4 w = __ldg(q + u);
            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&w);
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                float2 f = __bfloat1622float2(h[j]);
                v[8 * u + 2 * j] = f.x;
                v[8 * u + 2 * j + 1] = f.y;
            }
        }
    }
};
template <> struct In<float> {
    template <int E>
    static __device__ __forceinline__ void load(const float* p, float (&v)[E]) {
        const float4* q = reinterpret_cast<const float4*>(p);
        #pragma unroll
        for (int u = 0; u < E / 4; ++u) {
            float4 w = __ldg(q + u);
            v[4 * u] = w.x; v[4 * u + 1] = w.y; v[4 * u + 2] = w.z; v[4 * u + 3] = w.w;
        }
    }
};

__device__ __forceinline__ void butterfly(float& lo, float& hi) {
    const float a = lo, b = hi;
    lo = __fadd_rn(a, b);
    hi = __fsub_rn(a, b);
}

// Butterflies between registers i and i + s for every i with (i & s) == 0,
// for s = s_lo, 2 s_lo, ... while s < s_end.
template <int E>
__device__ __forceinline__ void inlane_stages(float (&v)[E], int s_lo, int s_end) {
    #pragma unroll
    for (int s = 1; s < E; s <<= 1) {
        if (s >= s_lo && s < s_end) {
            #pragma unroll
            for (int i = 0; i < E; ++i)
                if ((i & s) == 0) butterfly(v[i], v[i + s]);
        }
    }
}

// Shared-buffer index of chunk element e: one padding float after every E
// elements. Layout A (lane stride E + 1, odd) and layout B (consecutive
// lanes, consecutive words) are then both free of bank conflicts, and every
// access is a per-lane base plus a compile-time offset.
template <int E>
__device__ __forceinline__ int pad_idx(int e) { return e + e / E; }

// Full transform of one chunk held in layout A; `buf` is this warp's
// 32 E-float shared buffer.
template <int E>
__device__ __forceinline__ void chunk_fwht(float (&v)[E], int hb, int lane, float* buf) {
    inlane_stages<E>(v, 1, hb < E ? hb : E);                  // h = 1 .. min(hb, E)/2
    if (hb <= E) return;
    if (E < 32) {                                            // h = E .. 16 across lanes
        #pragma unroll
        for (int h = E; h < 32; h <<= 1) {
            if (h < hb) {
                const int m = h / E;
                const float sgn = (lane & m) ? -1.f : 1.f;
                #pragma unroll
                for (int i = 0; i < E; ++i) {
                    const float o = __shfl_xor_sync(0xffffffffu, v[i], m);
                    // lower lane: v + o; upper lane: o - v (the product by -1 is exact)
                    v[i] = __fmaf_rn(sgn, v[i], o);
                }
            }
        }
    }
    if (hb <= 32) return;
    // layout A -> B
    float* a_base = buf + (E + 1) * lane;      // = buf + pad_idx(E * lane)
    #pragma unroll
    for (int i = 0; i < E; ++i) a_base[i] = v[i];
    __syncwarp();
    #pragma unroll
    for (int i = 0; i < E; ++i) v[i] = buf[pad_idx<E>(lane + 32 * i)];
    // stages h = max(E, 32) .. hb/2: register distance h / 32 in layout B
    inlane_stages<E>(v, (E > 32 ? E : 32) / 32, hb / 32);
    __syncwarp();
    #pragma unroll
    for (int i = 0; i < E; ++i) buf[pad_idx<E>(lane + 32 * i)] = v[i];
    __syncwarp();
    #pragma unroll
    for (int i = 0; i < E; ++i) v[i] = a_base[i];
    __syncwarp();
}

// Eight 8-bit codes -> their bytes (two's complement, code k in byte k) and
// the same codes as fp16 numbers (exact), code k in half k.
__device__ __forceinline__ void codes8(const int* q, uint2& bytes, uint4& f16) {
    uint32_t b0 = 0, b1 = 0;
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        b0 |= (uint32_t)(q[k] & 0xFF) << (8 * k);
        b1 |= (uint32_t)(q[k + 4] & 0xFF) << (8 * k);
    }
    bytes = make_uint2(b0, b1);
    uint32_t h[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        const __half2 p = __floats2half2_rn((float)q[2 * k], (float)q[2 * k + 1]);
        h[k] = *reinterpret_cast<const uint32_t*>(&p);
    }
    f16 = make_uint4(h[0], h[1], h[2], h[3]);
}

// Eight codes in [0, 15] -> E4M3 bytes (byte k = code k).
__device__ __forceinline__ uint2 e4m3_of8(const int* q) {
    uint16_t h[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k)          // upper byte from the first operand
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(h[k]) : "f"((float)q[2 * k + 1]), "f"((float)q[2 * k]));
    return make_uint2((uint32_t)h[0] | ((uint32_t)h[1] << 16), (uint32_t)h[2] | ((uint32_t)h[3] << 16));
}

// The zero-point columns of an asymmetric row: 128 bytes of E4M3(-z) after
// its K codes, eight threads of 16 bytes each (t = 0 .. 7).
__device__ __forceinline__ void store_zero_point_columns(uint8_t* row_end, int z, int t) {
    uint16_t h;
    const float m = (float)(-z);
    asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %1;" : "=h"(h) : "f"(m));
    const uint32_t w = (uint32_t)h | ((uint32_t)h << 16);
    reinterpret_cast<uint4*>(row_end)[t] = make_uint4(w, w, w, w);
}

// Eight codes (int, |q| <= 7) -> packed nibbles, code k in bits 4k..4k+3.
__device__ __forceinline__ uint32_t pack8(const int* q) {
    uint32_t w = 0;
    #pragma unroll
    for (int k = 0; k < 8; ++k) w |= (uint32_t)(q[k] & 0xF) << (4 * k);
    return w;
}

// Up to 8 warps per row, or up to 20 when hb <= C (E = 16, at most two
// chunks per warp; no stage crosses warps then).
template <int E, int NC, typename Tin>
__global__ void __launch_bounds__(E == 16 && NC <= 2 ? 640 : 256)
sgat_quant_kernel(QuantArgs a, int warps_per_row, int rows_per_cta) {
    extern __shared__ float qsm[];
    constexpr int C = 32 * E;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int wr = warp % warps_per_row;                 // warp index within its row
    const int row = blockIdx.x * rows_per_cta + warp / warps_per_row;
    float* buf = qsm + warp * (C + 32);
    float* red = qsm + (blockDim.x >> 5) * (C + 32);     // [32] partial amax, [32] partial -min
    const bool row_ok = row < a.L;
    const int K = a.K;
    const int nchunks = (K + C - 1) / C;   // a partial last chunk only when hb < 512

    const bool masked = row_ok && a.mask != nullptr && a.mask[row] != 0;
    const float* sm = masked ? a.a_m : a.a_u;
    // Active coordinates of the row's state (Eq. 9): masked rows keep
    // [0, d_sh + d_m), unmasked rows keep [0, d_sh) and [d_sh + d_m, K).
    const int own_lo = masked ? a.d_sh : a.d_sh + a.d_m;
    const int own_hi = masked ? a.d_sh + a.d_m : K;
    const Tin* X = static_cast<const Tin*>(a.X) + (size_t)(row_ok ? row : 0) * K;

    float v[NC][E];
    float amax = 0.f, nmin = 0.f;                        // asym: X_max and -X_min
    #pragma unroll
    for (int j = 0; j < NC; ++j) {
        const int c = wr + j * warps_per_row;
        const int lo = c * C + E * lane;                 // first element of this lane
        // lanes lie wholly inside or outside the row: E | K when hb < 512
        const bool live = c < nchunks && row_ok && lo < K;
        if (live) {
            In<Tin>::template load<E>(X + lo, v[j]);
            if (sm != nullptr) {
                const float4* s4 = reinterpret_cast<const float4*>(sm + lo);
                #pragma unroll
                for (int u = 0; u < E / 4; ++u) {
                    const float4 w = __ldg(s4 + u);
                    v[j][4 * u] = __fmul_rn(v[j][4 * u], w.x);
                    v[j][4 * u + 1] = __fmul_rn(v[j][4 * u + 1], w.y);
                    v[j][4 * u + 2] = __fmul_rn(v[j][4 * u + 2], w.z);
                    v[j][4 * u + 3] = __fmul_rn(v[j][4 * u + 3], w.w);
                }
            }
        } else {
            #pragma unroll
            for (int i = 0; i < E; ++i) v[j][i] = 0.f;
        }
        if (c < nchunks) chunk_fwht<E>(v[j], a.hb, lane, buf);   // warp-uniform condition
        // Stages h = C .. hb/2 pair chunk c with chunk c ^ (h / C), held by
        // warp wr ^ (h / C) of the same row in the same round j (the warp
        // count of a row is a multiple of hb / C). Exchange in layout A
        // through the warps' padded buffers; all warps of the CTA take part.
        for (int m = 1; m * C < a.hb; m <<= 1) {
            float* mine = buf + (E + 1) * lane;
            const float* other = qsm + (warp ^ m) * (C + 32) + (E + 1) * lane;
            #pragma unroll
            for (int i = 0; i < E; ++i) mine[i] = v[j][i];
            __syncthreads();
            const bool upper = (wr & m) != 0;
            #pragma unroll
            for (int i = 0; i < E; ++i) {
                const float o = other[i];
                v[j][i] = upper ? __fsub_rn(o, v[j][i]) : __fadd_rn(v[j][i], o);
            }
            __syncthreads();
        }
        // gate: whole-lane decisions first, per element only where a lane
        // straddles a subspace boundary
        const bool all_keep = (lo + E <= a.d_sh) || (lo >= own_lo && lo + E <= own_hi);
        if (!all_keep) {
            #pragma unroll
            for (int i = 0; i < E; ++i) {
                const int e = lo + i;
                if (!(e < a.d_sh || (e >= own_lo && e < own_hi))) v[j][i] = 0.f;
            }
        }
        if (a.post_scale != 1.f) {
            #pragma unroll
            for (int i = 0; i < E; ++i) v[j][i] = __fmul_rn(v[j][i], a.post_scale);
        }
        if (a.asym) {
            #pragma unroll
            for (int i = 0; i < E; ++i) {
                amax = fmaxf(amax, v[j][i]);
                nmin = fmaxf(nmin, -v[j][i]);
            }
        } else {
            #pragma unroll
            for (int i = 0; i < E; ++i) amax = fmaxf(amax, fabsf(v[j][i]));
        }
        if (a.v_dbg != nullptr && live) {
            float4* d4 = reinterpret_cast<float4*>(a.v_dbg + (size_t)row * K + lo);
            #pragma unroll
            for (int u = 0; u < E / 4; ++u)
                d4[u] = make_float4(v[j][4 * u], v[j][4 * u + 1], v[j][4 * u + 2], v[j][4 * u + 3]);
        }
    }
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) {
        amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, m));
        nmin = fmaxf(nmin, __shfl_xor_sync(0xffffffffu, nmin, m));
    }
    if (warps_per_row > 1) {
        if (lane == 0) {
            red[warp] = amax;
            red[32 + warp] = nmin;
        }
        __syncthreads();
        amax = 0.f;
        nmin = 0.f;
        const int first = warp - wr;                     // first warp of this row
        for (int w = 0; w < warps_per_row; ++w) {
            amax = fmaxf(amax, red[first + w]);
            nmin = fmaxf(nmin, red[32 + first + w]);
        }
    }
    if (!row_ok) return;

    const float qmax = (float)a.qmax;
    const float range = a.asym ? __fadd_rn(amax, nmin) : amax;     // X_max - X_min, or amax
    const bool nz = range > 0.f;
    const float s = nz ? __fdiv_rn(range, qmax) : 0.f;
    const float r = nz ? __fdiv_rn(qmax, range) : 0.f;
    const int zp = a.asym ? min(max(__float2int_rn(__fmul_rn(nmin, r)), 0), a.qmax) : 0;
    if (wr == 0 && lane == 0) {
        a.s[row] = s;
        if (a.asym) a.z[row] = zp;
    }
    if (a.asym && a.Xe != nullptr && wr == 0 && lane < 8)
        store_zero_point_columns(a.Xe + (size_t)row * (K + 128) + K, zp, lane);
    #pragma unroll
    for (int j = 0; j < NC; ++j) {
        const int c = wr + j * warps_per_row;
        const int lo = c * C + E * lane;
        if (c >= nchunks || lo >= K) continue;
        if (a.asym) {                    // codes in [0, qmax]: unsigned nibbles and E4M3 bytes
            #pragma unroll
            for (int u = 0; u < E / 8; ++u) {
                int q[8];
                #pragma unroll
                for (int k = 0; k < 8; ++k)
                    q[k] = min(max(__float2int_rn(__fmul_rn(v[j][8 * u + k], r)) + zp, 0), a.qmax);
                if (a.Xq != nullptr) *reinterpret_cast<uint32_t*>(a.Xq + (size_t)row * (K / 2) + lo / 2 + 4 * u) = pack8(q);
                if (a.Xe != nullptr) *reinterpret_cast<uint2*>(a.Xe + (size_t)row * (K + 128) + lo + 8 * u) = e4m3_of8(q);
            }
            continue;
        }
        if (a.qmax > 15) {               // 8-bit codes: bytes and fp16
            #pragma unroll
            for (int u = 0; u < E / 8; ++u) {
                int q[8];
                #pragma unroll
                for (int k = 0; k < 8; ++k) q[k] = __float2int_rn(__fmul_rn(v[j][8 * u + k], r));
                uint2 bytes;
                uint4 f16;
                codes8(q, bytes, f16);
                if (a.Xq != nullptr) *reinterpret_cast<uint2*>(a.Xq + (size_t)row * K + lo + 8 * u) = bytes;
                if (a.Xe != nullptr) *reinterpret_cast<uint4*>(a.Xe + ((size_t)row * K + lo + 8 * u) * 2) = f16;
            }
            continue;
        }
        uint32_t packed[E / 8];
        #pragma unroll
        for (int u = 0; u < E / 8; ++u) {
            int q[8];
            #pragma unroll
            for (int k = 0; k < 8; ++k) q[k] = __float2int_rn(__fmul_rn(v[j][8 * u + k], r));
            packed[u] = pack8(q);
        }
        uint8_t* dst = a.Xq + (size_t)row * (K / 2) + lo / 2;
        if (a.Xq == nullptr) {
        } else if (E == 16) {
            *reinterpret_cast<uint2*>(dst) = make_uint2(packed[0], packed[1]);
        } else {
            #pragma unroll
            for (int u = 0; u < E / 32; ++u)
                reinterpret_cast<uint4*>(dst)[u] =
                    make_uint4(packed[4 * u], packed[4 * u + 1], packed[4 * u + 2], packed[4 * u + 3]);
        }
        if (a.Xe != nullptr) {   // E4M3 bytes of the same codes
            uint4* e4 = reinterpret_cast<uint4*>(a.Xe + (size_t)row * K + lo);
            #pragma unroll
            for (int u = 0; u < E / 16; ++u) {
                uint32_t o[4];
                int4x8_to_e4m3x8(packed[2 * u], o[0], o[1]);
                int4x8_to_e4m3x8(packed[2 * u + 1], o[2], o[3]);
                e4[u] = make_uint4(o[0], o[1], o[2], o[3]);
            }
        }
    }
}

template <typename T> struct To;
template <> struct To<__half> { static __device__ __forceinline__ float f(__half h) { return __half2float(h); } };
template <> struct To<__nv_bfloat16> { static __device__ __forceinline__ float f(__nv_bfloat16 h) { return __bfloat162float(h); } };
template <> struct To<float> { static __device__ __forceinline__ float f(float h) { return h; } };

// ---------------------------------------------------------------------------
// Rows with Hadamard blocks of 1024 elements or more (hb >= 1024, K a
// multiple of 1024, K <= 4096 NR), or of at most 512 (1024 <= K <= 4096,
// K % 512 == 0, a last chunk of 512 allowed): one CTA of four warps per
// row, in rounds of 4096 elements (four 1024-element chunks, chunk j of a
// round in warp j).
// A warp reads its chunk of x and of the smoothing vector with coalesced
// 16-byte loads (lane l at 16 l + 512 q) and passes each through its
// shared slice to take it back in layout A (18 KB of shared memory per CTA,
// so registers, not shared memory, bound the CTAs per SM).
//
//   layout A  lane l holds elements 32 l .. 32 l + 31 of its warp's chunk:
//             stages h = 1 .. 16 are between registers;
//   layout B  lane l holds elements l + 32 i (i = 0 .. 31) of the chunk,
//             after a transpose through the chunk's shared slice: stages
//             h = 32 .. 512 are between registers;
//   layout C  after the round's four chunks are in shared memory, lane l of
//             warp w holds elements j 1024 + 256 w + 8 l .. + 7 of every
//             chunk j: stages h = 1024, 2048 are between registers, and the
//             eight consecutive codes per chunk pack into one 32-bit word.
// Butterflies on pairs of registers use the packed f32x2 add and subtract
// (each half rounds like the scalar operation). The shared slice of a chunk
// holds its 32 x 32 floats in rows of 36 (four floats of padding): row r
// starts 4 r banks further on, so the row-wise 16-byte accesses (layouts A
// and C, eight lanes per phase) and the column-wise 4-byte accesses (layout
// B) are all free of bank conflicts, and every address is a per-thread base
// plus a constant.
// ---------------------------------------------------------------------------
constexpr int SROW = 36;                                   // floats per row of a 32 x 32 slice
constexpr int SLICE = 32 * SROW;                           // floats per slice
__device__ __forceinline__ int pad(int row, int col) {     // float index in a padded slice
    return row * SROW + col;
}

// Two butterflies (a0, b0) and (a1, b1) with one packed add and one packed
// subtract: a' = a + b, b' = a - b.
__device__ __forceinline__ void butterfly2(float& a0, float& a1, float& b0, float& b1) {
    asm("{\n\t.reg .b64 A, B, S, D;\n\t"
        "mov.b64 A, {%0, %1};\n\t"
        "mov.b64 B, {%2, %3};\n\t"
        "add.rn.f32x2 S, A, B;\n\t"
        "sub.rn.f32x2 D, A, B;\n\t"
        "mov.b64 {%0, %1}, S;\n\t"
        "mov.b64 {%2, %3}, D;\n\t}"
        : "+f"(a0), "+f"(a1), "+f"(b0), "+f"(b1));
}

// In-register stages of a 32-value array for register distances
// s = s_lo .. s_end / 2 (s = 1 scalar, s >= 2 on packed pairs).
__device__ __forceinline__ void reg_stages32(float (&v)[32], int s_lo, int s_end) {
    if (s_lo <= 1 && 1 < s_end) {
        #pragma unroll
        for (int i = 0; i < 32; i += 2) butterfly(v[i], v[i + 1]);
    }
    #pragma unroll
    for (int s = 2; s < 32; s <<= 1) {
        if (s >= s_lo && s < s_end) {
            #pragma unroll
            for (int i = 0; i < 32; i += 2)
                if ((i & s) == 0) butterfly2(v[i], v[i + 1], v[i + s], v[i + s + 1]);
        }
    }
}

// Codes of two values: q = rne(fl(v * r)). The product is a scalar
// round-to-nearest multiply (never contracted: a fused multiply-add would
// round the exact product and break ties differently). Adding M = 1.5 * 2^23
// then rounds it to an integer in one step (floats in [2^23, 2^24) are the
// integers, ties to even), fl(t - M) is that integer as a float (+0 for
// zero), and the low mantissa bits of t are the integer itself.
__device__ __forceinline__ void quant_pair(float v0, float v1, float r, float& q0, float& q1, int& i0, int& i1) {
    const float p0 = __fmul_rn(v0, r), p1 = __fmul_rn(v1, r);
    asm("{\n\t.reg .b64 V, M, T;\n\t"
        "mov.b64 V, {%4, %5};\n\t"
        "mov.b64 M, {%6, %6};\n\t"
        "add.rn.f32x2 T, V, M;\n\t"
        "sub.rn.f32x2 V, T, M;\n\t"
        "mov.b64 {%0, %1}, V;\n\t"
        "mov.b64 {%2, %3}, T;\n\t}"
        : "=f"(q0), "=f"(q1), "=r"(i0), "=r"(i1) : "f"(p0), "f"(p1), "f"(12582912.0f));
    i0 -= 0x4B400000;
    i1 -= 0x4B400000;
}

// Eight codes (ints) -> packed nibbles, code k in bits 4k .. 4k + 3.
__device__ __forceinline__ uint32_t pack_nibbles8(const int* qi) {
    uint32_t w = 0;
    #pragma unroll
    for (int k = 6; k >= 0; k -= 2)      // d = c << 8 | sat4(a) << 4 | sat4(b)
        asm("cvt.pack.sat.s4.s32.b32 %0, %1, %2, %0;" : "+r"(w) : "r"(qi[k + 1]), "r"(qi[k]));
    return w;
}
// Eight codes (floats) -> their eight E4M3 bytes (byte k = code k).
__device__ __forceinline__ uint2 e4m3_bytes8(const float* qf) {
    uint16_t h[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k)          // upper byte from the first operand
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(h[k]) : "f"(qf[2 * k + 1]), "f"(qf[2 * k]));
    return make_uint2((uint32_t)h[0] | ((uint32_t)h[1] << 16), (uint32_t)h[2] | ((uint32_t)h[3] << 16));
}

__device__ __forceinline__ float ld_shared_cluster_f32(uint32_t cluster_addr) {
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(cluster_addr) : "memory");
    return v;
}

// ASYM: the asymmetric mode (a compile-time copy, so that the symmetric
// kernel carries none of its reductions). CL > 1 (with NR = 1): a cluster
// of CL CTAs per row, CTA r taking the row's features 4096 r .. 4096 r +
// 4095; the CTAs exchange their maxima through distributed shared memory,
// so no thread holds more than one 4096-feature slice.
// G2: rows a0.L .. a0.L + b.L - 1 of the grid quantise problem b (the same
// K, hb, input type and code width; its own X, mask, transform and outputs):
// two quantisations in one launch.
template <int NR, typename Tin, bool ASYM, int CL = 1, bool G2 = false>
__global__ void __launch_bounds__(128, NR == 1 ? 7 : 1)
sgat_quant_rows_kernel(QuantArgs a0, QuantArgs b) {
    static_assert(CL == 1 || NR == 1, "one slice per CTA of a cluster");
    static_assert(!G2 || CL == 1, "grouped launches run one CTA per row");
    const bool p1 = G2 && (int)blockIdx.x >= a0.L;
    const QuantArgs& a = p1 ? b : a0;
    __shared__ __align__(16) float buf[4 * SLICE];
    __shared__ float red[8];              // [0, 4) amax or X_max, [4, 8) -X_min (asym)
    __shared__ float cl_red[2];           // this CTA's maximum (and -minimum) for its cluster
    // launched with programmatic serialisation: the rows of a problem whose
    // caller vouches that the preceding launch neither writes its inputs
    // nor touches its outputs start without waiting for that launch
    if (!a.independent) grid_dependency_wait();
    grid_launch_dependents();
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int rank = CL > 1 ? (int)cluster_ctarank() : 0;
    const int row = CL > 1 ? (int)blockIdx.x / CL : (int)blockIdx.x - (p1 ? a0.L : 0);
    const int K = a.K;
    const bool masked = a.mask != nullptr && a.mask[row] != 0;
    const float* sm = masked ? a.a_m : a.a_u;
    const int own_lo = masked ? a.d_sh : a.d_sh + a.d_m;
    const int own_hi = masked ? a.d_sh + a.d_m : K;
    const Tin* X = static_cast<const Tin*>(a.X) + (size_t)row * K;
    float* slice = buf + warp * SLICE;

    float v[NR][32];                      // layout C: v[R][8 j + k]
    float amax = 0.f, nmin = 0.f;         // asym: X_max and -X_min
    #pragma unroll
    for (int R = 0; R < NR; ++R) {
        const int base = (rank + R) * 4096;
        const int nch = min(4, (K - base + 1023) >> 10); // chunks in this round (>= 1)
        float u[32];
        if (warp < nch) {
            // coalesced loads (lane l: 16 bytes at 16 l + 512 q); x and then
            // the smoothing vector pass through the warp's slice and come
            // back in layout A
            const int c0 = base + warp * 1024;                   // first element of the chunk
            // a last chunk of 512 (hb <= 512 only): the upper half is zeros,
            // its own Hadamard blocks, never stored
            const bool half = K - c0 < 1024;
            float4 sr[8];
            if (sizeof(Tin) == 2) {
                uint4 xr[4];
                #pragma unroll
                for (int q = 0; q < 4; ++q)
                    xr[q] = (!half || q < 2) ? __ldg(reinterpret_cast<const uint4*>(X + c0) + lane + 32 * q)
                                             : make_uint4(0u, 0u, 0u, 0u);
                // 16-bit staging: 32 rows of 64 bytes, 16-byte group g of row R at g ^ ((R >> 1) & 3)
                uint8_t* st8 = reinterpret_cast<uint8_t*>(slice);
                #pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int R = (lane >> 2) + 8 * q, g = lane & 3;
                    *reinterpret_cast<uint4*>(st8 + R * 64 + 16 * (g ^ ((R >> 1) & 3))) = xr[q];
                }
                if (sm != nullptr) {
                    #pragma unroll
                    for (int q = 0; q < 8; ++q)
                        sr[q] = (!half || q < 4) ? __ldg(reinterpret_cast<const float4*>(sm + c0) + lane + 32 * q)
                                                 : make_float4(0.f, 0.f, 0.f, 0.f);
                }
                __syncwarp();
                #pragma unroll
                for (int g = 0; g < 4; ++g) {
                    const uint4 w = *reinterpret_cast<const uint4*>(st8 + lane * 64 + 16 * (g ^ ((lane >> 1) & 3)));
                    const Tin* h = reinterpret_cast<const Tin*>(&w);
                    #pragma unroll
                    for (int k = 0; k < 8; ++k) u[8 * g + k] = To<Tin>::f(h[k]);
                }
            } else {
                float4 xr[8];
                #pragma unroll
                for (int q = 0; q < 8; ++q)
                    xr[q] = (!half || q < 4) ? __ldg(reinterpret_cast<const float4*>(X + c0) + lane + 32 * q)
                                             : make_float4(0.f, 0.f, 0.f, 0.f);
                #pragma unroll
                for (int q = 0; q < 8; ++q)
                    *reinterpret_cast<float4*>(slice + pad((lane >> 3) + 4 * q, 4 * (lane & 7))) = xr[q];
                if (sm != nullptr) {
                    #pragma unroll
                    for (int q = 0; q < 8; ++q)
                        sr[q] = (!half || q < 4) ? __ldg(reinterpret_cast<const float4*>(sm + c0) + lane + 32 * q)
                                                 : make_float4(0.f, 0.f, 0.f, 0.f);
                }
                __syncwarp();
                #pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float4 w = *reinterpret_cast<const float4*>(slice + pad(lane, 4 * q));
                    u[4 * q] = w.x; u[4 * q + 1] = w.y; u[4 * q + 2] = w.z; u[4 * q + 3] = w.w;
                }
            }
            if (sm != nullptr) {
                __syncwarp();                                    // x has left the slice
                #pragma unroll
                for (int q = 0; q < 8; ++q)
                    *reinterpret_cast<float4*>(slice + pad((lane >> 3) + 4 * q, 4 * (lane & 7))) = sr[q];
                __syncwarp();
                #pragma unroll
                for (int q = 0; q < 8; ++q) {
                    const float4 w = *reinterpret_cast<const float4*>(slice + pad(lane, 4 * q));
                    u[4 * q] = __fmul_rn(u[4 * q], w.x);
                    u[4 * q + 1] = __fmul_rn(u[4 * q + 1], w.y);
                    u[4 * q + 2] = __fmul_rn(u[4 * q + 2], w.z);
                    u[4 * q + 3] = __fmul_rn(u[4 * q + 3], w.w);
                }
            }
            __syncwarp();
            reg_stages32(u, 1, a.hb < 32 ? a.hb : 32);          // h = 1 .. min(hb, 32) / 2
            #pragma unroll
            for (int q = 0; q < 8; ++q)                          // layout A -> slice
                *reinterpret_cast<float4*>(slice + pad(lane, 4 * q)) =
                    make_float4(u[4 * q], u[4 * q + 1], u[4 * q + 2], u[4 * q + 3]);
            __syncwarp();
            #pragma unroll
            for (int i = 0; i < 32; ++i) u[i] = slice[pad(i, lane)];   // layout B
            reg_stages32(u, 1, a.hb / 32);                       // h = 32 .. min(hb, 1024) / 2
            #pragma unroll
            for (int i = 0; i < 32; ++i) slice[pad(i, lane)] = u[i];
        }
        __syncthreads();
        #pragma unroll
        for (int j = 0; j < 4; ++j) {                            // layout C
            if (j < nch) {
                const int r = warp * 8 + (lane >> 2), c = (lane & 3) * 8;
                const float4 p0 = *reinterpret_cast<const float4*>(buf + j * SLICE + pad(r, c));
                const float4 p1 = *reinterpret_cast<const float4*>(buf + j * SLICE + pad(r, c + 4));
                v[R][8 * j] = p0.x; v[R][8 * j + 1] = p0.y; v[R][8 * j + 2] = p0.z; v[R][8 * j + 3] = p0.w;
                v[R][8 * j + 4] = p1.x; v[R][8 * j + 5] = p1.y; v[R][8 * j + 6] = p1.z; v[R][8 * j + 7] = p1.w;
            } else {
                #pragma unroll
                for (int k = 0; k < 8; ++k) v[R][8 * j + k] = 0.f;
            }
        }
        if (NR > 1) __syncthreads();                             // the next round reuses buf
        if (a.hb > 1024) {                                       // h = 1024: chunks j, j ^ 1
            #pragma unroll
            for (int k = 0; k < 8; k += 2) {
                butterfly2(v[R][k], v[R][k + 1], v[R][8 + k], v[R][9 + k]);
                butterfly2(v[R][16 + k], v[R][17 + k], v[R][24 + k], v[R][25 + k]);
            }
        }
        if (a.hb > 2048) {                                       // h = 2048: chunks j, j ^ 2
            #pragma unroll
            for (int k = 0; k < 8; k += 2) {
                butterfly2(v[R][k], v[R][k + 1], v[R][16 + k], v[R][17 + k]);
                butterfly2(v[R][8 + k], v[R][9 + k], v[R][24 + k], v[R][25 + k]);
            }
        }
        #pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e0 = base + j * 1024 + warp * 256 + 8 * lane;    // first element of the group
            if (j >= nch || e0 >= K) continue;
            const bool all_keep = (e0 + 8 <= a.d_sh) || (e0 >= own_lo && e0 + 8 <= own_hi);
            if (!all_keep) {
                #pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const int e = e0 + k;
                    if (!(e < a.d_sh || (e >= own_lo && e < own_hi))) v[R][8 * j + k] = 0.f;
                }
            }
            if (a.post_scale != 1.f) {
                #pragma unroll
                for (int k = 0; k < 8; ++k) v[R][8 * j + k] = __fmul_rn(v[R][8 * j + k], a.post_scale);
            }
            if (ASYM) {
                #pragma unroll
                for (int k = 0; k < 8; ++k) {
                    amax = fmaxf(amax, v[R][8 * j + k]);
                    nmin = fmaxf(nmin, -v[R][8 * j + k]);
                }
            } else {
                #pragma unroll
                for (int k = 0; k < 8; ++k) amax = fmaxf(amax, fabsf(v[R][8 * j + k]));
            }
            if (a.v_dbg != nullptr) {
                float4* d4 = reinterpret_cast<float4*>(a.v_dbg + (size_t)row * K + e0);
                d4[0] = make_float4(v[R][8 * j], v[R][8 * j + 1], v[R][8 * j + 2], v[R][8 * j + 3]);
                d4[1] = make_float4(v[R][8 * j + 4], v[R][8 * j + 5], v[R][8 * j + 6], v[R][8 * j + 7]);
            }
        }
    }
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, m));
    if (ASYM) {
        #pragma unroll
        for (int m = 16; m > 0; m >>= 1) nmin = fmaxf(nmin, __shfl_xor_sync(0xffffffffu, nmin, m));
    }
    if (lane == 0) {
        red[warp] = amax;
        if (ASYM) red[4 + warp] = nmin;
    }
    __syncthreads();
    amax = fmaxf(fmaxf(red[0], red[1]), fmaxf(red[2], red[3]));
    if (ASYM) nmin = fmaxf(fmaxf(red[4], red[5]), fmaxf(red[6], red[7]));
    if (CL > 1) {                      // the row's maximum over the cluster's slices
        if (threadIdx.x == 0) {
            cl_red[0] = amax;
            cl_red[1] = nmin;
        }
        cluster_sync();
        #pragma unroll
        for (int c = 0; c < CL; ++c) {
            amax = fmaxf(amax, ld_shared_cluster_f32(mapa_shared(smem_addr(&cl_red[0]), (uint32_t)c)));
            if (ASYM) nmin = fmaxf(nmin, ld_shared_cluster_f32(mapa_shared(smem_addr(&cl_red[1]), (uint32_t)c)));
        }
    }

    const float qmax = (float)a.qmax;
    const float range = ASYM ? __fadd_rn(amax, nmin) : amax;     // X_max - X_min, or amax
    const bool nz = range > 0.f;
    const float s = nz ? __fdiv_rn(range, qmax) : 0.f;
    const float r = nz ? __fdiv_rn(qmax, range) : 0.f;
    const int zp = ASYM ? min(max(__float2int_rn(__fmul_rn(nmin, r)), 0), a.qmax) : 0;
    if (threadIdx.x == 0 && rank == 0) {
        a.s[row] = s;
        if (ASYM) a.z[row] = zp;
    }
    if (ASYM && a.Xe != nullptr && threadIdx.x < 8 && rank == 0)
        store_zero_point_columns(a.Xe + (size_t)row * (K + 128) + K, zp, threadIdx.x);
    #pragma unroll
    for (int R = 0; R < NR; ++R) {
        const int base = (rank + R) * 4096;
        const int nch = min(4, (K - base + 1023) >> 10);
        #pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e0 = base + j * 1024 + warp * 256 + 8 * lane;
            if (j >= nch || e0 >= K) continue;
            float qf[8];
            int qi[8];
            #pragma unroll
            for (int k = 0; k < 8; k += 2)
                quant_pair(v[R][8 * j + k], v[R][8 * j + k + 1], r, qf[k], qf[k + 1], qi[k], qi[k + 1]);
            if (ASYM) {                  // codes in [0, qmax]: unsigned nibbles and E4M3 bytes
                int q[8];
                #pragma unroll
                for (int k = 0; k < 8; ++k) q[k] = min(max(qi[k] + zp, 0), a.qmax);
                if (a.Xq != nullptr) *reinterpret_cast<uint32_t*>(a.Xq + (size_t)row * (K / 2) + e0 / 2) = pack8(q);
                if (a.Xe != nullptr) *reinterpret_cast<uint2*>(a.Xe + (size_t)row * (K + 128) + e0) = e4m3_of8(q);
                continue;
            }
            if (a.qmax > 15) {           // 8-bit codes: bytes and fp16
                uint2 bytes;
                uint4 f16;
                codes8(qi, bytes, f16);
                if (a.Xq != nullptr) *reinterpret_cast<uint2*>(a.Xq + (size_t)row * K + e0) = bytes;
                if (a.Xe != nullptr) *reinterpret_cast<uint4*>(a.Xe + ((size_t)row * K + e0) * 2) = f16;
                continue;
            }
            if (a.Xq != nullptr)
                *reinterpret_cast<uint32_t*>(a.Xq + (size_t)row * (K / 2) + e0 / 2) = pack_nibbles8(qi);
            if (a.Xe != nullptr) *reinterpret_cast<uint2*>(a.Xe + (size_t)row * K + e0) = e4m3_bytes8(qf);
        }
    }
    if (CL > 1) cluster_sync();        // no CTA leaves while its maximum may still be read
}

template <int NR, typename Tin>
cudaError_t launch_rows_nr(const QuantArgs& a, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1] = {pdl_attribute()};
    cfg.gridDim = dim3(a.L);
    cfg.blockDim = dim3(128);
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return a.asym ? cudaLaunchKernelEx(&cfg, sgat_quant_rows_kernel<NR, Tin, true>, a, a)
                  : cudaLaunchKernelEx(&cfg, sgat_quant_rows_kernel<NR, Tin, false>, a, a);
}

// Rows longer than 4096: a cluster of CL CTAs per row, one 4096-feature
// slice each.
template <int CL, typename Tin>
cudaError_t launch_rows_cl(const QuantArgs& a, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[2];
    at[0] = pdl_attribute();
    at[1].id = cudaLaunchAttributeClusterDimension;
    at[1].val.clusterDim.x = CL;
    at[1].val.clusterDim.y = 1;
    at[1].val.clusterDim.z = 1;
    cfg.gridDim = dim3((unsigned)a.L * CL);
    cfg.blockDim = dim3(128);
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return a.asym ? cudaLaunchKernelEx(&cfg, sgat_quant_rows_kernel<1, Tin, true, CL>, a, a)
                  : cudaLaunchKernelEx(&cfg, sgat_quant_rows_kernel<1, Tin, false, CL>, a, a);
}

// Two symmetric quantisations of rows up to 4096 features in one launch
// (one CTA per row of either problem).
template <typename Tin>
cudaError_t launch_rows_grouped(const QuantArgs& a, const QuantArgs& b, cudaStream_t stream) {
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1] = {pdl_attribute()};
    cfg.gridDim = dim3((unsigned)(a.L + b.L));
    cfg.blockDim = dim3(128);
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, sgat_quant_rows_kernel<1, Tin, false, 1, true>, a, b);
}

template <typename Tin>
cudaError_t launch_rows(const QuantArgs& a, cudaStream_t stream) {
    switch ((a.K + 4095) / 4096) {
        case 1: return launch_rows_nr<1, Tin>(a, stream);
        case 2: return launch_rows_cl<2, Tin>(a, stream);
        case 3: return launch_rows_cl<3, Tin>(a, stream);
        case 4: return launch_rows_cl<4, Tin>(a, stream);
        case 5: return launch_rows_cl<5, Tin>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <int E, typename Tin>
cudaError_t launch_e(const QuantArgs& a, cudaStream_t stream) {
    constexpr int C = 32 * E;
    const int n = (a.K + C - 1) / C;                 // chunks per row
    int wpr, nc;                                     // warps per row, rounds
    if (E == 16 && a.hb <= C && n > 8) {             // no stage crosses warps: up to 20 warps, 2 rounds
        nc = (n + 19) / 20;
        wpr = (n + nc - 1) / nc;
    } else {
        wpr = n < 8 ? n : 8;                         // a multiple of hb / C
        nc = (n + wpr - 1) / wpr;
    }
    const int rpc = wpr <= 4 ? 8 / wpr : 1;          // rows per CTA
    const int warps = wpr * rpc;
    const size_t smem = (size_t)warps * (C + 32) * 4 + 64 * 4;
    dim3 grid((a.L + rpc - 1) / rpc), block(32 * warps);
    #define STARQ_QUANT_LAUNCH(NCV)                                                            \
        {                                                                                      \
            static DeviceCache<int> attr;                                                      \
            int done = 0;                                                                      \
            const cudaError_t e = attr.get(&done, [](int, int* v) {                            \
                *v = 1;                                                                        \
                return cudaFuncSetAttribute(sgat_quant_kernel<E, NCV, Tin>,                    \
                        cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);              \
            });                                                                                \
            if (e != cudaSuccess) return e;                                                    \
            sgat_quant_kernel<E, NCV, Tin><<<grid, block, smem, stream>>>(a, wpr, rpc);        \
        }
    switch (nc) {
        case 1: STARQ_QUANT_LAUNCH(1); break;
        case 2: STARQ_QUANT_LAUNCH(2); break;
        case 3: STARQ_QUANT_LAUNCH(3); break;
        case 4: STARQ_QUANT_LAUNCH(4); break;
        case 5: if constexpr (E <= 16) STARQ_QUANT_LAUNCH(5); break;
        default: return cudaErrorInvalidValue;
    }
    #undef STARQ_QUANT_LAUNCH
    return cudaGetLastError();
}

template <typename Tin>
cudaError_t launch_typed(const QuantArgs& a, cudaStream_t stream) {
    // otherwise a warp's chunk is 1024 elements (hb >= 1024, blocks finish
    // across warps) or 512 elements holding 512 / hb blocks
    // up to 20480 features in 4096-feature slices (a cluster of CTAs per row
    // beyond 4096): blocks of 1024 or more with K % 1024 == 0, or of up to
    // 512 with K % 512 == 0 (a last chunk of 512 allowed)
    if (a.K <= 20480 && ((a.hb >= 1024 && a.K % 1024 == 0) || (a.hb <= 512 && a.K >= 1024 && a.K % 512 == 0)))
        return launch_rows<Tin>(a, stream);
    return a.hb >= 1024 ? launch_e<32, Tin>(a, stream) : launch_e<16, Tin>(a, stream);
}

}  // namespace

cudaError_t launch_sgat_quant(const QuantArgs& a, cudaStream_t stream) {
    if (a.L == 0) return cudaSuccess;
    switch (a.x_dtype) {
        case STARQ_F16: return launch_typed<__half>(a, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_typed<float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

// Whether the row kernel with one CTA per row takes this problem.
static bool rows_one_cta(const QuantArgs& a) {
    return !a.asym && a.K <= 4096 &&
           ((a.hb >= 1024 && a.K % 1024 == 0) || (a.hb <= 512 && a.K >= 1024 && a.K % 512 == 0));
}

cudaError_t launch_sgat_quant_grouped(const QuantArgs& a, const QuantArgs& b, cudaStream_t stream) {
    const bool same = a.x_dtype == b.x_dtype && a.K == b.K && a.hb == b.hb && a.qmax == b.qmax &&
                      a.post_scale == b.post_scale && rows_one_cta(a) && rows_one_cta(b);
    if (!same || a.L == 0 || b.L == 0) {             // two launches
        cudaError_t e = launch_sgat_quant(a, stream);
        return e != cudaSuccess ? e : launch_sgat_quant(b, stream);
    }
    switch (a.x_dtype) {
        case STARQ_F16: return launch_rows_grouped<__half>(a, b, stream);
        case STARQ_BF16: return launch_rows_grouped<__nv_bfloat16>(a, b, stream);
        case STARQ_F32: return launch_rows_grouped<float>(a, b, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
