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
// [rows][2K] holds the nibble split c = 16 h + l, l = ((c + 8) mod 16) - 8 in
// [-8, 7], h = (c - l) / 16 in [-8, 8]: E4M3 bytes of h in columns 0..K-1
// and of l in columns K..2K-1 (both exact in E4M3), the operands of the
// 8-bit GEMM.
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
// the E4M3 bytes of their split c = 16 h + l (see the file comment).
__device__ __forceinline__ void split_codes8(const int* q, uint2& bytes, uint2& eh, uint2& el) {
    uint32_t b0 = 0, b1 = 0;
    #pragma unroll
    for (int k = 0; k < 4; ++k) {
        b0 |= (uint32_t)(q[k] & 0xFF) << (8 * k);
        b1 |= (uint32_t)(q[k + 4] & 0xFF) << (8 * k);
    }
    bytes = make_uint2(b0, b1);
    uint16_t hh[4], ll[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k) {        // upper byte from the first operand
        const int l0 = ((q[2 * k] + 8) & 15) - 8, l1 = ((q[2 * k + 1] + 8) & 15) - 8;
        const int h0 = (q[2 * k] - l0) >> 4, h1 = (q[2 * k + 1] - l1) >> 4;
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(hh[k]) : "f"((float)h1), "f"((float)h0));
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(ll[k]) : "f"((float)l1), "f"((float)l0));
    }
    eh = make_uint2((uint32_t)hh[0] | ((uint32_t)hh[1] << 16), (uint32_t)hh[2] | ((uint32_t)hh[3] << 16));
    el = make_uint2((uint32_t)ll[0] | ((uint32_t)ll[1] << 16), (uint32_t)ll[2] | ((uint32_t)ll[3] << 16));
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

template <int E, int NC, typename Tin>
__global__ void __launch_bounds__(256)
sgat_quant_kernel(QuantArgs a, int warps_per_row, int rows_per_cta) {
    extern __shared__ float qsm[];
    constexpr int C = 32 * E;
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int wr = warp % warps_per_row;                 // warp index within its row
    const int row = blockIdx.x * rows_per_cta + warp / warps_per_row;
    float* buf = qsm + warp * (C + 32);
    float* red = qsm + (blockDim.x >> 5) * (C + 32);     // [warps] partial amax
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
            red[8 + warp] = nmin;
        }
        __syncthreads();
        amax = 0.f;
        nmin = 0.f;
        const int first = warp - wr;                     // first warp of this row
        for (int w = 0; w < warps_per_row; ++w) {
            amax = fmaxf(amax, red[first + w]);
            nmin = fmaxf(nmin, red[8 + first + w]);
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
                *reinterpret_cast<uint32_t*>(a.Xq + (size_t)row * (K / 2) + lo / 2 + 4 * u) = pack8(q);
                if (a.Xe != nullptr) *reinterpret_cast<uint2*>(a.Xe + (size_t)row * (K + 128) + lo + 8 * u) = e4m3_of8(q);
            }
            continue;
        }
        if (a.qmax > 15) {               // 8-bit codes: bytes and their E4M3 split
            #pragma unroll
            for (int u = 0; u < E / 8; ++u) {
                int q[8];
                #pragma unroll
                for (int k = 0; k < 8; ++k) q[k] = __float2int_rn(__fmul_rn(v[j][8 * u + k], r));
                uint2 bytes, eh, el;
                split_codes8(q, bytes, eh, el);
                *reinterpret_cast<uint2*>(a.Xq + (size_t)row * K + lo + 8 * u) = bytes;
                if (a.Xe != nullptr) {
                    *reinterpret_cast<uint2*>(a.Xe + (size_t)row * 2 * K + lo + 8 * u) = eh;
                    *reinterpret_cast<uint2*>(a.Xe + (size_t)row * 2 * K + K + lo + 8 * u) = el;
                }
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
        if (E == 16) {
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

__device__ __forceinline__ int swz(int row, int col) {      // float index in a 32 x 32 slice
    return row * 32 + ((((col >> 2) ^ (row & 7))) << 2) + (col & 3);
}

// Packed float32 pairs (sm_100 family): each half rounds like the scalar
// operation (PTX add / sub / mul with the explicit .rn rounding). A packed
// product that feeds a packed sum can still be fused by the compiler, so no
// f2mul result is ever added by f2add / f2sub (see quant2).
__device__ __forceinline__ float2 f2op_add(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 A, B, D;\n\tmov.b64 A, {%2, %3};\n\tmov.b64 B, {%4, %5};\n\t"
        "add.rn.f32x2 D, A, B;\n\tmov.b64 {%0, %1}, D;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 f2op_sub(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 A, B, D;\n\tmov.b64 A, {%2, %3};\n\tmov.b64 B, {%4, %5};\n\t"
        "sub.rn.f32x2 D, A, B;\n\tmov.b64 {%0, %1}, D;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 f2op_mul(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 A, B, D;\n\tmov.b64 A, {%2, %3};\n\tmov.b64 B, {%4, %5};\n\t"
        "mul.rn.f32x2 D, A, B;\n\tmov.b64 {%0, %1}, D;\n\t}"
        : "=f"(d.x), "=f"(d.y) : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 f2add(float2 a, float2 b) { return f2op_add(a, b); }
__device__ __forceinline__ float2 f2sub(float2 a, float2 b) { return f2op_sub(a, b); }
__device__ __forceinline__ float2 f2mul(float2 a, float2 b) { return f2op_mul(a, b); }
__device__ __forceinline__ void bfly2(float2& a, float2& b) {
    const float2 x = a, y = b;
    a = f2add(x, y);
    b = f2sub(x, y);
}

// In-register butterfly stages of 32 values held as 16 pairs (value e in
// u[e / 2], .x for even e): value distances s = s_lo .. s_end / 2; s = 1
// pairs the two halves of each float2 (scalar), s >= 2 pairs float2 i with
// i + s / 2 (packed).
__device__ __forceinline__ void reg_stages16(float2 (&u)[16], int s_lo, int s_end) {
    if (s_lo <= 1 && 1 < s_end) {
        #pragma unroll
        for (int i = 0; i < 16; ++i) {
            const float a = u[i].x, b = u[i].y;
            u[i] = make_float2(__fadd_rn(a, b), __fsub_rn(a, b));
        }
    }
    #pragma unroll
    for (int s = 2; s < 32; s <<= 1) {
        if (s >= s_lo && s < s_end) {
            #pragma unroll
            for (int i = 0; i < 16; ++i)
                if ((i & (s / 2)) == 0) bfly2(u[i], u[i + s / 2]);
        }
    }
}

// Codes of a pair: q = rne(fl(v * r)). The product rounds once (never a
// fused multiply-add, which would round the exact product and break ties
// differently); adding M = 1.5 * 2^23 then rounds it to an integer in one
// step (the floats of [2^23, 2^24) are the integers, ties to even). t holds
// M + q, whose low byte is q in two's complement; fl(t - M) is q as a float
// (+0 for zero).
// The product is two scalar round-to-nearest multiplies: a packed multiply
// followed by the packed add is fused into one packed FMA by the compiler
// even when both are written as .rn PTX, and an FMA rounds the exact product
// (a value whose product rounds onto a half-integer would then round the
// other way; on the LLaDA weights 6 of 50 M codes).
constexpr float ROUND_M = 12582912.0f;
__device__ __forceinline__ void quant2(float2 v, float2 rr, float2& q, float2& t) {
    const float2 p = make_float2(__fmul_rn(v.x, rr.x), __fmul_rn(v.y, rr.y));
    t = f2add(p, make_float2(ROUND_M, ROUND_M));
    q = f2add(t, make_float2(-ROUND_M, -ROUND_M));
}

// Eight codes in four pairs (q float values, t biased forms) -> packed
// nibbles (code k in bits 4k .. 4k + 3) and their eight E4M3 bytes. The
// nibbles come from the low bytes of the biased forms: the even codes' bytes
// and the odd codes' bytes are gathered by byte permutes, then the low
// nibbles of the even ones and the odd ones shifted up are merged.
__device__ __forceinline__ void pack_codes8(const float2 (&q)[4], const float2 (&t)[4], uint32_t& nib, uint2& e4) {
    const uint32_t ev = prmt(prmt(__float_as_uint(t[0].x), __float_as_uint(t[1].x), 0x40u),
                             prmt(__float_as_uint(t[2].x), __float_as_uint(t[3].x), 0x40u), 0x5410u);
    const uint32_t od = prmt(prmt(__float_as_uint(t[0].y), __float_as_uint(t[1].y), 0x40u),
                             prmt(__float_as_uint(t[2].y), __float_as_uint(t[3].y), 0x40u), 0x5410u);
    nib = (ev & 0x0F0F0F0Fu) | ((od << 4) & 0xF0F0F0F0u);
    uint16_t h[4];
    #pragma unroll
    for (int k = 0; k < 4; ++k)          // upper byte from the first operand
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(h[k]) : "f"(q[k].y), "f"(q[k].x));
    e4.x = (uint32_t)h[0] | ((uint32_t)h[1] << 16);
    e4.y = (uint32_t)h[2] | ((uint32_t)h[3] << 16);
}
__device__ __forceinline__ int code_of(float t) { return (int)(__float_as_uint(t) - 0x4B400000u); }

// Staging of one row's slice of 1024 elements for layout A. The row arrives
// by TMA in 128-byte lines with the 128-byte swizzle (16-byte unit u of line
// i at unit u ^ (i & 7)); lane l's 32 elements are 64 bytes (16-bit input,
// half of line l / 2) or 128 bytes (float, line l), and the swizzle spreads
// each quarter-warp's 16-byte reads over all banks.
template <typename Tin> struct Stage;
__device__ __forceinline__ float2 to_f2(__half2 h) { return __half22float2(h); }
__device__ __forceinline__ float2 to_f2(__nv_bfloat162 h) { return __bfloat1622float2(h); }
template <typename T2>
struct Stage16 {
    static __device__ __forceinline__ void load(uint32_t chunk, int lane, float2 (&u)[16]) {
        const uint32_t line = chunk + (uint32_t)(lane >> 1) * 128u;
        #pragma unroll
        for (int q = 0; q < 4; ++q) {
            const uint32_t unit = (uint32_t)(4 * (lane & 1) + q) ^ (uint32_t)((lane >> 1) & 7);
            const uint4 w = ld_shared_v4(line + (unit << 4));
            const T2* h = reinterpret_cast<const T2*>(&w);
            #pragma unroll
            for (int k = 0; k < 4; ++k) u[4 * q + k] = to_f2(h[k]);
        }
    }
};
template <> struct Stage<__half> : Stage16<__half2> {};
template <> struct Stage<__nv_bfloat16> : Stage16<__nv_bfloat162> {};
template <> struct Stage<float> {
    static __device__ __forceinline__ void load(uint32_t chunk, int lane, float2 (&u)[16]) {
        const uint32_t line = chunk + (uint32_t)lane * 128u;
        #pragma unroll
        for (int q = 0; q < 8; ++q) {
            const uint4 w = ld_shared_v4(line + ((uint32_t)(q ^ (lane & 7)) << 4));
            u[2 * q] = make_float2(__uint_as_float(w.x), __uint_as_float(w.y));
            u[2 * q + 1] = make_float2(__uint_as_float(w.z), __uint_as_float(w.w));
        }
    }
};

namespace rowsk {
constexpr int G = 2;                          // row groups (four warps each) per CTA
constexpr int THREADS = 128 * G;
constexpr int SLICES_BYTES = 4 * 1024 * 4;    // the four warps' transpose slices
constexpr int SMOOTH_RESIDENT_MAX_K = 8192;   // a_m and a_u stay in shared memory up to here
constexpr int LINES_PER_COPY = 16;            // 2 KB per TMA copy
constexpr unsigned STATUS_TIMEOUT_QUANT = 1u << 5;

// Dynamic shared memory: [a_m | a_u, K floats each, swizzled like float
// staging, when resident][per group: two row buffers of K * esize bytes,
// then the slices][barriers and reductions]; every region 1024-aligned.
struct Layout {
    int smooth_bytes, stage_bytes, group_bytes, total;
    __host__ __device__ Layout(int K, int esize, bool resident) {
        smooth_bytes = resident ? 2 * K * 4 : 0;
        stage_bytes = K * esize;
        group_bytes = 2 * stage_bytes + SLICES_BYTES;
        total = 1024 + smooth_bytes + G * group_bytes + 256;
    }
};
struct Ctl {
    uint64_t full[G][2];
    float red[G][8];
    int abort[G];
};
}  // namespace rowsk

// ---------------------------------------------------------------------------
// Rows with Hadamard blocks of 1024 elements or more (hb >= 1024, K a
// multiple of 1024, K <= 4096 NR). Persistent CTAs of G row groups; a group
// of four warps transforms and quantises one row at a time, in rounds of
// 4096 elements (four 1024-element chunks, chunk j of a round in warp j),
// while the next two rows arrive by TMA into the group's two row buffers.
// The smoothing vectors are copied into shared memory once per CTA (K <=
// 8192; larger rows read them from global memory, where they stay cached).
//
//   layout A  lane l holds elements 32 l .. 32 l + 31 of its warp's chunk:
//             stages h = 1 .. 16 are between registers;
//   layout B  lane l holds elements l + 32 i (i = 0 .. 31) of the chunk,
//             after a transpose through the warp's shared slice: stages
//             h = 32 .. 512 are between registers;
//   layout C  after the round's four chunks are in shared memory, lane l of
//             warp w holds elements j 1024 + 256 w + 8 l .. + 7 of every
//             chunk j: stages h = 1024, 2048 are between registers, and the
//             eight consecutive codes per chunk pack into one 32-bit word.
// Butterflies, the smoothing multiply and the quantiser's multiply work on
// register pairs with the packed f32x2 instructions (each half rounds like
// the scalar operation). A slice holds its 32 x 32 floats with 16-byte
// column groups XOR-swizzled by the row (row & 7), so the row-wise 16-byte
// accesses (layouts A and C) and the column-wise 4-byte accesses (layout B)
// are free of bank conflicts. Every wait is bounded.
// ---------------------------------------------------------------------------
template <int NR, typename Tin, bool ASYM, bool RESIDENT>
__global__ void __launch_bounds__(rowsk::THREADS, NR == 1 ? 2 : 1)
sgat_quant_rows_kernel(QuantArgs a, const __grid_constant__ CUtensorMap tmx) {
    using namespace rowsk;
    extern __shared__ uint8_t qrow_smem[];
    const int K = a.K;
    const Layout lay(K, (int)sizeof(Tin), RESIDENT);
    const uint32_t raw = smem_addr(qrow_smem);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t* const gbase = qrow_smem + (base - raw);
    const int lane = threadIdx.x & 31;
    const int g = threadIdx.x >> 7;                    // row group
    const int warp = (threadIdx.x >> 5) & 3;           // warp within the group
    const int gtid = threadIdx.x & 127;
    const uint32_t smooth = base;
    const uint32_t gstage = base + lay.smooth_bytes + g * lay.group_bytes;
    float* const slices = reinterpret_cast<float*>(gbase + lay.smooth_bytes + g * lay.group_bytes +
                                                   2 * lay.stage_bytes);
    float* const slice = slices + warp * 1024;
    Ctl* const ctl = reinterpret_cast<Ctl*>(gbase + lay.smooth_bytes + G * lay.group_bytes);
    volatile int* abort = &ctl->abort[g];
    const int copies = lay.stage_bytes / (LINES_PER_COPY * 128);
    const long long lines_per_row = (long long)lay.stage_bytes / 128;
    // rows of group g: first = blockIdx.x * G + g, then + gridDim.x * G
    const int stride = gridDim.x * G;
    const int first = blockIdx.x * G + g;

    if (threadIdx.x == 0) {
        for (int i = 0; i < G; ++i) {
            mbar_init(smem_addr(&ctl->full[i][0]), 1);
            mbar_init(smem_addr(&ctl->full[i][1]), 1);
            ctl->abort[i] = 0;
        }
        mbar_fence_init();
    }
    __syncthreads();
    grid_dependency_wait();            // launched with programmatic serialisation
    grid_launch_dependents();
    auto issue = [&](int row, int buf) {             // one thread of the group
        const uint32_t bar = smem_addr(&ctl->full[g][buf]);
        mbar_arrive_expect_tx(bar, (uint32_t)lay.stage_bytes);
        const uint32_t dst = gstage + (uint32_t)(buf * lay.stage_bytes);
        for (int c = 0; c < copies; ++c)
            tma_load_2d(dst + c * LINES_PER_COPY * 128, &tmx, 0,
                        (int)(row * lines_per_row + c * LINES_PER_COPY), bar);
    };
    if (gtid == 0) {
        if (first < a.L) issue(first, 0);
        if (first + stride < a.L) issue(first + stride, 1);
    }
    if (RESIDENT) {
        // a_m then a_u (NULL: ones), 4 floats per thread and step, stored in
        // the swizzled float staging layout of their lines
        const int n4 = K / 4;
        for (int f = threadIdx.x; f < 2 * n4; f += THREADS) {
            const int s = f >= n4, i = f - s * n4;
            const float* src = s ? a.a_u : a.a_m;
            const float4 v = src != nullptr ? __ldg(reinterpret_cast<const float4*>(src) + i)
                                            : make_float4(1.f, 1.f, 1.f, 1.f);
            const int line = s * (K / 32) + i / 8, unit = (i & 7) ^ (line & 7);
            st_shared_v4(smooth + line * 128 + unit * 16, __float_as_uint(v.x), __float_as_uint(v.y),
                         __float_as_uint(v.z), __float_as_uint(v.w));
        }
        __syncthreads();
    }
    auto group_sync = [&]() { asm volatile("bar.sync %0, 128;" :: "r"(1 + g) : "memory"); };

    const float qmax = (float)a.qmax;
    int it = 0;
    bool ok = true;
    for (int row = first; row < a.L; row += stride, ++it) {
        const int buf = it & 1;
        const uint32_t stage = gstage + (uint32_t)(buf * lay.stage_bytes);
        // a wait that runs out marks the group; every thread of the group
        // sees the mark after the round's first group barrier and leaves
        if (!mbar_wait_bounded(smem_addr(&ctl->full[g][buf]), (uint32_t)((it >> 1) & 1), abort)) *abort = 1;
        const bool masked = a.mask != nullptr && a.mask[row] != 0;
        const float* gsm = masked ? a.a_m : a.a_u;             // global copy (RESIDENT = false)
        const bool smooth_on = RESIDENT ? (masked ? a.a_m : a.a_u) != nullptr : gsm != nullptr;
        const int own_lo = masked ? a.d_sh : a.d_sh + a.d_m;
        const int own_hi = masked ? a.d_sh + a.d_m : K;

        float2 v[NR][16];                 // layout C: v[R][4 j + k] = elements e0 + 2k, e0 + 2k + 1 of chunk j
        float amax = 0.f, nmin = 0.f;     // asym: X_max and -X_min
        #pragma unroll
        for (int R = 0; R < NR; ++R) {
            const int rbase = R * 4096;
            const int nch = min(4, (K - rbase) >> 10);        // chunks in this round (>= 1)
            if (warp < nch) {
                const int c0 = rbase + warp * 1024;             // first element of the chunk
                float2 u[16];
                Stage<Tin>::load(stage + (uint32_t)(c0 * (int)sizeof(Tin)), lane, u);
                if (smooth_on) {
                    if (RESIDENT) {
                        const uint32_t sl = smooth + (uint32_t)(((masked ? 0 : K) + c0) * 4 + lane * 128);
                        #pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            const uint4 w = ld_shared_v4(sl + ((uint32_t)(q ^ (lane & 7)) << 4));
                            u[2 * q] = f2mul(u[2 * q], make_float2(__uint_as_float(w.x), __uint_as_float(w.y)));
                            u[2 * q + 1] = f2mul(u[2 * q + 1], make_float2(__uint_as_float(w.z), __uint_as_float(w.w)));
                        }
                    } else {
                        const float4* s4 = reinterpret_cast<const float4*>(gsm + c0 + 32 * lane);
                        #pragma unroll
                        for (int q = 0; q < 8; ++q) {
                            const float4 w = __ldg(s4 + q);
                            u[2 * q] = f2mul(u[2 * q], make_float2(w.x, w.y));
                            u[2 * q + 1] = f2mul(u[2 * q + 1], make_float2(w.z, w.w));
                        }
                    }
                }
                reg_stages16(u, 1, 32);                          // h = 1 .. 16
                #pragma unroll
                for (int q = 0; q < 8; ++q)                      // layout A -> slice
                    *reinterpret_cast<float4*>(slice + swz(lane, 4 * q)) =
                        make_float4(u[2 * q].x, u[2 * q].y, u[2 * q + 1].x, u[2 * q + 1].y);
                __syncwarp();
                #pragma unroll
                for (int i = 0; i < 16; ++i)                     // layout B: u[i] = rows 2i, 2i + 1
                    u[i] = make_float2(slice[swz(2 * i, lane)], slice[swz(2 * i + 1, lane)]);
                reg_stages16(u, 1, a.hb / 32);                   // h = 32 .. min(hb, 1024) / 2
                #pragma unroll
                for (int i = 0; i < 16; ++i) {
                    slice[swz(2 * i, lane)] = u[i].x;
                    slice[swz(2 * i + 1, lane)] = u[i].y;
                }
            }
            group_sync();
            if (*abort) { ok = false; break; }
            // the row buffer has been read in full: it takes the row after next
            if (R == NR - 1 && gtid == 0 && row + 2 * stride < a.L) {
                fence_proxy_async_smem();
                issue(row + 2 * stride, buf);
            }
            #pragma unroll
            for (int j = 0; j < 4; ++j) {                        // layout C
                if (j < nch) {
                    const int r = warp * 8 + (lane >> 2), c = (lane & 3) * 8;
                    const float4 p0 = *reinterpret_cast<const float4*>(slices + j * 1024 + swz(r, c));
                    const float4 p1 = *reinterpret_cast<const float4*>(slices + j * 1024 + swz(r, c + 4));
                    v[R][4 * j] = make_float2(p0.x, p0.y);
                    v[R][4 * j + 1] = make_float2(p0.z, p0.w);
                    v[R][4 * j + 2] = make_float2(p1.x, p1.y);
                    v[R][4 * j + 3] = make_float2(p1.z, p1.w);
                } else {
                    #pragma unroll
                    for (int k = 0; k < 4; ++k) v[R][4 * j + k] = make_float2(0.f, 0.f);
                }
            }
            if (NR > 1) group_sync();                            // the next round reuses the slices
            if (a.hb > 1024) {                                   // h = 1024: chunks j, j ^ 1
                #pragma unroll
                for (int k = 0; k < 4; ++k) {
                    bfly2(v[R][k], v[R][4 + k]);
                    bfly2(v[R][8 + k], v[R][12 + k]);
                }
            }
            if (a.hb > 2048) {                                   // h = 2048: chunks j, j ^ 2
                #pragma unroll
                for (int k = 0; k < 4; ++k) {
                    bfly2(v[R][k], v[R][8 + k]);
                    bfly2(v[R][4 + k], v[R][12 + k]);
                }
            }
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int e0 = rbase + j * 1024 + warp * 256 + 8 * lane;    // first element of the group
                if (j >= nch) continue;
                const bool all_keep = (e0 + 8 <= a.d_sh) || (e0 >= own_lo && e0 + 8 <= own_hi);
                if (!all_keep) {
                    #pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        const int e = e0 + k;
                        if (!(e < a.d_sh || (e >= own_lo && e < own_hi))) {
                            if (k & 1) v[R][4 * j + k / 2].y = 0.f;
                            else v[R][4 * j + k / 2].x = 0.f;
                        }
                    }
                }
                if (a.post_scale != 1.f) {
                    #pragma unroll
                    for (int k = 0; k < 4; ++k) v[R][4 * j + k] = f2mul(v[R][4 * j + k], make_float2(a.post_scale, a.post_scale));
                }
                if (ASYM) {
                    #pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const float2 w = v[R][4 * j + k];
                        amax = fmaxf(amax, fmaxf(w.x, w.y));
                        nmin = fmaxf(nmin, fmaxf(-w.x, -w.y));
                    }
                } else {
                    #pragma unroll
                    for (int k = 0; k < 4; ++k)
                        amax = fmaxf(amax, fmaxf(fabsf(v[R][4 * j + k].x), fabsf(v[R][4 * j + k].y)));
                }
                if (a.v_dbg != nullptr) {
                    float4* d4 = reinterpret_cast<float4*>(a.v_dbg + (size_t)row * K + e0);
                    d4[0] = make_float4(v[R][4 * j].x, v[R][4 * j].y, v[R][4 * j + 1].x, v[R][4 * j + 1].y);
                    d4[1] = make_float4(v[R][4 * j + 2].x, v[R][4 * j + 2].y, v[R][4 * j + 3].x, v[R][4 * j + 3].y);
                }
            }
        }
        if (!ok) break;
        #pragma unroll
        for (int m = 16; m > 0; m >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, m));
        if (ASYM) {
            #pragma unroll
            for (int m = 16; m > 0; m >>= 1) nmin = fmaxf(nmin, __shfl_xor_sync(0xffffffffu, nmin, m));
        }
        if (lane == 0) {
            ctl->red[g][warp] = amax;
            if (ASYM) ctl->red[g][4 + warp] = nmin;
        }
        group_sync();
        amax = fmaxf(fmaxf(ctl->red[g][0], ctl->red[g][1]), fmaxf(ctl->red[g][2], ctl->red[g][3]));
        if (ASYM) nmin = fmaxf(fmaxf(ctl->red[g][4], ctl->red[g][5]), fmaxf(ctl->red[g][6], ctl->red[g][7]));

        const float range = ASYM ? __fadd_rn(amax, nmin) : amax;     // X_max - X_min, or amax
        const bool nz = range > 0.f;
        const float s = nz ? __fdiv_rn(range, qmax) : 0.f;
        const float r = nz ? __fdiv_rn(qmax, range) : 0.f;
        const float2 rr = make_float2(r, r);
        const int zp = ASYM ? min(max(__float2int_rn(__fmul_rn(nmin, r)), 0), a.qmax) : 0;
        if (gtid == 0) {
            a.s[row] = s;
            if (ASYM) a.z[row] = zp;
        }
        if (ASYM && a.Xe != nullptr && gtid < 8)
            store_zero_point_columns(a.Xe + (size_t)row * (K + 128) + K, zp, gtid);
        #pragma unroll
        for (int R = 0; R < NR; ++R) {
            const int rbase = R * 4096;
            const int nch = min(4, (K - rbase) >> 10);
            #pragma unroll
            for (int j = 0; j < 4; ++j) {
                if (j >= nch) continue;
                const int e0 = rbase + j * 1024 + warp * 256 + 8 * lane;
                float2 qf[4], qt[4];
                #pragma unroll
                for (int k = 0; k < 4; ++k) quant2(v[R][4 * j + k], rr, qf[k], qt[k]);
                if (ASYM || a.qmax > 15) {
                    int qi[8];
                    #pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        qi[2 * k] = code_of(qt[k].x);
                        qi[2 * k + 1] = code_of(qt[k].y);
                    }
                    if (ASYM) {          // codes in [0, qmax]: unsigned nibbles and E4M3 bytes
                        int q[8];
                        #pragma unroll
                        for (int k = 0; k < 8; ++k) q[k] = min(max(qi[k] + zp, 0), a.qmax);
                        *reinterpret_cast<uint32_t*>(a.Xq + (size_t)row * (K / 2) + e0 / 2) = pack8(q);
                        if (a.Xe != nullptr) *reinterpret_cast<uint2*>(a.Xe + (size_t)row * (K + 128) + e0) = e4m3_of8(q);
                    } else {             // 8-bit codes: bytes and their E4M3 split
                        uint2 bytes, eh, el;
                        split_codes8(qi, bytes, eh, el);
                        *reinterpret_cast<uint2*>(a.Xq + (size_t)row * K + e0) = bytes;
                        if (a.Xe != nullptr) {
                            *reinterpret_cast<uint2*>(a.Xe + (size_t)row * 2 * K + e0) = eh;
                            *reinterpret_cast<uint2*>(a.Xe + (size_t)row * 2 * K + K + e0) = el;
                        }
                    }
                    continue;
                }
                uint32_t nib;
                uint2 e4;
                pack_codes8(qf, qt, nib, e4);
                if (a.Xq != nullptr) *reinterpret_cast<uint32_t*>(a.Xq + (size_t)row * (K / 2) + e0 / 2) = nib;
                if (a.Xe != nullptr) *reinterpret_cast<uint2*>(a.Xe + (size_t)row * K + e0) = e4;
            }
        }
    }
    if (!ok && gtid == 0) {
        // record the timeout, then give the copies this group issued (the
        // row that did not arrive, and the one after it) a bounded chance to
        // land before the CTA's shared memory is released
        if (a.status != nullptr) atomicOr(a.status, STATUS_TIMEOUT_QUANT);
        volatile int never = 0;
        for (int k = it; k < it + 2; ++k)
            if (first + k * stride < a.L)
                mbar_wait_bounded(smem_addr(&ctl->full[g][k & 1]), (uint32_t)((k >> 1) & 1), &never);
    }
}

// Tensor map of the rows of X as 128-byte lines ([L * K * esize / 128][128]
// bytes), boxes of LINES_PER_COPY lines with the 128-byte swizzle.
bool encode_rows_tmap(CUtensorMap* m, const void* X, size_t bytes) {
    const PFN_cuTensorMapEncodeTiled_v12000 fn = tensor_map_encoder();
    if (fn == nullptr) return false;
    const cuuint64_t dims[2] = {128, bytes / 128};
    const cuuint64_t strides[1] = {128};
    const cuuint32_t box[2] = {128, rowsk::LINES_PER_COPY};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(X), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int NR, typename Tin, bool ASYM, bool RES>
cudaError_t launch_rows_inst(const QuantArgs& a, const CUtensorMap& tm, cudaStream_t stream) {
    const rowsk::Layout lay(a.K, (int)sizeof(Tin), RES);
    auto kernel = sgat_quant_rows_kernel<NR, Tin, ASYM, RES>;
    // CTAs resident per SM at this size (once per device and size)
    static DeviceCache<int> attr;
    int done = 0;
    cudaError_t e = attr.get(&done, [&](int, int* v) {
        *v = 1;
        return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, 227 * 1024);
    });
    if (e != cudaSuccess) return e;
    int per_sm = 0;
    if ((e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, rowsk::THREADS, lay.total)) != cudaSuccess)
        return e;
    if (per_sm < 1) return cudaErrorInvalidConfiguration;
    const long long groups = ((long long)a.L + rowsk::G - 1) / rowsk::G;
    const long long slots = (long long)num_sms() * per_sm;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1] = {pdl_attribute()};
    cfg.gridDim = dim3((unsigned)(groups < slots ? groups : slots));
    cfg.blockDim = dim3(rowsk::THREADS);
    cfg.dynamicSmemBytes = lay.total;
    cfg.stream = stream;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, a, tm);
}

template <int NR, typename Tin>
cudaError_t launch_rows_nr(const QuantArgs& a, cudaStream_t stream) {
    CUtensorMap tm;
    if (!encode_rows_tmap(&tm, a.X, (size_t)a.L * a.K * sizeof(Tin))) return cudaErrorInvalidValue;
    const bool res = a.K <= rowsk::SMOOTH_RESIDENT_MAX_K;
    if (a.asym)
        return res ? launch_rows_inst<NR, Tin, true, true>(a, tm, stream)
                   : launch_rows_inst<NR, Tin, true, false>(a, tm, stream);
    return res ? launch_rows_inst<NR, Tin, false, true>(a, tm, stream)
               : launch_rows_inst<NR, Tin, false, false>(a, tm, stream);
}

template <typename Tin>
cudaError_t launch_rows(const QuantArgs& a, cudaStream_t stream) {
    switch ((a.K + 4095) / 4096) {
        case 1: return launch_rows_nr<1, Tin>(a, stream);
        case 2: return launch_rows_nr<2, Tin>(a, stream);
        case 3: return launch_rows_nr<3, Tin>(a, stream);
        case 4: return launch_rows_nr<4, Tin>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

template <int E, typename Tin>
cudaError_t launch_e(const QuantArgs& a, cudaStream_t stream) {
    constexpr int C = 32 * E;
    const int n = (a.K + C - 1) / C;                 // chunks per row
    const int wpr = n < 8 ? n : 8;                   // warps per row (a multiple of hb / C)
    const int rpc = wpr <= 4 ? 8 / wpr : 1;          // rows per CTA
    const int nc = (n + wpr - 1) / wpr;              // rounds
    const int warps = wpr * rpc;
    const size_t smem = (size_t)warps * (C + 32) * 4 + 16 * 4;
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
    // hb >= 1024 and up to 16384 features: the persistent row kernel (when
    // its shared memory fits); otherwise a warp's chunk is 1024 elements
    // (hb >= 1024, blocks finish across warps) or 512 elements holding
    // 512 / hb blocks
    if (a.hb >= 1024 && a.K % 1024 == 0 && a.K <= 16384 &&
        rowsk::Layout(a.K, (int)sizeof(Tin), a.K <= rowsk::SMOOTH_RESIDENT_MAX_K).total <= 227 * 1024)
        return launch_rows<Tin>(a, stream);
    return a.hb >= 1024 ? launch_e<32, Tin>(a, stream) : launch_e<16, Tin>(a, stream);
}

}  // namespace

cudaError_t launch_sgat_quant(const QuantArgs& args, cudaStream_t stream) {
    if (args.L == 0) return cudaSuccess;
    QuantArgs a = args;
    if (a.status == nullptr) a.status = device_status_word();
    switch (a.x_dtype) {
        case STARQ_F16: return launch_typed<__half>(a, stream);
        case STARQ_BF16: return launch_typed<__nv_bfloat16>(a, stream);
        case STARQ_F32: return launch_typed<float>(a, stream);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace starq
