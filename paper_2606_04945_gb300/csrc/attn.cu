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
//
// attn_vquant_kernel   V codes per channel, written as fp16 values into
//                      Vt [128 H][L] (keys contiguous: the K-major B
//                      operand of P V^T), and the channel scales t.
// attn_pv_tac_kernel   one CTA per (128-query tile, head); 8 softmax /
//                      epilogue warps, a TMA warp and an MMA warp;
//                      tcgen05 kind::f16 on one CTA (M = N = 128, K = 16).
//   pass 1  S = Q K^T chunk by chunk (128 keys, double-buffered in TMEM);
//           each thread keeps the running maximum of its row's half of S.
//   pass 2  S again; each thread turns its 64 scores into e = exp2((s - m)
//           log2(e) / sqrt(d)), adds them to l and writes the codes rne(255 e)
//           as fp16 into the shared A tile of P V^T. The MMA warp
//           accumulates P V^T one chunk behind the scores (exact integers).
//   epilogue  Z_hat from the accumulator, split into fp16 hi + lo (Z_hat =
//           hi + lo to ~2^-22), written as the A tiles of the TAC product;
//           Z_hi M_hi^T + Z_hi M_lo^T + Z_lo M_hi^T with M's prepared halves
//           (tac_prepare); + d; rounded to fp16 and stored by TMA.
// Shared memory: Q, two K chunks, two V chunks and P (six 32 KB tiles);
// after the passes the K buffers hold M's halves, the V buffers Z_hat's
// and the Q tile the output boxes. TMEM: two S buffers, the P V^T and the
// TAC accumulators (4 x 128 columns). Every wait is bounded.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "attn.cuh"
#include "common.cuh"

namespace starq {
namespace {

constexpr unsigned STATUS_TIMEOUT_ATTN = 1u << 4;
constexpr int ATT_THREADS = 320;
constexpr int ATT_TMA_WARP = 8, ATT_MMA_WARP = 9, ATT_SOFTMAX_THREADS = 256;
constexpr int TILE_BYTES = ATTN_TILE * ATTN_D * 2;            // 128 x 128 fp16, two 128-byte-swizzled atoms
constexpr int ATOM_BYTES = TILE_BYTES / 2;
constexpr int OFF_Q = 0, OFF_K = TILE_BYTES, OFF_V = 3 * TILE_BYTES, OFF_P = 5 * TILE_BYTES;
constexpr int ATT_TILES_BYTES = 6 * TILE_BYTES;

struct AttSm {
    uint64_t q_full, k_full[2], k_empty[2], v_full[2], v_empty[2], s_full[2], s_empty[2];
    uint64_t p_full, p_empty, pv_done, z_full, m_full, tac_done;
    uint32_t tmem_base;
    int abort;
    float xm[2][ATTN_TILE];            // row maxima / sums of the two column halves
};
constexpr size_t ATT_SMEM = ATT_TILES_BYTES + 1024 + sizeof(AttSm);

// log2(e) / sqrt(128): S (unscaled Q K^T) to base-2 exponents
constexpr float EXP_SCALE = (float)(1.4426950408889634 / 11.313708498984761);

__device__ __forceinline__ void named_sync_softmax() {
    asm volatile("bar.sync 1, %0;" :: "r"(ATT_SOFTMAX_THREADS) : "memory");
}

// Byte offset of element (row, col) of a 128 x 128 fp16 K-major tile (two
// atoms of 64 columns, 128-byte swizzle).
__device__ __forceinline__ uint32_t tile_off(int row, int col) {
    return (uint32_t)(col >> 6) * ATOM_BYTES + sw128_offset((uint32_t)row, (uint32_t)((col & 63) >> 3)) +
           (uint32_t)(col & 7) * 2;
}

__global__ void __launch_bounds__(256) attn_vquant_kernel(AttnArgs a) {
    __shared__ float red[16][32];
    __shared__ float rcp[32];
    __shared__ uint16_t tile[32][64 + 2];
    const __half* V = static_cast<const __half*>(a.V);
    const int c0 = blockIdx.x * 32;
    const int tid = threadIdx.x, cp = tid & 15, rg = tid >> 4;
    float m0 = 0.f, m1 = 0.f;
    for (int r = rg; r < a.L; r += 16) {
        const float2 f = __half22float2(*reinterpret_cast<const __half2*>(V + (size_t)r * a.ld + c0 + 2 * cp));
        m0 = fmaxf(m0, fabsf(f.x));
        m1 = fmaxf(m1, fabsf(f.y));
    }
    red[rg][2 * cp] = m0;
    red[rg][2 * cp + 1] = m1;
    __syncthreads();
    if (tid < 32) {
        float m = 0.f;
        #pragma unroll
        for (int g = 0; g < 16; ++g) m = fmaxf(m, red[g][tid]);
        const bool nz = m > 0.f;
        a.t[c0 + tid] = nz ? __fdiv_rn(m, 7.f) : 0.f;
        rcp[tid] = nz ? __fdiv_rn(7.f, m) : 0.f;
    }
    __syncthreads();
    for (int r0 = 0; r0 < a.L; r0 += 64) {
        #pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int r = r0 + rg + 16 * k;
            const float2 f = __half22float2(*reinterpret_cast<const __half2*>(V + (size_t)r * a.ld + c0 + 2 * cp));
            tile[2 * cp][rg + 16 * k] = __half_as_ushort(__float2half_rn(rintf(__fmul_rn(f.x, rcp[2 * cp]))));
            tile[2 * cp + 1][rg + 16 * k] = __half_as_ushort(__float2half_rn(rintf(__fmul_rn(f.y, rcp[2 * cp + 1]))));
        }
        __syncthreads();
        const int c = tid >> 3, rs = (tid & 7) * 8;
        uint32_t w[4];
        #pragma unroll
        for (int u = 0; u < 4; ++u) w[u] = (uint32_t)tile[c][rs + 2 * u] | ((uint32_t)tile[c][rs + 2 * u + 1] << 16);
        *reinterpret_cast<uint4*>(a.Vt + (size_t)(c0 + c) * a.L + r0 + rs) = make_uint4(w[0], w[1], w[2], w[3]);
        __syncthreads();
    }
}

__global__ void __launch_bounds__(ATT_THREADS, 1)
attn_pv_tac_kernel(AttnArgs a, const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_k,
                   const __grid_constant__ CUtensorMap tm_v, const __grid_constant__ CUtensorMap tm_z) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    AttSm* sh = reinterpret_cast<AttSm*>(smem_raw + (base - raw) + ATT_TILES_BYTES);
    const uint32_t sQ = base + OFF_Q, sK = base + OFF_K, sV = base + OFF_V, sP = base + OFF_P;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q0 = blockIdx.x * ATTN_TILE, h = blockIdx.y;
    const int nk = a.L / ATTN_TILE;
    volatile int* abort = &sh->abort;
    auto B = [&](const uint64_t& bar) { return smem_addr(&bar); };

    if (threadIdx.x == 0) {
        mbar_init(B(sh->q_full), 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(B(sh->k_full[b]), 1);
            mbar_init(B(sh->k_empty[b]), 1);
            mbar_init(B(sh->v_full[b]), 1);
            mbar_init(B(sh->v_empty[b]), 1);
            mbar_init(B(sh->s_full[b]), 1);
            mbar_init(B(sh->s_empty[b]), ATT_SOFTMAX_THREADS / 32);
        }
        mbar_init(B(sh->p_full), ATT_SOFTMAX_THREADS / 32);
        mbar_init(B(sh->p_empty), 1);
        mbar_init(B(sh->pv_done), 1);
        mbar_init(B(sh->z_full), ATT_SOFTMAX_THREADS / 32);
        mbar_init(B(sh->m_full), 1);
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
        if (elect_one()) {
            mbar_arrive_expect_tx(B(sh->q_full), TILE_BYTES);
            tma_load_2d(sQ, &tm_q, h * ATTN_D, q0, B(sh->q_full));
            tma_load_2d(sQ + ATOM_BYTES, &tm_q, h * ATTN_D + 64, q0, B(sh->q_full));
        }
        __syncwarp();
        for (int it = 0; it < 2 * nk && ok; ++it) {
            const int b = it & 1, n = it >> 1, kc = it < nk ? it : it - nk;
            if (!mbar_wait_bounded_warp(B(sh->k_empty[b]), (uint32_t)(n & 1) ^ 1u, abort)) { ok = false; break; }
            const uint32_t kt = sK + b * TILE_BYTES;
            if (elect_one()) {
                mbar_arrive_expect_tx(B(sh->k_full[b]), TILE_BYTES);
                tma_load_2d(kt, &tm_k, h * ATTN_D, kc * ATTN_TILE, B(sh->k_full[b]));
                tma_load_2d(kt + ATOM_BYTES, &tm_k, h * ATTN_D + 64, kc * ATTN_TILE, B(sh->k_full[b]));
            }
            __syncwarp();
            if (it >= nk) {
                const int j = it - nk, vb = j & 1, vn = j >> 1;
                if (!mbar_wait_bounded_warp(B(sh->v_empty[vb]), (uint32_t)(vn & 1) ^ 1u, abort)) { ok = false; break; }
                const uint32_t vt = sV + vb * TILE_BYTES;
                if (elect_one()) {
                    mbar_arrive_expect_tx(B(sh->v_full[vb]), TILE_BYTES);
                    tma_load_2d(vt, &tm_v, j * ATTN_TILE, h * ATTN_D, B(sh->v_full[vb]));
                    tma_load_2d(vt + ATOM_BYTES, &tm_v, j * ATTN_TILE + 64, h * ATTN_D, B(sh->v_full[vb]));
                }
                __syncwarp();
            }
        }
        // M's two halves into the K buffers once the last score MMA has read them
        for (int b = 0; b < 2 && ok; ++b)
            ok = mbar_wait_bounded_warp(B(sh->k_empty[b]), (uint32_t)((nk - 1) & 1), abort);
        if (ok && elect_one()) {
            mbar_arrive_expect_tx(B(sh->m_full), 2 * TILE_BYTES);
            bulk_load(sK, static_cast<const uint8_t*>(a.Mp) + (size_t)h * 2 * TILE_BYTES, 2 * TILE_BYTES,
                      B(sh->m_full));
        }
        __syncwarp();
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_ATTN); }
    } else if (warp == ATT_MMA_WARP) {
        // f16 A and B, f32 D, N = 128 (bits 17..22), M = 128 (bits 24..28)
        constexpr uint32_t IDESC = (1u << 4) | ((uint32_t)(ATTN_TILE >> 3) << 17) | ((uint32_t)(ATTN_TILE >> 4) << 24);
        bool ok = mbar_wait_bounded_warp(B(sh->q_full), 0, abort);
        auto mma_tile = [&](uint32_t d, uint32_t at, uint32_t bt, bool acc0) {
            if (elect_one()) {
                #pragma unroll
                for (int ks = 0; ks < ATTN_D / 16; ++ks) {
                    const uint32_t koff = (uint32_t)(ks >> 2) * ATOM_BYTES + (uint32_t)(ks & 3) * 32;
                    mma_f16(d, smem_desc_sw128(at + koff), smem_desc_sw128(bt + koff), IDESC, (acc0 || ks > 0) ? 1u : 0u);
                }
            }
            __syncwarp();
        };
        auto pv = [&](int j) {                 // P V^T of pass-2 chunk j
            const int vb = j & 1, vn = j >> 1;
            ok = ok && mbar_wait_bounded_warp(B(sh->p_full), (uint32_t)(j & 1), abort) &&
                 mbar_wait_bounded_warp(B(sh->v_full[vb]), (uint32_t)(vn & 1), abort);
            if (!ok) return;
            tc_fence_after();
            mma_tile(tmem + 256, sP, sV + vb * TILE_BYTES, j > 0);
            if (elect_one()) {
                tc_commit(B(sh->p_empty));
                tc_commit(B(sh->v_empty[vb]));
            }
            __syncwarp();
        };
        tc_fence_after();
        for (int it = 0; it < 2 * nk && ok; ++it) {
            const int b = it & 1, n = it >> 1;
            ok = mbar_wait_bounded_warp(B(sh->k_full[b]), (uint32_t)(n & 1), abort) &&
                 mbar_wait_bounded_warp(B(sh->s_empty[b]), (uint32_t)(n & 1) ^ 1u, abort);
            if (!ok) break;
            tc_fence_after();
            mma_tile(tmem + b * ATTN_TILE, sQ, sK + b * TILE_BYTES, false);
            if (elect_one()) {
                tc_commit(B(sh->k_empty[b]));
                tc_commit(B(sh->s_full[b]));
            }
            __syncwarp();
            if (it > nk) pv(it - 1 - nk);        // one chunk behind the scores
        }
        if (ok) pv(nk - 1);
        if (elect_one()) tc_commit(B(sh->pv_done));
        __syncwarp();
        ok = ok && mbar_wait_bounded_warp(B(sh->z_full), 0, abort) && mbar_wait_bounded_warp(B(sh->m_full), 0, abort);
        if (ok) {
            tc_fence_after();
            const uint32_t dt = tmem + 384;
            mma_tile(dt, sV, sK, false);                               // Z_hi M_hi^T
            mma_tile(dt, sV, sK + TILE_BYTES, true);                   // + Z_hi M_lo^T
            mma_tile(dt, sV + TILE_BYTES, sK, true);                   // + Z_lo M_hi^T
        }
        if (elect_one()) tc_commit(B(sh->tac_done));
        __syncwarp();
        if (lane == 0) {
            // every MMA of this thread has completed before TMEM is released
            volatile int never = 0;
            if (!mbar_wait_bounded(B(sh->tac_done), 0, &never)) ok = false;
            if (!ok) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_ATTN); }
        }
        __syncwarp();
    } else {
        const int quarter = warp & 3, hf = warp >> 2;
        const int row = quarter * 32 + lane;                // query within the tile (TMEM lane)
        const uint32_t tl = tmem + ((uint32_t)(quarter * 32) << 16);
        bool ok = true;
        uint32_t r[32];
        // pass 1: row maxima
        float mx = -INFINITY;
        for (int it = 0; it < nk && ok; ++it) {
            const int b = it & 1, n = it >> 1;
            if (!mbar_wait_bounded_warp(B(sh->s_full[b]), (uint32_t)(n & 1), abort)) { ok = false; break; }
            tc_fence_after();
            #pragma unroll
            for (int c = 0; c < 2; ++c) {
                tmem_ld_32x32b_x32(tl + b * ATTN_TILE + hf * 64 + c * 32, r);
                tmem_ld_wait();
                #pragma unroll
                for (int k = 0; k < 32; ++k) mx = fmaxf(mx, __uint_as_float(r[k]));
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(sh->s_empty[b]));
        }
        sh->xm[hf][row] = mx;
        named_sync_softmax();
        mx = fmaxf(sh->xm[0][row], sh->xm[1][row]);
        named_sync_softmax();
        // pass 2: probabilities, their codes and the row sums
        float l = 0.f;
        for (int j = 0; j < nk && ok; ++j) {
            const int it = nk + j, b = it & 1, n = it >> 1;
            if (!mbar_wait_bounded_warp(B(sh->s_full[b]), (uint32_t)(n & 1), abort)) { ok = false; break; }
            tc_fence_after();
            float e[64];
            #pragma unroll
            for (int c = 0; c < 2; ++c) {
                tmem_ld_32x32b_x32(tl + b * ATTN_TILE + hf * 64 + c * 32, r);
                tmem_ld_wait();
                #pragma unroll
                for (int k = 0; k < 32; ++k) e[32 * c + k] = exp2f((__uint_as_float(r[k]) - mx) * EXP_SCALE);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(sh->s_empty[b]));
            uint32_t packed[32];
            #pragma unroll
            for (int k = 0; k < 64; k += 2) {
                l += e[k];
                l += e[k + 1];
                const __half c0 = __float2half_rn(rintf(__fmul_rn(255.f, e[k])));
                const __half c1 = __float2half_rn(rintf(__fmul_rn(255.f, e[k + 1])));
                packed[k / 2] = (uint32_t)__half_as_ushort(c0) | ((uint32_t)__half_as_ushort(c1) << 16);
            }
            if (a.dbg_codes != nullptr) {
                uint8_t* dc = a.dbg_codes + ((size_t)h * a.L + q0 + row) * a.L + j * ATTN_TILE + hf * 64;
                #pragma unroll
                for (int k = 0; k < 32; ++k) {
                    dc[2 * k] = (uint8_t)__half2float(__ushort_as_half((uint16_t)(packed[k] & 0xFFFFu)));
                    dc[2 * k + 1] = (uint8_t)__half2float(__ushort_as_half((uint16_t)(packed[k] >> 16)));
                }
            }
            // the previous chunk's P V^T has read the P tile
            if (!mbar_wait_bounded_warp(B(sh->p_empty), (uint32_t)(j & 1) ^ 1u, abort)) { ok = false; break; }
            #pragma unroll
            for (int c = 0; c < 8; ++c)
                st_shared_v4(sP + tile_off(row, hf * 64 + 8 * c), packed[4 * c], packed[4 * c + 1], packed[4 * c + 2],
                             packed[4 * c + 3]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(sh->p_full));
        }
        sh->xm[hf][row] = l;
        named_sync_softmax();
        l = sh->xm[0][row] + sh->xm[1][row];
        const float sp = __fdiv_rn(1.f, __fmul_rn(255.f, l));
        if (a.dbg_l != nullptr && hf == 0) a.dbg_l[(size_t)h * a.L + q0 + row] = l;
        // epilogue 1: Z_hat = (acc sp) t as fp16 hi + lo A tiles of the TAC product
        ok = ok && mbar_wait_bounded_warp(B(sh->pv_done), 0, abort);
        if (ok) {
            tc_fence_after();
            #pragma unroll 1
            for (int c = 0; c < 2; ++c) {
                const int ch = hf * 64 + c * 32;
                tmem_ld_32x32b_x32(tl + 256 + ch, r);
                tmem_ld_wait();
                if (a.dbg_acc != nullptr) {
                    int32_t* da = a.dbg_acc + ((size_t)h * a.L + q0 + row) * ATTN_D + ch;
                    #pragma unroll
                    for (int k = 0; k < 32; ++k) da[k] = __float2int_rn(__uint_as_float(r[k]));
                }
                uint32_t hi[16], lo[16];
                #pragma unroll
                for (int k = 0; k < 32; k += 2) {
                    float z[2];
                    #pragma unroll
                    for (int u = 0; u < 2; ++u)
                        z[u] = __fmul_rn(__fmul_rn(__uint_as_float(r[k + u]), sp), __ldg(a.t + h * ATTN_D + ch + k + u));
                    const __half h0 = __float2half_rn(z[0]), h1 = __float2half_rn(z[1]);
                    const __half l0 = __float2half_rn(z[0] - __half2float(h0)), l1 = __float2half_rn(z[1] - __half2float(h1));
                    hi[k / 2] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
                    lo[k / 2] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1) << 16);
                }
                #pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint32_t off = tile_off(row, ch + 8 * q);
                    st_shared_v4(sV + off, hi[4 * q], hi[4 * q + 1], hi[4 * q + 2], hi[4 * q + 3]);
                    st_shared_v4(sV + TILE_BYTES + off, lo[4 * q], lo[4 * q + 1], lo[4 * q + 2], lo[4 * q + 3]);
                }
            }
            tc_fence_before();
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(B(sh->z_full));
        }
        // epilogue 2: + d, fp16, TMA store
        ok = ok && mbar_wait_bounded_warp(B(sh->tac_done), 0, abort);
        if (ok) {
            tc_fence_after();
            #pragma unroll 1
            for (int c = 0; c < 2; ++c) {
                const int ch = hf * 64 + c * 32;
                tmem_ld_32x32b_x32(tl + 384 + ch, r);
                tmem_ld_wait();
                const uint32_t box = sQ + (uint32_t)(warp * 2 + c) * 2048;
                #pragma unroll
                for (int g = 0; g < 4; ++g) {
                    uint32_t w[4];
                    #pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int k = 8 * g + 2 * u;
                        float y0 = __uint_as_float(r[k]), y1 = __uint_as_float(r[k + 1]);
                        if (a.d != nullptr) {
                            y0 = __fadd_rn(y0, __ldg(a.d + h * ATTN_D + ch + k));
                            y1 = __fadd_rn(y1, __ldg(a.d + h * ATTN_D + ch + k + 1));
                        }
                        const __half2 hv = __floats2half2_rn(y0, y1);
                        w[u] = *reinterpret_cast<const uint32_t*>(&hv);
                    }
                    st_shared_v4(box + lane * 64 + 16 * (g ^ ((lane >> 1) & 3)), w[0], w[1], w[2], w[3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tm_z, h * ATTN_D + ch, q0 + quarter * 32, box);
                    bulk_commit();
                }
            }
            if (lane == 0) bulk_wait0();
            __syncwarp();
        }
        if (!ok && lane == 0) { sh->abort = 1; atomicOr(a.status, STATUS_TIMEOUT_ATTN); }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == ATT_MMA_WARP) tmem_dealloc(tmem, 512);
}

bool encode_2d(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols, uint64_t row_elems,
               uint32_t box_rows, uint32_t box_cols, CUtensorMapSwizzle swz) {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (fn == nullptr) {
        cudaDriverEntryPointQueryResult q;
        void* f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) !=
                cudaSuccess || q != cudaDriverEntryPointSuccess || f == nullptr)
            return false;
        fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    }
    const cuuint64_t dims[2] = {cols, rows};
    const cuuint64_t strides[1] = {row_elems * 2};
    const cuuint32_t box[2] = {box_cols, box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_attention_pv_tac(const AttnArgs& a, cudaStream_t stream) {
    const int C = ATTN_D * a.H;
    attn_vquant_kernel<<<C / 32, 256, 0, stream>>>(a);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    CUtensorMap tq, tk, tv, tz;
    if (!encode_2d(&tq, a.Q, (uint64_t)a.L, (uint64_t)C, (uint64_t)a.ld, ATTN_TILE, 64, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_2d(&tk, a.K, (uint64_t)a.L, (uint64_t)C, (uint64_t)a.ld, ATTN_TILE, 64, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_2d(&tv, a.Vt, (uint64_t)C, (uint64_t)a.L, (uint64_t)a.L, ATTN_D, 64, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_2d(&tz, a.Z, (uint64_t)a.L, (uint64_t)C, (uint64_t)C, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B))
        return cudaErrorInvalidValue;
    static bool attr_set[64] = {false};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 64 && !attr_set[dev]) {
        e = cudaFuncSetAttribute(attn_pv_tac_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ATT_SMEM);
        if (e != cudaSuccess) return e;
        attr_set[dev] = true;
    }
    attn_pv_tac_kernel<<<dim3(a.L / ATTN_TILE, a.H), ATT_THREADS, ATT_SMEM, stream>>>(a, tq, tk, tv, tz);
    return cudaGetLastError();
}

}  // namespace starq
