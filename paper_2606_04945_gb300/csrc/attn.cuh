// Launcher interface of the quantised softmax-value product with the TAC
// epilogue (attn.cu), called by the C ABI after validation.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace starq {

constexpr int ATTN_D = 128;          // head dimension (= TAC block)
constexpr int ATTN_TILE = 128;       // query tile and key chunk

struct AttnArgs {
    const void* Q; const void* K; const void* V;   // [L][ld] each; query head h = Q columns h*128 ..,
                                                   // key/value head k = K, V columns k*128 ..
    int ld;                                        // row stride of Q, K, V in elements
    int L; int H;
    const void* Mp;                                // tac_prepare output for C = 128 H, g = 128
    const float* d;                                // [H][128] or NULL
    void* Z;                                       // [L][128 H] out (TAC applied)
    uint16_t* Vt;                                  // workspace: V codes as fp16, [128 Hkv][L]
    float* t;                                      // workspace: V channel scales [128 Hkv]
    uint8_t* dbg_codes; float* dbg_l; int32_t* dbg_acc;   // optional [H][L][L], [H][L], [H][L][128]
    unsigned* status;
    int Hkv = 0;                                   // key/value heads (H % Hkv == 0)
    int dtype = 0;                                 // STARQ_F16 or STARQ_BF16 (Q, K, V, Z)
};

// Workspace of Hkv key/value heads: the transposed V codes, then the scales.
inline size_t attn_workspace_bytes(int L, int Hkv) {
    return ((size_t)ATTN_D * Hkv * L * 2 + 255) / 256 * 256 + (size_t)ATTN_D * Hkv * 4;
}

cudaError_t launch_attention_pv_tac(const AttnArgs& a, cudaStream_t stream);

}  // namespace starq
