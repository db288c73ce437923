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
    const void* Q; const void* K; const void* V;   // fp16 [L][ld] each; head h = columns h*128 ..
    int ld;                                        // row stride of Q, K, V in elements
    int L; int H;
    const void* Mp;                                // tac_prepare output for C = 128 H, g = 128
    const float* d;                                // [H][128] or NULL
    void* Z;                                       // fp16 [L][128 H] out (TAC applied)
    uint16_t* Vt;                                  // workspace: V codes as fp16, [128 H][L]
    float* t;                                      // workspace: V channel scales [128 H]
    uint8_t* dbg_codes; float* dbg_l; int32_t* dbg_acc;   // optional [H][L][L], [H][L], [H][L][128]
    unsigned* status;
};

inline size_t attn_workspace_bytes(int L, int H) {
    return ((size_t)ATTN_D * H * L * 2 + 255) / 256 * 256 + (size_t)ATTN_D * H * 4;
}

cudaError_t launch_attention_pv_tac(const AttnArgs& a, cudaStream_t stream);

}  // namespace starq
