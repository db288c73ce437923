// sgat_linear_noalloc: sgat_linear for callers that cannot allocate device
// memory.
//
// Some callers of this library are not allowed to call cudaMalloc at all:
// a serving runtime that plans every device buffer at start-up and owns the
// whole memory pool, a custom-operator or plugin interface that hands the
// operator only its input and output buffers, or a latency-critical path
// where cudaMalloc's implicit device synchronisation is unacceptable. Such a
// caller cannot provide the workspace that sgat_linear needs for its
// intermediates (packed codes, per-token scales, TAC output). This entry
// point uses a fixed scratch array that lives in the library's own device
// image instead, so it allocates nothing.
//
// The scratch is a file-scope __device__ array of STARQ_NOALLOC_SCRATCH_BYTES
// bytes; every GPU that loads the library holds it until the process exits.
// Host code cannot use the array's name as a device address, so the device
// address is looked up with cudaGetSymbolAddress once per device (with that
// device current) on the first call, cached, and handed to sgat_linear as
// its workspace. The cached address belongs to the device's current primary
// context: after cudaDeviceReset it is stale, and the process must not call
// this entry point on that device again.
#include <cstdio>
#include <mutex>

#include "common.cuh"

namespace starq {
namespace {

static __device__ __align__(256) uint8_t g_noalloc_scratch[STARQ_NOALLOC_SCRATCH_BYTES];

std::mutex g_scratch_mu;
void* g_scratch_addr[64] = {nullptr};

// Device address of the scratch array on the current device (looked up once
// per device). Returns nullptr and sets *rc on failure.
void* scratch_address(int* rc, cudaError_t* err) {
    int dev = 0;
    *err = cudaGetDevice(&dev);
    if (*err != cudaSuccess || dev < 0 || dev >= 64) {
        *rc = STARQ_ERR_CUDA;
        return nullptr;
    }
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (g_scratch_addr[dev] == nullptr) {
        void* p = nullptr;
        *err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (*err != cudaSuccess || p == nullptr) {
            *rc = STARQ_ERR_CUDA;
            return nullptr;
        }
        g_scratch_addr[dev] = p;
    }
    *rc = STARQ_OK;
    return g_scratch_addr[dev];
}

}  // namespace
}  // namespace starq

extern "C" int sgat_linear_noalloc(const void* X, int x_dtype, int L, int K, const uint8_t* mask,
                                   const float* a_m, const float* a_u, int hb, int d_sh, int d_m,
                                   int d_u, const float* tac_M, const float* tac_d, int tac_g, const void* tac_Mp,
                                   const uint8_t* Wq, const uint8_t* We, const float* s_w, const float* bias, int N,
                                   int bits, void* Y, int y_dtype, void* stream) {
    const size_t need = sgat_linear_workspace_size_bits(L, K, tac_M != nullptr, bits);
    if (L > 0 && need > (size_t)STARQ_NOALLOC_SCRATCH_BYTES) {
        char msg[160];
        snprintf(msg, sizeof(msg),
                 "sgat_linear_noalloc: L=%d, K=%d%s needs %zu scratch bytes, above the fixed %zu",
                 L, K, tac_M ? " with TAC" : "", need, (size_t)STARQ_NOALLOC_SCRATCH_BYTES);
        return starq::report_error(STARQ_ERR_SHAPE, msg);
    }
    int rc = STARQ_OK;
    cudaError_t err = cudaSuccess;
    void* scratch = starq::scratch_address(&rc, &err);
    if (scratch == nullptr) {
        char msg[160];
        snprintf(msg, sizeof(msg), "sgat_linear_noalloc: scratch address lookup failed: %s",
                 cudaGetErrorString(err));
        return starq::report_error(rc, msg);
    }
    return starq::sgat_linear_scratch(X, x_dtype, L, K, mask, a_m, a_u, hb, d_sh, d_m, d_u, tac_M, tac_d, tac_g,
                                      tac_Mp, Wq, We, s_w, bias, N, bits, Y, y_dtype, scratch,
                                      (size_t)STARQ_NOALLOC_SCRATCH_BYTES, stream);
}
