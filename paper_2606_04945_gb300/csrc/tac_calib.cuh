// Launcher interface of the TAC calibration kernels (tac_calib.cu), called
// by the C ABI after validation.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>

namespace starq {

struct CalArgs {
    const void* Z_fp; const void* Z_q; int z_dtype;   // [N][C] each
    int N; int C; int g;
    double rho, eps, eta, alpha;
    float* M; float* d;                              // [C/g][g][g], [C/g][g]
    double* ws;                                      // tac_calib_workspace_doubles(C, g) doubles
    unsigned* status;
};

// Doubles of workspace: per block the two representations' sums (2 g) and
// second moments (2 g g) and three g x g matrices of the solve.
inline size_t tac_calib_workspace_doubles(int C, int g) {
    return (size_t)(C / g) * (2 * (size_t)g + 5 * (size_t)g * g);
}

cudaError_t launch_tac_calibrate(const CalArgs& a, cudaStream_t stream);

}  // namespace starq
