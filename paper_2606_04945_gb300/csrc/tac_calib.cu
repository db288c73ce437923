// Closed-form TAC calibration on the GPU (App. C), in float64.
//
// From paired calibration activations Z_fp, Z_q [N][C] (the full-precision
// and quantised attention outputs of the same N tokens) and block size g:
//
//   tac_stats_kernel   the token reduction: per block b and representation,
//                      the sums s_b = sum_i z_ib and S_b = sum_i z_ib z_ib^T.
//                      Grid (block, token chunk, representation); each CTA
//                      stages batches of 32 tokens of its block in shared
//                      memory and keeps 4 x 4 tiles of the upper triangle of
//                      S_b in registers, then adds them to the float64
//                      accumulators in the workspace.
//   tac_power_kernel   one CTA per block and representation: mu = s / N,
//                      Sigma = S / N - mu mu^T (population statistics);
//                      F1 = (Sigma^FP)^(1/2), F2 = (Sigma^Q + lambda_b I)^(-1/2)
//                      with lambda_b = rho max(Tr Sigma^Q / g, eps) and
//                      A^p = Q diag(max(lambda_i, 1e-12)^p) Q^T from a
//                      symmetric eigendecomposition;
//   tac_final_kernel   one CTA per block: M = F1 F2, its singular values
//                      smoothed toward their mean by eta, M_final =
//                      (1 - alpha) M_sv + alpha I, d = mu^FP - M_final mu^Q.
//
// The eigendecompositions are parallel cyclic Jacobi: each sweep visits
// every index pair once in n - 1 steps of n / 2 disjoint rotations (round-
// robin order), the matrix in float64 and the accumulated rotations in
// float32 in shared memory (row stride g + 1). The SVD of M is the one-
// sided (Hestenes) Jacobi method on the same schedule: rotations of column
// pairs until all columns are orthogonal, so that M V = U diag(sigma) with
// sigma the column norms. It works on M itself, not on M^T M, and so keeps
// the small singular values of an ill-conditioned M (fewer calibration
// tokens than channels) accurate.
#include "common.cuh"
#include "tac_calib.cuh"

namespace starq {
namespace {

constexpr int CAL_THREADS = 256;
constexpr int STAT_TOK = 32;          // tokens per staged batch (32 KB of doubles at g = 128)
constexpr int CAL_MAX_G = 128;
constexpr int STAT_TPT = 3;           // 4 x 4 upper tiles per thread: ceil(528 / 256) at g = 128
constexpr int JACOBI_SWEEPS = 40;

template <typename T> __device__ __forceinline__ double to_d(T x);
template <> __device__ __forceinline__ double to_d<__half>(__half x) { return (double)__half2float(x); }
template <> __device__ __forceinline__ double to_d<__nv_bfloat16>(__nv_bfloat16 x) {
    return (double)__bfloat162float(x);
}
template <> __device__ __forceinline__ double to_d<float>(float x) { return (double)x; }

// Workspace, in doubles: s [2][B][g] | S [2][B][g][g] | F1, F2, MM [B][g][g].
struct Ws {
    double *s, *S, *F1, *F2, *MM;
    __host__ __device__ Ws(double* w, int B, int g) {
        s = w;
        S = s + 2 * (size_t)B * g;
        F1 = S + 2 * (size_t)B * g * g;
        F2 = F1 + (size_t)B * g * g;
        MM = F2 + (size_t)B * g * g;
    }
};

template <typename T>
__global__ void __launch_bounds__(CAL_THREADS) tac_stats_kernel(CalArgs a, int per) {
    __shared__ double zs[STAT_TOK * CAL_MAX_G];
    const int g = a.g, B = a.C / g;
    const int b = blockIdx.x, rep = blockIdx.z;
    const T* Z = static_cast<const T*>(rep == 0 ? a.Z_fp : a.Z_q);
    const int t0 = blockIdx.y * per, t1 = min(a.N, t0 + per);
    const Ws w(a.ws, B, g);
    const int T4 = g / 4, ntiles = T4 * (T4 + 1) / 2;
    // up to STAT_TPT tiles per thread when there are more tiles than
    // threads; with fewer (small g), `groups` threads share each tile and
    // split the batch's tokens between them
    const int groups = ntiles >= CAL_THREADS ? 1 : CAL_THREADS / ntiles;
    const int grp = groups > 1 ? threadIdx.x / ntiles : 0;
    int ti[STAT_TPT], tj[STAT_TPT];
    double acc[STAT_TPT][16];
    #pragma unroll
    for (int k = 0; k < STAT_TPT; ++k) {
        int t = groups == 1 ? threadIdx.x + k * CAL_THREADS
                            : (k == 0 && grp < groups ? threadIdx.x % ntiles : ntiles);
        int j = 0;                                      // column-major upper triangle: t = j (j + 1) / 2 + i
        while (t >= 0 && (j + 1) * (j + 2) / 2 <= t) ++j;
        ti[k] = t < ntiles ? t - j * (j + 1) / 2 : -1;
        tj[k] = j;
        #pragma unroll
        for (int e = 0; e < 16; ++e) acc[k][e] = 0.0;
    }
    double col = 0.0;
    for (int tb = t0; tb < t1; tb += STAT_TOK) {
        const int nt = min(STAT_TOK, t1 - tb);
        __syncthreads();
        for (int e = threadIdx.x; e < nt * g; e += CAL_THREADS) {
            const int r = e / g, c = e - r * g;
            zs[r * g + c] = to_d(Z[(size_t)(tb + r) * a.C + (size_t)b * g + c]);
        }
        __syncthreads();
        if (threadIdx.x < g)
            for (int r = 0; r < nt; ++r) col += zs[r * g + threadIdx.x];
        #pragma unroll
        for (int k = 0; k < STAT_TPT; ++k) {
            if (ti[k] < 0) continue;
            const double* zi = zs + 4 * ti[k];
            const double* zj = zs + 4 * tj[k];
            for (int r = grp; r < nt; r += groups) {
                double x[4], y[4];
                #pragma unroll
                for (int u = 0; u < 4; ++u) { x[u] = zi[r * g + u]; y[u] = zj[r * g + u]; }
                #pragma unroll
                for (int u = 0; u < 4; ++u)
                    #pragma unroll
                    for (int v = 0; v < 4; ++v) acc[k][4 * u + v] = fma(x[u], y[v], acc[k][4 * u + v]);
            }
        }
    }
    if (threadIdx.x < g) atomicAdd(w.s + ((size_t)rep * B + b) * g + threadIdx.x, col);
    double* S = w.S + ((size_t)rep * B + b) * g * g;
    #pragma unroll
    for (int k = 0; k < STAT_TPT; ++k) {
        if (ti[k] < 0) continue;
        #pragma unroll
        for (int u = 0; u < 4; ++u)
            #pragma unroll
            for (int v = 0; v < 4; ++v)
                atomicAdd(S + (size_t)(4 * ti[k] + u) * g + 4 * tj[k] + v, acc[k][4 * u + v]);
    }
}

// ---- CTA-wide helpers of the solve (all threads call them) ---------------

__device__ double block_sum(double v, double* red) {
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) v += __shfl_xor_sync(0xffffffffu, v, m);
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    double t = 0.0;
    #pragma unroll
    for (int k = 0; k < CAL_THREADS / 32; ++k) t += red[k];
    return t;
}

// Symmetric eigendecomposition of A (g x g, row stride g + 1, float64) by
// parallel cyclic Jacobi. On return A's diagonal holds the eigenvalues
// (copied to lam) and V's columns the eigenvectors (float32, stride g + 1).
__device__ void jacobi(double* A, float* V, double* lam, double* cs, int* pq, double* red, int g) {
    const int ld = g + 1, half = g / 2;
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
        const int i = e / g, j = e - i * g;
        V[i * ld + j] = i == j ? 1.f : 0.f;
    }
    __syncthreads();
    for (int sweep = 0; sweep < JACOBI_SWEEPS; ++sweep) {
        double off = 0.0, dia = 0.0;
        for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
            const int i = e / g, j = e - i * g;
            const double x = A[i * ld + j];
            if (i == j) dia += x * x; else off += x * x;
        }
        off = block_sum(off, red);
        dia = block_sum(dia, red);
        if (off <= 1e-26 * dia) break;                    // off-diagonal norm below 1e-13 of the diagonal's
        for (int step = 0; step < g - 1; ++step) {
            if (threadIdx.x < half) {
                const int k = threadIdx.x;
                int p = k == 0 ? 0 : (k - 1 + step) % (g - 1) + 1;
                int q = (g - 2 - k + step) % (g - 1) + 1;        // position g - 1 - k of the round
                if (p > q) { const int t = p; p = q; q = t; }
                const double apq = A[p * ld + q];
                double c = 1.0, s = 0.0;
                if (apq != 0.0) {
                    const double theta = (A[q * ld + q] - A[p * ld + p]) / (2.0 * apq);
                    const double t = (theta >= 0.0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
                    c = 1.0 / sqrt(t * t + 1.0);
                    s = t * c;
                }
                cs[k] = c;
                cs[half + k] = s;
                pq[k] = p;
                pq[half + k] = q;
            }
            __syncthreads();
            for (int e = threadIdx.x; e < half * g; e += CAL_THREADS) {     // rows p, q
                const int k = e / g, j = e - k * g;
                const int p = pq[k], q = pq[half + k];
                const double c = cs[k], s = cs[half + k];
                const double x = A[p * ld + j], y = A[q * ld + j];
                A[p * ld + j] = c * x - s * y;
                A[q * ld + j] = s * x + c * y;
            }
            __syncthreads();
            for (int e = threadIdx.x; e < half * g; e += CAL_THREADS) {     // columns p, q (and of V)
                const int k = e / g, i = e - k * g;
                const int p = pq[k], q = pq[half + k];
                const double c = cs[k], s = cs[half + k];
                const double x = A[i * ld + p], y = A[i * ld + q];
                A[i * ld + p] = c * x - s * y;
                A[i * ld + q] = s * x + c * y;
                const float cf = (float)c, sf = (float)s;
                const float vx = V[i * ld + p], vy = V[i * ld + q];
                V[i * ld + p] = cf * vx - sf * vy;
                V[i * ld + q] = sf * vx + cf * vy;
            }
            __syncthreads();
        }
    }
    for (int i = threadIdx.x; i < g; i += CAL_THREADS) lam[i] = A[i * ld + i];
    __syncthreads();
}

__device__ double block_max(double v, double* red) {
    #pragma unroll
    for (int m = 16; m > 0; m >>= 1) v = fmax(v, __shfl_xor_sync(0xffffffffu, v, m));
    __syncthreads();
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
    __syncthreads();
    double t = 0.0;
    #pragma unroll
    for (int k = 0; k < CAL_THREADS / 32; ++k) t = fmax(t, red[k]);
    return t;
}

// One-sided Jacobi SVD of A (g x g, row stride g + 1, float64): rotations
// of column pairs (p, q) that make them orthogonal, applied to A and to V
// (float32, from I), until every pair's |a_p . a_q| / (|a_p| |a_q|) is
// below 1e-13 (float64 dot products of g <= 128 terms carry ~1e-14). On
// return A = M V holds U diag(sigma) column by column.
__device__ void svd_onesided(double* A, float* V, double* cs, int* pq, double* red, int g) {
    const int ld = g + 1, half = g / 2;
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
        const int i = e / g, j = e - i * g;
        V[i * ld + j] = i == j ? 1.f : 0.f;
    }
    __syncthreads();
    for (int sweep = 0; sweep < 2 * JACOBI_SWEEPS; ++sweep) {
        double worst = 0.0;
        for (int step = 0; step < g - 1; ++step) {
            if (threadIdx.x < half) {
                const int k = threadIdx.x;
                int p = k == 0 ? 0 : (k - 1 + step) % (g - 1) + 1;
                int q = (g - 2 - k + step) % (g - 1) + 1;
                if (p > q) { const int t = p; p = q; q = t; }
                double al = 0.0, be = 0.0, ga = 0.0;
                for (int i = 0; i < g; ++i) {
                    const double x = A[i * ld + p], y = A[i * ld + q];
                    al = fma(x, x, al);
                    be = fma(y, y, be);
                    ga = fma(x, y, ga);
                }
                double c = 1.0, s = 0.0;
                if (ga != 0.0 && al > 0.0 && be > 0.0) {
                    worst = fmax(worst, fabs(ga) / sqrt(al * be));
                    const double zeta = (be - al) / (2.0 * ga);
                    const double t = (zeta >= 0.0 ? 1.0 : -1.0) / (fabs(zeta) + sqrt(1.0 + zeta * zeta));
                    c = 1.0 / sqrt(1.0 + t * t);
                    s = c * t;
                }
                cs[k] = c;
                cs[half + k] = s;
                pq[k] = p;
                pq[half + k] = q;
            }
            __syncthreads();
            for (int e = threadIdx.x; e < half * g; e += CAL_THREADS) {     // columns p, q of A and V
                const int k = e / g, i = e - k * g;
                const int p = pq[k], q = pq[half + k];
                const double c = cs[k], s = cs[half + k];
                const double x = A[i * ld + p], y = A[i * ld + q];
                A[i * ld + p] = c * x - s * y;
                A[i * ld + q] = s * x + c * y;
                const float cf = (float)c, sf = (float)s;
                const float vx = V[i * ld + p], vy = V[i * ld + q];
                V[i * ld + p] = cf * vx - sf * vy;
                V[i * ld + q] = sf * vx + cf * vy;
            }
            __syncthreads();
        }
        if (block_max(worst, red) < 1e-13) break;
    }
}

// F = V diag(f) V^T (float64, dense g x g in global memory).
__device__ void spectral(double* F, const float* V, const double* f, int g) {
    const int ld = g + 1;
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
        const int i = e / g, j = e - i * g;
        double t = 0.0;
        for (int k = 0; k < g; ++k) t = fma((double)V[i * ld + k] * f[k], (double)V[j * ld + k], t);
        F[e] = t;
    }
    __syncthreads();
}

// Out = op(X) Y for dense g x g float64 matrices in global memory, op(X) =
// X or X^T; Y is staged in shared memory (row stride g + 1).
__device__ void matmul(double* Out, const double* X, const double* Y, bool transX, double* Ys, int g) {
    const int ld = g + 1;
    __syncthreads();
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) Ys[(e / g) * ld + e % g] = Y[e];
    __syncthreads();
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
        const int i = e / g, j = e - i * g;
        double t = 0.0;
        for (int k = 0; k < g; ++k) t = fma(transX ? X[k * g + i] : X[i * g + k], Ys[k * ld + j], t);
        Out[e] = t;
    }
    __syncthreads();
}

// A <- (S / N - mu mu^T) + shift I, with S's upper triangle accumulated and
// mirrored.
__device__ void load_cov(double* A, const double* S, const double* mu, double invN, double shift, int g) {
    const int ld = g + 1;
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
        const int i = e / g, j = e - i * g;
        const double sij = i <= j ? S[(size_t)i * g + j] : S[(size_t)j * g + i];
        A[i * ld + j] = sij * invN - mu[i] * mu[j] + (i == j ? shift : 0.0);
    }
    __syncthreads();
}

// Shared-memory layout of the solve kernels: A (g x (g + 1) doubles), five
// g-vectors and the reduction scratch (doubles), the rotation pairs (ints),
// then V (g x (g + 1) floats).
struct SolveSmem {
    double *A, *mu_fp, *mu_q, *lam, *f, *cs, *red;
    int* pq;
    float* V;
    __device__ SolveSmem(uint8_t* raw, int g) {
        A = reinterpret_cast<double*>(raw);
        mu_fp = A + g * (g + 1);
        mu_q = mu_fp + g;
        lam = mu_q + g;
        f = lam + g;
        cs = f + g;
        red = cs + g;
        pq = reinterpret_cast<int*>(red + CAL_THREADS / 32);
        V = reinterpret_cast<float*>(pq + g);
    }
};

// grid (B, 2): the matrix functions of block b, F1 = (Sigma^FP)^(1/2)
// (blockIdx.y = 0) and F2 = (Sigma^Q + lambda_b I)^(-1/2) (blockIdx.y = 1),
// each Q diag(max(lambda_i, 1e-12)^p) Q^T.
__global__ void __launch_bounds__(CAL_THREADS) tac_power_kernel(CalArgs a) {
    extern __shared__ __align__(16) uint8_t cal_smem[];
    const int g = a.g, B = a.C / g, b = blockIdx.x, rep = blockIdx.y, ld = g + 1;
    SolveSmem sm(cal_smem, g);
    const Ws w(a.ws, B, g);
    const double invN = 1.0 / (double)a.N;
    const double* sv = w.s + ((size_t)rep * B + b) * g;
    for (int i = threadIdx.x; i < g; i += CAL_THREADS) sm.mu_fp[i] = sv[i] * invN;
    __syncthreads();
    load_cov(sm.A, w.S + ((size_t)rep * B + b) * g * g, sm.mu_fp, invN, 0.0, g);
    if (rep == 1) {                                   // damping (App. C)
        double tr = 0.0;
        for (int i = threadIdx.x; i < g; i += CAL_THREADS) tr += sm.A[i * ld + i];
        tr = block_sum(tr, sm.red);
        const double damp = a.rho * fmax(tr / (double)g, a.eps);
        for (int i = threadIdx.x; i < g; i += CAL_THREADS) sm.A[i * ld + i] += damp;
        __syncthreads();
    }
    jacobi(sm.A, sm.V, sm.lam, sm.cs, sm.pq, sm.red, g);
    for (int i = threadIdx.x; i < g; i += CAL_THREADS) {
        const double l = fmax(sm.lam[i], 1e-12);
        sm.f[i] = rep == 0 ? sqrt(l) : 1.0 / sqrt(l);
    }
    __syncthreads();
    spectral((rep == 0 ? w.F1 : w.F2) + (size_t)b * g * g, sm.V, sm.f, g);
}

// grid B: M = F1 F2, its SVD M V = U diag(sigma), the smoothed singular
// values, the identity shrinkage and the bias of block b.
__global__ void __launch_bounds__(CAL_THREADS) tac_final_kernel(CalArgs a) {
    extern __shared__ __align__(16) uint8_t cal_smem[];
    const int g = a.g, B = a.C / g, b = blockIdx.x, ld = g + 1;
    SolveSmem sm(cal_smem, g);
    const Ws w(a.ws, B, g);
    const double invN = 1.0 / (double)a.N;
    for (int i = threadIdx.x; i < g; i += CAL_THREADS) {
        sm.mu_fp[i] = w.s[(size_t)b * g + i] * invN;
        sm.mu_q[i] = w.s[((size_t)B + b) * g + i] * invN;
    }
    double* F1 = w.F1 + (size_t)b * g * g;
    double* F2 = w.F2 + (size_t)b * g * g;
    double* MM = w.MM + (size_t)b * g * g;
    double* A = sm.A;
    matmul(MM, F1, F2, false, A, g);
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) A[(e / g) * ld + e % g] = MM[e];
    __syncthreads();
    svd_onesided(A, sm.V, sm.cs, sm.pq, sm.red, g);
    double ssum = 0.0;
    for (int j = threadIdx.x; j < g; j += CAL_THREADS) {
        double t = 0.0;
        for (int i = 0; i < g; ++i) t = fma(A[i * ld + j], A[i * ld + j], t);
        sm.lam[j] = sqrt(t);
        ssum += sm.lam[j];
    }
    const double sbar = block_sum(ssum, sm.red) / (double)g;
    // singular values smoothed toward their mean: column j of U diag(sigma)
    // scaled by ((1 - eta) sigma_j + eta sbar) / sigma_j
    for (int j = threadIdx.x; j < g; j += CAL_THREADS)
        sm.f[j] = sm.lam[j] > 0.0 ? ((1.0 - a.eta) * sm.lam[j] + a.eta * sbar) / sm.lam[j] : 0.0;
    __syncthreads();
    // M_final = (1 - alpha) U diag(sigma') V^T + alpha I, and d
    float* Mo = a.M + (size_t)b * g * g;
    for (int e = threadIdx.x; e < g * g; e += CAL_THREADS) {
        const int i = e / g, k = e - i * g;
        double t = 0.0;
        for (int j = 0; j < g; ++j) t = fma(A[i * ld + j] * sm.f[j], (double)sm.V[k * ld + j], t);
        const double mf = (1.0 - a.alpha) * t + (i == k ? a.alpha : 0.0);
        F1[e] = mf;
        Mo[e] = (float)mf;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < g; i += CAL_THREADS) {
        double t = 0.0;
        for (int j = 0; j < g; ++j) t = fma(F1[(size_t)i * g + j], sm.mu_q[j], t);
        a.d[(size_t)b * g + i] = (float)(sm.mu_fp[i] - t);
    }
}

size_t solve_smem(int g) {
    return (size_t)g * (g + 1) * 8 + (size_t)(5 * g + CAL_THREADS / 32) * 8 + (size_t)g * 4 +
           (size_t)g * (g + 1) * 4;
}

template <typename T>
cudaError_t launch_stats(const CalArgs& a, cudaStream_t stream) {
    const int B = a.C / a.g;
    // about four CTAs per SM over both representations, at least 32 tokens each
    int chunks = (4 * num_sms() + 2 * B - 1) / (2 * B);
    const int max_chunks = (a.N + STAT_TOK - 1) / STAT_TOK;
    if (chunks > max_chunks) chunks = max_chunks;
    if (chunks < 1) chunks = 1;
    const int per = (a.N + chunks - 1) / chunks;
    tac_stats_kernel<T><<<dim3(B, chunks, 2), CAL_THREADS, 0, stream>>>(a, per);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_tac_calibrate(const CalArgs& a, cudaStream_t stream) {
    const int B = a.C / a.g;
    const Ws w(a.ws, B, a.g);
    cudaError_t e = cudaMemsetAsync(w.s, 0, (2 * (size_t)B * a.g + 2 * (size_t)B * a.g * a.g) * sizeof(double),
                                    stream);
    if (e != cudaSuccess) return e;
    switch (a.z_dtype) {
        case STARQ_F16: e = launch_stats<__half>(a, stream); break;
        case STARQ_BF16: e = launch_stats<__nv_bfloat16>(a, stream); break;
        case STARQ_F32: e = launch_stats<float>(a, stream); break;
        default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    const size_t smem = solve_smem(a.g);
    static DeviceCache<int> attr;
    int done = 0;
    e = attr.get(&done, [](int, int* v) {
        *v = 1;
        cudaError_t r = cudaFuncSetAttribute(tac_power_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)solve_smem(CAL_MAX_G));
        if (r != cudaSuccess) return r;
        return cudaFuncSetAttribute(tac_final_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    (int)solve_smem(CAL_MAX_G));
    });
    if (e != cudaSuccess) return e;
    tac_power_kernel<<<dim3(B, 2), CAL_THREADS, smem, stream>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    tac_final_kernel<<<B, CAL_THREADS, smem, stream>>>(a);
    return cudaGetLastError();
}

}  // namespace starq
