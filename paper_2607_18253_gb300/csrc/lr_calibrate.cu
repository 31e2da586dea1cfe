// Least-squares calibration of the Eq. 9 batch-time coefficients per model from a
// log of executed token batches (Sec. 4.1: the coefficients are calibrated from
// observed token-batch processing times).
//
// One pass over the log accumulates, per model, the normal equations G = sum x x^T,
// b = sum x t and the row count in fp64; the feature products are exact integers
// below 2^53.  A per-model solve then forms the chosen regressors (the paper's four,
// with F1 + F2 as the token count, or the five features), scales the system by
// powers of two so that its diagonal is near 1 (exact, and it restores the
// conditioning the raw feature magnitudes take away) and solves it by Cholesky.
#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;

// Packed upper triangle of a 5x5 symmetric matrix.
__device__ __forceinline__ int tri(int a, int b) {
    if (a > b) {
        const int t = a;
        a = b;
        b = t;
    }
    return a * kCalCols - a * (a - 1) / 2 + (b - a);
}

// Rows grouped by model are the common case (per-instance logs), so each thread keeps
// the sums of the model it is reading in registers and flushes them to shared memory
// only when the model changes.
__global__ void __launch_bounds__(256) k_calib_accum(long long N, const long long *F, const int32_t *model,
                                                     const double *time, int M, double *acc, DevCtl *ctl) {
    extern __shared__ double sacc[];  // [M][kCalAcc]
    for (int i = threadIdx.x; i < M * kCalAcc; i += blockDim.x) sacc[i] = 0.0;
    __syncthreads();
    double r[kCalAcc];
#pragma unroll
    for (int k = 0; k < kCalAcc; ++k) r[k] = 0.0;
    int cur = -1;
    bool bad = false;
    auto flush = [&]() {
        if (cur >= 0)
            for (int k = 0; k < kCalAcc; ++k) atomicAdd(&sacc[cur * kCalAcc + k], r[k]);
#pragma unroll
        for (int k = 0; k < kCalAcc; ++k) r[k] = 0.0;
    };
    // contiguous slices per thread keep a thread's rows within one model's group
    const long long nthreads = (long long)gridDim.x * blockDim.x;
    const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    const long long per = (N + nthreads - 1) / nthreads;
    const long long i0 = tid * per, i1 = min(N, i0 + per);
    for (long long i = i0; i < i1; ++i) {
        const int m = model[i];
        const double t = time[i];
        if (m < 0 || m >= M || !isfinite(t)) {
            bad = true;
            continue;
        }
        if (m != cur) {
            flush();
            cur = m;
        }
        double x[kCalCols];
#pragma unroll
        for (int k = 0; k < kCalCols; ++k) x[k] = (double)F[i * kCalCols + k];
#pragma unroll
        for (int a = 0; a < kCalCols; ++a) {
#pragma unroll
            for (int b = a; b < kCalCols; ++b) r[tri(a, b)] = __fma_rn(x[a], x[b], r[tri(a, b)]);
            r[15 + a] = __fma_rn(x[a], t, r[15 + a]);
        }
        r[20] += 1.0;
    }
    flush();
    if (__any_sync(kFull, bad) && (threadIdx.x & 31) == 0) record_status(ctl, kEInval);
    __syncthreads();
    for (int i = threadIdx.x; i < M * kCalAcc; i += blockDim.x)
        if (sacc[i] != 0.0) atomicAdd(&acc[i], sacc[i]);
}

// One thread per model: regressors, power-of-two Jacobi scaling, Cholesky, unscaling.
__global__ void k_calib_solve(int M, const double *acc, int shared_beta1, double *coef) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M) return;
    const double *s = acc + (size_t)m * kCalAcc;
    // regressor c of the fit is the sum of features grp[c]
    const int d = shared_beta1 ? 4 : 5;
    int lo[5], hi[5];  // feature range [lo, hi] of each regressor
    if (shared_beta1) {
        const int l4[4] = {0, 1, 3, 4}, h4[4] = {0, 2, 3, 4};
        for (int c = 0; c < 4; ++c) {
            lo[c] = l4[c];
            hi[c] = h4[c];
        }
    } else {
        for (int c = 0; c < 5; ++c) lo[c] = hi[c] = c;
    }
    double G[5][5], b[5];
    for (int p = 0; p < d; ++p) {
        b[p] = 0.0;
        for (int a = lo[p]; a <= hi[p]; ++a) b[p] += s[15 + a];
        for (int q = 0; q < d; ++q) {
            double g = 0.0;
            for (int a = lo[p]; a <= hi[p]; ++a)
                for (int c = lo[q]; c <= hi[q]; ++c) g += s[tri(a, c)];
            G[p][q] = g;
        }
    }
    double out[5];
    const double nan = __longlong_as_double(0x7ff8000000000000LL);
    bool ok = s[20] >= (double)d;
    // scale regressor p by 2^-e_p with 2^e_p ~ sqrt(G_pp)
    double sc[5];
    for (int p = 0; p < d && ok; ++p) {
        ok = G[p][p] > 0.0;
        int e = 0;
        if (ok) frexp(sqrt(G[p][p]), &e);
        sc[p] = ldexp(1.0, -e);
    }
    double L[5][5];
    for (int p = 0; p < d && ok; ++p)
        for (int q = 0; q <= p && ok; ++q) {
            double v = G[p][q] * sc[p] * sc[q];
            for (int k = 0; k < q; ++k) v -= L[p][k] * L[q][k];
            if (p == q) {
                ok = v > 1e-13;  // rank-deficient design
                if (ok) L[p][p] = sqrt(v);
            } else {
                L[p][q] = v / L[q][q];
            }
        }
    if (ok) {
        double z[5], w[5];
        for (int p = 0; p < d; ++p) {
            double v = b[p] * sc[p];
            for (int k = 0; k < p; ++k) v -= L[p][k] * z[k];
            z[p] = v / L[p][p];
        }
        for (int p = d - 1; p >= 0; --p) {
            double v = z[p];
            for (int k = p + 1; k < d; ++k) v -= L[k][p] * w[k];
            w[p] = v / L[p][p];
        }
        for (int p = 0; p < d; ++p) w[p] *= sc[p];
        if (shared_beta1) {
            out[0] = w[0];
            out[1] = out[2] = w[1];
            out[3] = w[2];
            out[4] = w[3];
        } else {
            for (int p = 0; p < 5; ++p) out[p] = w[p];
        }
    } else {
        for (int p = 0; p < 5; ++p) out[p] = nan;
    }
    for (int p = 0; p < 5; ++p) coef[(size_t)m * 5 + p] = out[p];
}

}  // namespace

cudaError_t launch_calibrate(long long N, const long long *F, const int32_t *model, const double *time, int M,
                             int shared_beta1, double *acc, double *coef, DevCtl *ctl, int grid, cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(acc, 0, sizeof(double) * (size_t)M * kCalAcc, st);
    if (e != cudaSuccess) return e;
    if (N > 0) {
        k_calib_accum<<<grid, 256, sizeof(double) * (size_t)M * kCalAcc, st>>>(N, F, model, time, M, acc, ctl);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    k_calib_solve<<<(M + 63) / 64, 64, 0, st>>>(M, acc, shared_beta1, coef);
    return cudaGetLastError();
}

cudaError_t set_calib_smem(int M) {
    return cudaFuncSetAttribute(k_calib_accum, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                (int)(sizeof(double) * (size_t)M * kCalAcc));
}

}  // namespace lr
