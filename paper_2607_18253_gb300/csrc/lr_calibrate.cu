// Least-squares calibration of the Eq. 9 batch-time coefficients per model from a
// log of executed token batches (Sec. 4.1: the coefficients are calibrated from
// observed token-batch processing times).
//
// One pass over the log accumulates, per model, the normal equations G = sum x x^T,
// b = sum x t and the row count as exact 128-bit integers (times in 2^-44 s fixed
// point).  A per-model solve then forms the chosen regressors (the paper's four,
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

// A 128-bit unsigned sum kept as (lo, hi) 64-bit halves.
struct U128 {
    unsigned long long lo, hi;
};
__device__ __forceinline__ void add128(U128 &a, unsigned long long lo, unsigned long long hi) {
    const unsigned long long s = a.lo + lo;
    a.hi += hi + (s < lo ? 1ull : 0ull);
    a.lo = s;
}
// Atomic version: the carry of this addition into the low word follows from the old
// value the atomic returns, so the pair is right once every addition has landed.
__device__ __forceinline__ void atomic_add128(unsigned long long *lo_p, unsigned long long *hi_p,
                                              unsigned long long lo, unsigned long long hi) {
    if (lo == 0ull && hi == 0ull) return;
    const unsigned long long old = atomicAdd(lo_p, lo);
    const unsigned long long c = (old + lo < old) ? 1ull : 0ull;
    if (hi + c != 0ull) atomicAdd(hi_p, hi + c);
}

__device__ __forceinline__ bool mbar_wait(uint32_t mbar, uint32_t parity) {
    for (int it = 0; it < (1 << 22); ++it) {
        uint32_t done;
        asm volatile(
            "{\n .reg .pred P;\n mbarrier.try_wait.parity.shared::cta.b64 P, [%1], %2;\n selp.u32 %0, 1, 0, P;\n}"
            : "=r"(done)
            : "r"(mbar), "r"(parity)
            : "memory");
        if (done) return true;
    }
    return false;
}

// Exact integer sums: features below 2^32 make every product of two of them exact
// in 64 bits, and a time below 2^19 s becomes a 2^-44 s fixed-point integer below
// 2^63, so that feature x time fits 96 bits.  Nothing here uses the (slow) fp64 pipe
// but the time scaling.  Rows grouped by model are the common case (per-instance
// logs): each CTA takes a contiguous slice of the log and each thread keeps the sums
// of the model it is reading in registers, flushing them to shared memory only when
// the model changes.  One CTA per SM: the register sums take most of the register file.
//
// TMA: the slice streams through a ring of kCalStages shared-memory tiles of
// kCalTile rows (features, times, model ids), each filled by bulk copies that
// complete on its mbarrier, which keeps enough bytes in flight to reach HBM rates
// with eight warps per SM.  Without it (inputs not 16-byte aligned) and for the
// slice's last partial tile, rows are read directly.
template <bool TMA>
__global__ void __launch_bounds__(256) k_calib_accum(long long N, const long long *F, const int32_t *model,
                                                     const double *time, int M, unsigned long long *acc, DevCtl *ctl) {
    extern __shared__ __align__(16) unsigned char cal_smem[];
    // Shared sums [copies][M][kCalAcc][2] (lo, hi): one copy per warp when the models
    // are few, so that a flush contends with its own warp only, not the whole CTA.
    const int copies = cal_copies(M);
    unsigned long long *sall = reinterpret_cast<unsigned long long *>(cal_smem);
    unsigned long long *sacc = sall + (size_t)(copies > 1 ? (threadIdx.x >> 5) : 0) * M * kCalAcc * 2;
    unsigned char *stages = cal_smem + cal_sums_bytes(M);
    __shared__ __align__(8) unsigned long long s_mbar[kCalStages];
    for (int i = threadIdx.x; i < copies * M * kCalAcc * 2; i += blockDim.x) sall[i] = 0ull;
    // Exact sums in two levels.  Rows whose features are below 2^26 (and times below
    // 2^8 s) have products below 2^52, and feature x time splits into 32-bit limbs of
    // the time with products below 2^58: those add into plain 64-bit sums, one
    // multiply-add each, settled into the 128-bit totals every 32 rows, before any
    // of them can overflow.  Other rows add to the 128-bit totals directly.
    U128 r[kCalAcc];                     // settled totals: G (15), b (5, 2^-44 s), count
    unsigned long long fg[15], fbl[5], fbh[5];  // 64-bit sums since the last settle
    int nfast = 0;
#pragma unroll
    for (int k = 0; k < kCalAcc; ++k) r[k] = U128{0ull, 0ull};
#pragma unroll
    for (int k = 0; k < 15; ++k) fg[k] = 0ull;
#pragma unroll
    for (int k = 0; k < 5; ++k) fbl[k] = fbh[k] = 0ull;
    int cur = -1;
    bool bad = false;
    auto settle = [&]() {
#pragma unroll
        for (int k = 0; k < 15; ++k) {
            add128(r[k], fg[k], 0ull);
            fg[k] = 0ull;
        }
#pragma unroll
        for (int a = 0; a < 5; ++a) {
            add128(r[15 + a], fbl[a], 0ull);
            add128(r[15 + a], fbh[a] << 32, fbh[a] >> 32);
            fbl[a] = fbh[a] = 0ull;
        }
        add128(r[20], (unsigned long long)nfast, 0ull);
        nfast = 0;
    };
    auto flush = [&]() {
        settle();
        if (cur >= 0)
#pragma unroll
            for (int k = 0; k < kCalAcc; ++k)
                atomic_add128(&sacc[(cur * kCalAcc + k) * 2], &sacc[(cur * kCalAcc + k) * 2 + 1], r[k].lo, r[k].hi);
#pragma unroll
        for (int k = 0; k < kCalAcc; ++k) r[k] = U128{0ull, 0ull};
    };
    auto row = [&](int m, double t, const long long *f) {
        long long v[kCalCols];
        long long any = 0;
#pragma unroll
        for (int k = 0; k < kCalCols; ++k) {
            v[k] = f[k];
            any |= v[k];
        }
        // every feature in [0, 2^32): no bit of any of them at 2^32 or above (nor the sign)
        if (!(m >= 0 && m < M && t >= 0.0 && t < kCalTimeMax) || (any >> 32) != 0) {  // also a NaN time
            bad = true;
            return;
        }
        if (m != cur) {
            flush();
            cur = m;
        }
        const unsigned long long tf = __double2ull_rn(t * kCalTimeScale);
        const uint32_t tlo = (uint32_t)tf, thi = (uint32_t)(tf >> 32);
        uint32_t xs[kCalCols];
#pragma unroll
        for (int k = 0; k < kCalCols; ++k) xs[k] = (uint32_t)v[k];
        if ((any >> 26) == 0 && thi < (1u << 20)) {
#pragma unroll
            for (int a = 0; a < kCalCols; ++a) {
#pragma unroll
                for (int b = a; b < kCalCols; ++b) fg[tri(a, b)] += (unsigned long long)xs[a] * xs[b];
                fbl[a] += (unsigned long long)xs[a] * tlo;
                fbh[a] += (unsigned long long)xs[a] * thi;
            }
            if (++nfast == 32) settle();
            return;
        }
#pragma unroll
        for (int a = 0; a < kCalCols; ++a) {
#pragma unroll
            for (int b = a; b < kCalCols; ++b) add128(r[tri(a, b)], (unsigned long long)xs[a] * xs[b], 0ull);
            // x * t = x * t_lo + (x * t_hi) * 2^32, below 2^96
            const unsigned long long p0 = (unsigned long long)xs[a] * tlo;
            const unsigned long long p1 = (unsigned long long)xs[a] * thi;
            add128(r[15 + a], p0, 0ull);
            add128(r[15 + a], p1 << 32, p1 >> 32);
        }
        add128(r[20], 1ull, 0ull);
    };
    // this CTA's contiguous slice, starting on a tile boundary
    const long long per = ((N + gridDim.x - 1) / gridDim.x + kCalTile - 1) / kCalTile * kCalTile;
    const long long c0 = (long long)blockIdx.x * per, c1 = min(N, c0 + per);
    long long rest = c0;
    bool ok = true;
    if (TMA && c0 < c1) {
        const int ntiles = (int)((c1 - c0) / kCalTile);
        constexpr uint32_t kFeat = kCalTile * kCalCols * 8, kTime = kCalTile * 8, kModel = kCalTile * 4;
        constexpr uint32_t kStage = kFeat + kTime + kModel;
        auto issue = [&](int k) {
            const int st = k % kCalStages;
            const long long r0 = c0 + (long long)k * kCalTile;
            const uint32_t mb = (uint32_t)__cvta_generic_to_shared(&s_mbar[st]);
            const uint32_t dst = (uint32_t)__cvta_generic_to_shared(stages + (size_t)st * kStage);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(mb), "r"(kStage) : "memory");
            asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                             dst),
                         "l"(F + r0 * kCalCols), "r"(kFeat), "r"(mb)
                         : "memory");
            asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                             dst + kFeat),
                         "l"(time + r0), "r"(kTime), "r"(mb)
                         : "memory");
            asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                             dst + kFeat + kTime),
                         "l"(model + r0), "r"(kModel), "r"(mb)
                         : "memory");
        };
        if (threadIdx.x == 0) {
            for (int st = 0; st < kCalStages; ++st) {
                const uint32_t mb = (uint32_t)__cvta_generic_to_shared(&s_mbar[st]);
                asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mb) : "memory");
            }
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        __syncthreads();
        int issued = min(ntiles, kCalStages);
        if (threadIdx.x == 0)
            for (int k = 0; k < issued; ++k) issue(k);
        int k = 0;
        for (; k < ntiles && ok; ++k) {
            const int st = k % kCalStages;
            const bool landed =
                mbar_wait((uint32_t)__cvta_generic_to_shared(&s_mbar[st]), (uint32_t)((k / kCalStages) & 1));
            if (__syncthreads_or(!landed)) {  // a copy that never lands is reported, not waited out
                ok = false;
                break;
            }
            const unsigned char *sb = stages + (size_t)st * kStage;
            const long long *sf = reinterpret_cast<const long long *>(sb);
            const double *stt = reinterpret_cast<const double *>(sb + kFeat);
            const int32_t *sm = reinterpret_cast<const int32_t *>(sb + kFeat + kTime);
            for (int j = threadIdx.x; j < kCalTile; j += blockDim.x) row(sm[j], stt[j], sf + j * kCalCols);
            __syncthreads();  // the stage is free again
            if (k + kCalStages < ntiles) {
                if (threadIdx.x == 0) issue(k + kCalStages);
                issued = k + kCalStages + 1;
            }
        }
        if (!ok && threadIdx.x == 0)  // let the copies still in flight land (bounded) before leaving
            for (int q = k; q < issued; ++q)
                mbar_wait((uint32_t)__cvta_generic_to_shared(&s_mbar[q % kCalStages]),
                          (uint32_t)((q / kCalStages) & 1));
        rest = c0 + (long long)ntiles * kCalTile;
    }
    __syncthreads();
    if (!ok) {
        if (threadIdx.x == 0) record_status(ctl, kECuda);
        return;
    }
    for (long long i = rest + threadIdx.x; i < c1; i += blockDim.x) row(model[i], time[i], F + i * kCalCols);
    // Final flush, warp-synchronous.  When the whole warp holds the same model (the
    // usual case), each 128-bit sum is added across the warp as eight 16-bit limbs
    // with redux.sync (each limb total stays below 2^21) and one lane adds the
    // warp's total; otherwise every lane adds its own.
    settle();
    const int lead = __shfl_sync(kFull, cur, 0);
    if (__all_sync(kFull, cur == lead) && lead >= 0) {
        const int lane = threadIdx.x & 31;
#pragma unroll 1
        for (int k = 0; k < kCalAcc; ++k) {
            U128 tot{0ull, 0ull};
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                const unsigned long long word = q < 4 ? r[k].lo : r[k].hi;
                const unsigned limb = (unsigned)(word >> (16 * (q & 3))) & 0xffffu;
                const unsigned long long sum = __reduce_add_sync(kFull, limb);
                const int sh = 16 * q;  // place sum * 2^sh into 128 bits
                if (sh < 64) add128(tot, sum << sh, sh == 0 ? 0ull : (sum >> (64 - sh)));
                else add128(tot, 0ull, sum << (sh - 64));
            }
            if (lane == 0) atomic_add128(&sacc[(lead * kCalAcc + k) * 2], &sacc[(lead * kCalAcc + k) * 2 + 1], tot.lo, tot.hi);
        }
#pragma unroll
        for (int k = 0; k < kCalAcc; ++k) r[k] = U128{0ull, 0ull};
    } else {
        flush();
    }
    if (__any_sync(kFull, bad) && (threadIdx.x & 31) == 0) record_status(ctl, kEInval);
    __syncthreads();
    for (int i = threadIdx.x; i < M * kCalAcc; i += blockDim.x) {
        U128 sum{0ull, 0ull};
        for (int w = 0; w < copies; ++w) {
            const unsigned long long *c = sall + (size_t)w * M * kCalAcc * 2;
            add128(sum, c[2 * i], c[2 * i + 1]);
        }
        atomic_add128(&acc[2 * i], &acc[2 * i + 1], sum.lo, sum.hi);
    }
}

__device__ __forceinline__ double to_double(const unsigned long long *p) {
    return __fma_rn((double)p[1], 18446744073709551616.0, (double)p[0]);
}

// One thread per model: regressors, power-of-two Jacobi scaling, Cholesky, unscaling.
// D regressors: 4 (the paper's form, F1 + F2 as one token count) or 5; every loop
// is unrolled so that the small matrices stay in registers.
template <int D>
__global__ void k_calib_solve(int M, const unsigned long long *acc, double *coef) {
    const int m = blockIdx.x * blockDim.x + threadIdx.x;
    if (m >= M) return;
    double s[kCalAcc];  // the model's sums, b in seconds
#pragma unroll
    for (int k = 0; k < kCalAcc; ++k) s[k] = to_double(acc + 2 * ((size_t)m * kCalAcc + k));
#pragma unroll
    for (int a = 0; a < kCalCols; ++a) s[15 + a] *= 1.0 / kCalTimeScale;
    // regressor p sums features lo(p) .. hi(p)
    auto lo = [](int p) { return D == 4 ? (p == 0 ? 0 : p == 1 ? 1 : p + 1) : p; };
    auto hi = [](int p) { return D == 4 ? (p == 0 ? 0 : p == 1 ? 2 : p + 1) : p; };
    double G[D][D], b[D], sc[D], L[D][D], z[D], w[D];
#pragma unroll
    for (int p = 0; p < D; ++p) {
        b[p] = 0.0;
#pragma unroll
        for (int a = lo(p); a <= hi(p); ++a) b[p] += s[15 + a];
#pragma unroll
        for (int q = 0; q < D; ++q) {
            double g = 0.0;
#pragma unroll
            for (int a = lo(p); a <= hi(p); ++a)
#pragma unroll
                for (int c = lo(q); c <= hi(q); ++c) g += s[tri(a, c)];
            G[p][q] = g;
        }
    }
    bool ok = s[20] >= (double)D;
#pragma unroll
    for (int p = 0; p < D; ++p) {  // scale regressor p by 2^-e with 2^e ~ sqrt(G_pp)
        ok = ok && G[p][p] > 0.0;
        int e = 0;
        frexp(sqrt(fmax(G[p][p], 1e-300)), &e);
        sc[p] = ldexp(1.0, -e);
    }
#pragma unroll
    for (int p = 0; p < D; ++p)
#pragma unroll
        for (int q = 0; q <= p; ++q) {
            double v = G[p][q] * sc[p] * sc[q];
#pragma unroll
            for (int k = 0; k < q; ++k) v -= L[p][k] * L[q][k];
            if (p == q) {
                ok = ok && v > 1e-13;  // rank-deficient design
                L[p][p] = sqrt(fmax(v, 1e-300));
            } else {
                L[p][q] = v / L[q][q];
            }
        }
#pragma unroll
    for (int p = 0; p < D; ++p) {
        double v = b[p] * sc[p];
#pragma unroll
        for (int k = 0; k < p; ++k) v -= L[p][k] * z[k];
        z[p] = v / L[p][p];
    }
#pragma unroll
    for (int p = D - 1; p >= 0; --p) {
        double v = z[p];
#pragma unroll
        for (int k = p + 1; k < D; ++k) v -= L[k][p] * w[k];
        w[p] = v / L[p][p];
    }
    double out[5];
    if (D == 4) {
        out[0] = w[0] * sc[0];
        out[1] = out[2] = w[1] * sc[1];
        out[3] = w[2] * sc[2];
        out[4] = w[3 % D] * sc[3 % D];
    } else {
#pragma unroll
        for (int p = 0; p < 5; ++p) out[p] = w[p % D] * sc[p % D];
    }
    const double nan = __longlong_as_double(0x7ff8000000000000LL);
#pragma unroll
    for (int p = 0; p < 5; ++p) coef[(size_t)m * 5 + p] = ok ? out[p] : nan;
}

}  // namespace

cudaError_t launch_calibrate(long long N, const long long *F, const int32_t *model, const double *time, int M,
                             int shared_beta1, unsigned long long *acc, double *coef, DevCtl *ctl, int grid,
                             cudaStream_t st) {
    cudaError_t e = cudaMemsetAsync(acc, 0, sizeof(unsigned long long) * 2 * (size_t)M * kCalAcc, st);
    if (e != cudaSuccess) return e;
    if (N > 0) {
        const size_t sums = cal_sums_bytes(M);
        const bool tma = ((uintptr_t)F | (uintptr_t)model | (uintptr_t)time) % 16 == 0;
        if (tma) k_calib_accum<true><<<grid, 256, sums + kCalStageBytes * kCalStages, st>>>(N, F, model, time, M, acc, ctl);
        else k_calib_accum<false><<<grid, 256, sums, st>>>(N, F, model, time, M, acc, ctl);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    if (shared_beta1) k_calib_solve<4><<<(M + 63) / 64, 64, 0, st>>>(M, acc, coef);
    else k_calib_solve<5><<<(M + 63) / 64, 64, 0, st>>>(M, acc, coef);
    return cudaGetLastError();
}

cudaError_t set_calib_smem(int M) {
    const size_t sums = cal_sums_bytes(M);
    cudaError_t e = cudaFuncSetAttribute(k_calib_accum<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)(sums + kCalStageBytes * kCalStages));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_calib_accum<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)sums);
    return e;
}

}  // namespace lr
