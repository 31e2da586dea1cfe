// Least-squares calibration of the Eq. 9 batch-time coefficients per model from a
// log of executed token batches (Sec. 4.1: the coefficients are calibrated from
// observed token-batch processing times).
//
// One kernel, one pass over the log: per model the normal equations G = sum x x^T,
// b = sum x t and the row count, as exact 128-bit integers (times in 2^-44 s fixed
// point); the last CTA to finish then solves every model's system (the paper's four
// regressors, with F1 + F2 as the token count, or the five features), scaled by
// powers of two so that its diagonal is near 1 (exact, and it restores the
// conditioning the raw feature magnitudes take away), by an LDL^T factorization,
// and clears the sums for the next call.
#include "lr_internal.cuh"

#include <algorithm>

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;

// Packed upper triangle of a 5x5 symmetric matrix.
__device__ __forceinline__ int tri(int a, int b) {
    const int lo = a < b ? a : b, hi = a < b ? b : a;
    return lo * kCalCols - lo * (lo - 1) / 2 + (hi - lo);
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
__device__ __forceinline__ void atomic_add128(unsigned long long *p, unsigned long long lo, unsigned long long hi) {
    if (lo == 0ull && hi == 0ull) return;
    const unsigned long long old = atomicAdd(p, lo);
    const unsigned long long c = (old + lo < old) ? 1ull : 0ull;
    if (hi + c != 0ull) atomicAdd(p + 1, hi + c);
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

constexpr unsigned long long kTimeMaxBits = 0x4120000000000000ull;  // the bits of 2^19 (kCalTimeMax)

// floor(t * 2^44) for 0 <= t < 2^19 given the bits of t: the IEEE-754 value of t is
// m * 2^(E - 1075) with the 53-bit significand m, so the product is m shifted left by
// E - 1031 bits, or right (dropping what lies below 2^-44 s) when that is negative.
// Integer operations only.
__device__ __forceinline__ unsigned long long fixed_time(unsigned long long bits) {
    const int E = (int)(bits >> 52);
    const unsigned long long m = (bits & ((1ull << 52) - 1)) | (E != 0 ? (1ull << 52) : 0ull);
    const int sh = max(E, 1) - 1031;
    return sh >= 0 ? m << sh : m >> min(-sh, 63);  // sh <= 10 below 2^19 s
}

// acc += a * b with the 64-bit product of two 32-bit factors, one instruction
__device__ __forceinline__ void mad64(unsigned long long &acc, uint32_t a, uint32_t b) {
    asm("mad.wide.u32 %0, %1, %2, %0;" : "+l"(acc) : "r"(a), "r"(b));
}

// v * 2^e2 as the nearest double (ties to even) for a 128-bit unsigned v, assuming the
// result is a normal number: the leading bit gives the exponent, the next 52 bits the
// fraction, and the bits below round it.  Integer operations only.
__device__ __forceinline__ double u128_to_double(const U128 &v, int e2) {
    if ((v.lo | v.hi) == 0ull) return 0.0;
    const int p = v.hi ? 127 - __clzll((long long)v.hi) : 63 - __clzll((long long)v.lo);  // leading bit
    unsigned long long q;
    int e = p;
    if (p <= 52) {
        q = v.lo << (52 - p);
    } else {
        const int s = p - 52;  // 1 .. 75 bits dropped
        q = s < 64 ? (v.lo >> s) | (s > 0 ? v.hi << (64 - s) : 0ull) : v.hi >> (s - 64);
        const int h = s - 1;   // the highest dropped bit
        const unsigned long long half = h < 64 ? (v.lo >> h) & 1ull : (v.hi >> (h - 64)) & 1ull;
        const bool sticky = h < 64 ? (v.lo & ((1ull << h) - 1ull)) != 0ull
                                   : (v.lo != 0ull || (v.hi & ((1ull << (h - 64)) - 1ull)) != 0ull);
        q += (half && (sticky || (q & 1ull))) ? 1ull : 0ull;
        if (q >> 53) {
            q >>= 1;
            ++e;
        }
    }
    return __longlong_as_double((long long)(((unsigned long long)(e + e2 + 1023) << 52) | (q & ((1ull << 52) - 1))));
}

// The solve of every model's system, on the last CTA: regressors, power-of-two Jacobi
// scaling, LDL^T, unscaling.  D regressors: 4 (the paper's form, F1 + F2 as one token
// count) or 5; with four, a unit fifth regressor uncoupled from the others keeps one
// code path (its weight is 0).  The regressor sums are formed exactly in 128 bits; each
// enters fp64 once, already scaled by the powers of two that bring the diagonal into
// [1, 4) (regressor p scaled by 2^-h_p with h_p half the leading-bit position of G_pp),
// so the conditioning that the raw feature magnitudes take away is restored without a
// rounding.  The code runs once per call from cold instruction caches, and the fp64
// pipe is narrow on this part: the 20 scaled entries of every model are formed by one
// thread each (integer pipes only), then one thread per model factors its system with
// straight-line code in registers, whose only fp64 divisions are the pivot reciprocals.
constexpr int kCalSolveWords = 24;  // per model in shared memory: 15 + 5 scaled entries, 5 exponents

__device__ __forceinline__ void calib_lohi(bool four, int p, int &lo, int &hi) {  // regressor p: features lo..hi
    lo = four ? (p == 0 ? 0 : p == 1 ? 1 : p + 1) : p;
    hi = four ? (p == 0 ? 0 : p == 1 ? 2 : p + 1) : p;
}

// G_pq (b_p when q < 0) of model m from its exact sums S [kCalAcc] (U128 pairs)
__device__ U128 calib_gsum(const unsigned long long *S, bool four, int p, int q) {
    U128 g{0ull, 0ull};
    if (four && p == 4) {  // the unit regressor
        if (q == 4) g.lo = 1ull;
        return g;
    }
    int pl, ph, ql, qh;
    calib_lohi(four, p, pl, ph);
    if (q < 0) {
        for (int a = pl; a <= ph; ++a) add128(g, S[2 * (15 + a)], S[2 * (15 + a) + 1]);
        return g;
    }
    if (four && q == 4) return g;
    calib_lohi(four, q, ql, qh);
    for (int a = pl; a <= ph; ++a)
        for (int c = ql; c <= qh; ++c) add128(g, S[2 * tri(a, c)], S[2 * tri(a, c) + 1]);
    return g;
}

__device__ __forceinline__ int half_lead(const U128 &g) {
    const int e = g.hi ? 127 - __clzll((long long)g.hi) : (g.lo ? 63 - __clzll((long long)g.lo) : 0);
    return e >> 1;
}

// entry e of model m: e < 15 the packed lower triangle of A (row p, column q <= p), else b
__device__ void calib_entry(int m, int e, bool four, const unsigned long long *S, double *W) {
    const unsigned long long *Sm = S + (size_t)m * kCalAcc * 2;
    double *Wm = W + (size_t)m * kCalSolveWords;
    int p = e - 15, q = -1;
    if (e < 15) {
        p = 0;
        while ((p + 1) * (p + 2) / 2 <= e) ++p;
        q = e - p * (p + 1) / 2;
    }
    const int *h = reinterpret_cast<const int *>(Wm + 20);
    Wm[e] = u128_to_double(calib_gsum(Sm, four, p, q), -(h[p] + (q < 0 ? 44 : h[q])));  // b carries 2^-44 s
}

// the scale exponent h_p of regressor p of model m (before the entries)
__device__ void calib_scale(int m, int p, bool four, const unsigned long long *S, double *W) {
    reinterpret_cast<int *>(W + (size_t)m * kCalSolveWords + 20)[p] =
        half_lead(calib_gsum(S + (size_t)m * kCalAcc * 2, four, p, p));
}

// On this part the SM's fp64 unit is narrow: each fp64 instruction of a warp costs
// tens of cycles whatever the active lanes, so the solve keeps its fp64 instructions
// few and does comparisons, clamps and power-of-two scalings on the bits.

// 1/x for a positive normal double: the fp32 reciprocal of its significand truncated to
// 24 bits (built from the bits, relative error below 2^-23), rescaled by the exponent,
// then one Newton-Raphson step r <- r (2 - x r), which squares the error (2^-46).
__device__ __forceinline__ double recip_pos(double x) {
    const unsigned long long bx = (unsigned long long)__double_as_longlong(x);
    const long long e = (long long)((bx >> 52) & 0x7ff) - 1023;
    const float m = __int_as_float((int)((127u << 23) | (unsigned)((bx >> 29) & 0x7fffffu)));  // [1, 2)
    const unsigned rb = (unsigned)__float_as_int(__frcp_rn(m));                                  // (1/2, 1]
    const long long re = (long long)((rb >> 23) & 0xff) - 127 - e;
    const double r = __longlong_as_double((long long)(((unsigned long long)(re + 1023) << 52) |
                                                      ((unsigned long long)(rb & 0x7fffffu) << 29)));
    return __fma_rn(r, __fma_rn(-x, r, 1.0), r);
}

// v * 2^-h for a finite v (0 stays 0; the results here stay normal): the exponent field
__device__ __forceinline__ double scale_pow2(double v, int h) {
    const long long bv = __double_as_longlong(v);
    return (bv & 0x7ff0000000000000LL) ? __longlong_as_double(bv - ((long long)h << 52)) : v;
}

// The scaled 5x5 system of model m by LDL^T, with straight-line code in registers.
__device__ void calib_factor(int m, int D, const unsigned long long *S, const double *W, double *coef) {
    const double *Wm = W + (size_t)m * kCalSolveWords;
    const int *h = reinterpret_cast<const int *>(Wm + 20);
    const unsigned long long *cnt = S + ((size_t)m * kCalAcc + 20) * 2;
    bool ok = cnt[1] != 0ull || cnt[0] >= (unsigned long long)D;
    double A[5][5], b[5], LD[5][5], L[5][5], inv[5], y[5], w[5];
#pragma unroll
    for (int p = 0; p < 5; ++p) {
        b[p] = Wm[15 + p];
#pragma unroll
        for (int q = 0; q <= p; ++q) A[p][q] = Wm[p * (p + 1) / 2 + q];
    }
    constexpr long long kMinPivot = 0x3d3c25c268497682LL;  // the bits of 1e-13
#pragma unroll
    for (int p = 0; p < 5; ++p) {
#pragma unroll
        for (int q = 0; q < p; ++q) {
            double v = A[p][q];
#pragma unroll
            for (int k = 0; k < q; ++k) v = __fma_rn(-LD[p][k], L[q][k], v);
            LD[p][q] = v;  // L[p][q] d[q]
            L[p][q] = v * inv[q];
        }
        double v = A[p][p];
#pragma unroll
        for (int k = 0; k < p; ++k) v = __fma_rn(-LD[p][k], L[p][k], v);
        // v > 1e-13 on the bits (a positive double orders as its bits; NaN fails)
        const long long bv = __double_as_longlong(v);
        const bool piv = bv > kMinPivot && bv < 0x7ff0000000000000LL;
        ok = ok && piv;  // rank-deficient design (or a zero G_pp)
        inv[p] = piv ? recip_pos(v) : 0.0;
    }
#pragma unroll
    for (int p = 0; p < 5; ++p) {
        double v = b[p];
#pragma unroll
        for (int k = 0; k < p; ++k) v = __fma_rn(-L[p][k], y[k], v);
        y[p] = v;
    }
#pragma unroll
    for (int p = 4; p >= 0; --p) {
        double v = y[p] * inv[p];
#pragma unroll
        for (int k = p + 1; k < 5; ++k) v = __fma_rn(-L[k][p], w[k], v);
        w[p] = v;
    }
    // the five coefficients, unscaled by 2^-h_p: with four regressors the token slope
    // serves prefill and decode
    const double nan = __longlong_as_double(0x7ff8000000000000LL);
    const bool four = D == 4;
    double out[5];
    out[0] = scale_pow2(w[0], h[0]);
    out[1] = scale_pow2(w[1], h[1]);
    out[2] = four ? out[1] : scale_pow2(w[2], h[2]);
    out[3] = four ? scale_pow2(w[2], h[2]) : scale_pow2(w[3], h[3]);
    out[4] = four ? scale_pow2(w[3], h[3]) : scale_pow2(w[4], h[4]);
#pragma unroll
    for (int k = 0; k < 5; ++k) coef[(size_t)m * 5 + k] = ok ? out[k] : nan;
}

// The pass over the log.  Exact integer sums: features below 2^32 make every product
// of two of them exact in 64 bits, and a time below 2^19 s becomes a 2^-44 s fixed-
// point integer below 2^63, so that feature x time fits 96 bits.  Rows whose features
// are below 2^26 and whose time is below 2^8 s (the usual case) add their 15 products,
// and the products of each feature with the two 26-bit halves of the time, into plain
// 64-bit sums in registers: every product is below 2^52, so a lane's sums of up to 128
// rows stay below 2^59 and a warp's below 2^64.  The warp flushes them into the
// 128-bit sums in shared memory when a lane's model changes (rows grouped by model are
// the usual case), before 128 rows and at the end: a reduce-scatter over the 32 lanes
// (five rounds of exchanging half of the remaining values with the partner lane) leaves
// lane k with the warp total of sum k, which it adds to the model's shared sum -- one
// shared atomic per sum, model and warp.  The warp decides together whether to flush:
// one vote per tile of two rows a lane, one per row around a model change.  Other rows
// add to the shared 128-bit sums directly.  Nothing uses the fp64 pipe.
//
// TMA: each CTA streams a contiguous slice of the log through a ring of `nst`
// shared-memory tiles of kCalTile rows (features, times, model ids), each filled by
// bulk copies that complete on its mbarrier.  Without it (inputs not 16-byte aligned)
// and for the slice's last partial tile, rows are read directly.
template <bool TMA>
__global__ void __launch_bounds__(kCalThreads, 1) k_calibrate(long long N, const long long *F, const int32_t *model,
                                                              const double *time, int M, int D, int nst,
                                                              unsigned long long *acc, double *coef, DevCtl *ctl) {
    extern __shared__ __align__(16) unsigned char cal_smem[];
    unsigned long long *sacc = reinterpret_cast<unsigned long long *>(cal_smem);  // [M][kCalAcc][2] (lo, hi)
    // the flushes' totals in carry-save form: [M][26][2], sum k = w0 + 2^32 w1, each flush
    // adding the low and the high 32 bits of its (below 2^64) total with a reduction that
    // returns nothing (no carry to wait for)
    unsigned long long *scs = sacc + (size_t)M * kCalAcc * 2;
    const int lane = threadIdx.x & 31;
    unsigned char *stages = cal_smem + cal_sums_bytes(M);
    __shared__ __align__(8) unsigned long long s_mbar[kCalStagesMax];
    __shared__ int s_last;
    unsigned int *done = reinterpret_cast<unsigned int *>(acc + 2 * (size_t)M * kCalAcc);
    for (int i = threadIdx.x; i < M * (kCalAcc + kCalFlushSums) * 2; i += blockDim.x) sacc[i] = 0ull;
    unsigned long long g[15], bl[5], bh[5];  // 64-bit sums since the last flush
    int nfast = 0, cur = -1;
    bool bad = false;
#pragma unroll
    for (int k = 0; k < 15; ++k) g[k] = 0ull;
#pragma unroll
    for (int q = 0; q < 5; ++q) bl[q] = bh[q] = 0ull;
    auto flush = [&]() {  // every lane of the warp calls it
        const int key = nfast > 0 ? cur : -1;
        unsigned pend = __ballot_sync(kFull, key >= 0);
        while (pend) {
            const int mk = __shfl_sync(kFull, key, __ffs(pend) - 1);
            const bool mine = key == mk;
            // sums 0..14: G; 15..19: x t_lo halves of b; 20..24: x t_hi halves (weight
            // 2^26); 25: the row count
            unsigned long long a[32];
#pragma unroll
            for (int k = 0; k < 15; ++k) a[k] = mine ? g[k] : 0ull;
#pragma unroll
            for (int q = 0; q < 5; ++q) {
                a[15 + q] = mine ? bl[q] : 0ull;
                a[20 + q] = mine ? bh[q] : 0ull;
            }
            a[25] = mine ? (unsigned long long)nfast : 0ull;
#pragma unroll
            for (int k = 26; k < 32; ++k) a[k] = 0ull;
#pragma unroll
            for (int w = 16; w >= 1; w >>= 1) {  // keep the half of a[0..2w) that this lane's bit w selects
                const bool up = (lane & w) != 0;
#pragma unroll
                for (int j = 0; j < w; ++j) {
                    const unsigned long long give = up ? a[j] : a[j + w];
                    a[j] = (up ? a[j + w] : a[j]) + __shfl_xor_sync(kFull, give, w);
                }
            }
            if (lane < kCalFlushSums) {  // a[0]: the warp's total of sum `lane`
                const uint32_t sa = (uint32_t)__cvta_generic_to_shared(scs + ((size_t)mk * kCalFlushSums + lane) * 2);
                asm volatile("red.shared.add.u64 [%0], %1;" ::"r"(sa), "l"(a[0] & 0xffffffffull) : "memory");
                asm volatile("red.shared.add.u64 [%0], %1;" ::"r"(sa + 8u), "l"(a[0] >> 32) : "memory");
            }
            pend &= ~__ballot_sync(kFull, mine);
        }
#pragma unroll
        for (int k = 0; k < 15; ++k) g[k] = 0ull;
#pragma unroll
        for (int q = 0; q < 5; ++q) bl[q] = bh[q] = 0ull;
        nfast = 0;
    };
    // One row per lane, the whole warp together (`in` false: no row).  With `vote` the
    // warp first flushes if a lane's model changes or its sums reach 128 rows; without
    // it the caller has made sure that neither happens.
    auto row = [&](bool in, bool vote, int m, double t, const long long *f) {
        long long v[kCalCols];
        long long any = 0;
        unsigned long long tb = 0ull;
        if (in) {
#pragma unroll
            for (int k = 0; k < kCalCols; ++k) {
                v[k] = f[k];
                any |= v[k];
            }
            tb = (unsigned long long)__double_as_longlong(t);
        }
        // 0 <= t < 2^19 on the bits (-0 counts as 0; NaN fails), every feature in
        // [0, 2^32): no bit of any of them at 2^32 or above (nor the sign)
        const unsigned long long tmag = tb & 0x7fffffffffffffffull;
        const bool tok = (tb >> 63) == 0ull ? tb < kTimeMaxBits : tmag == 0ull;
        const bool ok = in && m >= 0 && m < M && tok && (any >> 32) == 0;
        bad |= in && !ok;
        if (vote && __any_sync(kFull, (ok && m != cur) || nfast >= kCalFlushRows)) flush();
        if (!ok) return;
        cur = m;
        const unsigned long long tf = fixed_time(tmag);
        uint32_t x[kCalCols];
#pragma unroll
        for (int k = 0; k < kCalCols; ++k) x[k] = (uint32_t)v[k];
        if ((any >> 26) == 0 && (tf >> 52) == 0ull) {
            const uint32_t tl = (uint32_t)tf & ((1u << 26) - 1), th = (uint32_t)(tf >> 26);
            // Eq. 9's constant feature is 1 (the usual row): its products are additions
            const int q0 = x[0] == 1u ? 1 : 0;
            if (q0) {
                g[tri(0, 0)] += 1ull;
#pragma unroll
                for (int r = 1; r < kCalCols; ++r) g[tri(0, r)] += x[r];
                bl[0] += tl;
                bh[0] += th;
            }
#pragma unroll
            for (int q = 0; q < kCalCols; ++q) {
                if (q == 0 && q0) continue;
#pragma unroll
                for (int r = q; r < kCalCols; ++r) mad64(g[tri(q, r)], x[q], x[r]);
                mad64(bl[q], x[q], tl);
                mad64(bh[q], x[q], th);
            }
            ++nfast;
            return;
        }
        // rows with larger values add exactly into the shared 128-bit sums
        unsigned long long *s = sacc + (size_t)m * kCalAcc * 2;
        const uint32_t tlo = (uint32_t)tf, thi = (uint32_t)(tf >> 32);
#pragma unroll
        for (int q = 0; q < kCalCols; ++q) {
#pragma unroll
            for (int r = q; r < kCalCols; ++r) atomic_add128(s + 2 * tri(q, r), (unsigned long long)x[q] * x[r], 0ull);
            // x * t = x * t_lo + (x * t_hi) * 2^32, below 2^96
            const unsigned long long p1 = (unsigned long long)x[q] * thi;
            U128 w{(unsigned long long)x[q] * tlo, 0ull};
            add128(w, p1 << 32, p1 >> 32);
            atomic_add128(s + 2 * (15 + q), w.lo, w.hi);
        }
        atomic_add128(s + 40, 1ull, 0ull);
    };
    // this CTA's contiguous slice, starting on a tile boundary
    const long long per = ((N + gridDim.x - 1) / gridDim.x + kCalTile - 1) / kCalTile * kCalTile;
    const long long c0 = min(N, (long long)blockIdx.x * per), c1 = min(N, c0 + per);
    long long rest = c0;
    bool ok = true;
    // per stage: `full` completes when its tile has landed, `empty` when every consumer
    // warp has read it
    __shared__ __align__(8) unsigned long long s_empty[kCalStagesMax];
    if (TMA && threadIdx.x == 0) {
        for (int st = 0; st < nst; ++st) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"((uint32_t)__cvta_generic_to_shared(&s_mbar[st]))
                         : "memory");
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(
                             (uint32_t)__cvta_generic_to_shared(&s_empty[st])),
                         "r"(kCalConsumerWarps)
                         : "memory");
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();  // the sums are zero and the barriers ready
    if (TMA && c0 < c1) {
        // The last warp produces (its lane 0 issues each tile once the consumers have
        // released the stage), the others consume at their own pace: no CTA barrier in
        // the loop, so a warp that finishes a tile early starts the next one.
        const int ntiles = (int)((c1 - c0) / kCalTile);
        constexpr uint32_t kFeat = kCalTile * kCalCols * 8, kTime = kCalTile * 8, kModel = kCalTile * 4;
        constexpr uint32_t kStage = kFeat + kTime + kModel;
        const int warp = threadIdx.x >> 5;
        bool failed = false;
        if (warp == kCalConsumerWarps) {
            if (lane == 0) {
                unsigned long long once;
                asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(once));
                int issued = 0;
                for (int k = 0; k < ntiles; ++k) {
                    const int st = k % nst, r = k / nst;
                    if (r > 0 && !mbar_wait((uint32_t)__cvta_generic_to_shared(&s_empty[st]), (uint32_t)((r - 1) & 1))) {
                        failed = true;  // a consumer never released the stage: stop issuing
                        break;
                    }
                    const long long r0 = c0 + (long long)k * kCalTile;
                    const uint32_t mb = (uint32_t)__cvta_generic_to_shared(&s_mbar[st]);
                    const uint32_t dst = (uint32_t)__cvta_generic_to_shared(stages + (size_t)st * kStage);
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(mb), "r"(kStage) : "memory");
                    // the log is read once: first out of L2, ahead of the code and the sums
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, "
                        "[%3], %4;" ::"r"(dst),
                        "l"(F + r0 * kCalCols), "r"(kFeat), "r"(mb), "l"(once)
                        : "memory");
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, "
                        "[%3], %4;" ::"r"(dst + kFeat),
                        "l"(time + r0), "r"(kTime), "r"(mb), "l"(once)
                        : "memory");
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, "
                        "[%3], %4;" ::"r"(dst + kFeat + kTime),
                        "l"(model + r0), "r"(kModel), "r"(mb), "l"(once)
                        : "memory");
                    issued = k + 1;
                }
                // every copy has landed before the CTA moves on: only the last nst issued
                // tiles can still be in flight (bounded waits)
                for (int q = max(0, issued - nst); q < issued; ++q)
                    failed |= !mbar_wait((uint32_t)__cvta_generic_to_shared(&s_mbar[q % nst]), (uint32_t)((q / nst) & 1));
            }
        } else {
            for (int k = 0; k < ntiles; ++k) {
                const int st = k % nst;
                if (!mbar_wait((uint32_t)__cvta_generic_to_shared(&s_mbar[st]), (uint32_t)((k / nst) & 1))) {
                    failed = true;  // never landed: stop (the producer's waits are bounded too)
                    break;
                }
                const unsigned char *sb = stages + (size_t)st * kStage;
                const long long *sf = reinterpret_cast<const long long *>(sb);
                const double *stt = reinterpret_cast<const double *>(sb + kFeat);
                const int32_t *sm = reinterpret_cast<const int32_t *>(sb + kFeat + kTime);
                // two rows a lane; one vote for both unless a model changes or the sums
                // near their limit
                const int j0 = threadIdx.x, j1 = threadIdx.x + kCalConsumerWarps * 32;
                const int m0 = sm[j0], m1 = sm[j1];
                const bool plain = !__any_sync(kFull, m0 != cur || m1 != cur || nfast > kCalFlushRows - 2);
                row(true, !plain, m0, stt[j0], sf + j0 * kCalCols);
                row(true, !plain, m1, stt[j1], sf + j1 * kCalCols);
                __syncwarp();
                if (lane == 0)  // this warp is done with the stage
                    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(
                                     (uint32_t)__cvta_generic_to_shared(&s_empty[st]))
                                 : "memory");
            }
        }
        ok = !__syncthreads_or(failed);
        rest = c0 + (long long)ntiles * kCalTile;
    }
    if (ok)  // the rest row by row, every warp through the same number of steps
        for (long long i0 = rest; i0 < c1; i0 += blockDim.x) {
            const long long i = i0 + threadIdx.x;
            const bool in = i < c1;
            row(in, true, in ? model[i] : 0, in ? time[i] : 0.0, F + (in ? i : 0) * kCalCols);
        }
    flush();
    if (__any_sync(kFull, bad) && lane == 0) record_status(ctl, kEInval);
    if (!ok && threadIdx.x == 0) record_status(ctl, kECuda);
    __syncthreads();
    // each sum: the direct adds plus the flushes' carry-save words (the x t_hi halves of b
    // weigh 2^26)
    for (int i = threadIdx.x; i < M * kCalAcc; i += blockDim.x) {
        const int mm = i / kCalAcc, k = i - mm * kCalAcc;
        U128 v{sacc[2 * i], sacc[2 * i + 1]};
        auto add_cs = [&](int f, int sh) {
            const unsigned long long *w = scs + ((size_t)mm * kCalFlushSums + f) * 2;
            // w0 + 2^32 w1, then shifted left by sh (< 32): below 2^128
            U128 c{w[0], 0ull};
            add128(c, w[1] << 32, w[1] >> 32);
            add128(v, c.lo << sh, sh ? (c.hi << sh) | (c.lo >> (64 - sh)) : c.hi);
        };
        if (k < 15) add_cs(k, 0);
        else if (k < 20) {
            add_cs(k, 0);
            add_cs(k + 5, 26);
        } else add_cs(25, 0);
        atomic_add128(acc + 2 * i, v.lo, v.hi);
    }
    // the last CTA to finish solves every model and clears the sums for the next call
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(done, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    // the totals into the CTA's (now free) shared sums, the scaled entries into the ring
    for (int i = threadIdx.x; i < 2 * M * kCalAcc; i += blockDim.x) sacc[i] = __ldcg(acc + i);
    __syncthreads();
    double *W = reinterpret_cast<double *>(stages);
    for (int i = threadIdx.x; i < 5 * M; i += blockDim.x) calib_scale(i / 5, i % 5, D == 4, sacc, W);
    __syncthreads();
    for (int i = threadIdx.x; i < 20 * M; i += blockDim.x) calib_entry(i / 20, i % 20, D == 4, sacc, W);
    __syncthreads();
    // model m on lane m / 4 of warp m % 4: the four warps sit on the four SM sub-partitions,
    // each with its own fp64 unit
    if (threadIdx.x < 128) {
        const int m = (threadIdx.x & 31) * 4 + (threadIdx.x >> 5);
        if (m < M) calib_factor(m, D, sacc, W, coef);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 2 * M * kCalAcc; i += blockDim.x) acc[i] = 0ull;
    if (threadIdx.x == 0) *done = 0u;
}

}  // namespace

static_assert(kCalMaxModels * (kCalAcc + kCalFlushSums) * 16 + 2 * kCalStageBytes <= kCalSmemMax,
              "two stages at most models");

static_assert((size_t)kCalMaxModels * kCalSolveWords * 8 <= 2 * kCalStageBytes, "the solve's entries fit the ring");
static size_t solve_bytes(int M) { return (size_t)M * kCalSolveWords * 8; }

static int calib_stages(int M) {
    const size_t fixed = cal_sums_bytes(M);
    return (int)std::min<size_t>(kCalStagesMax, (kCalSmemMax - fixed) / kCalStageBytes);
}

cudaError_t launch_calibrate(long long N, const long long *F, const int32_t *model, const double *time, int M,
                             int shared_beta1, unsigned long long *acc, double *coef, DevCtl *ctl, int grid,
                             cudaStream_t st) {
    const int D = shared_beta1 ? 4 : 5;
    const int nst = calib_stages(M);
    const size_t fixed = cal_sums_bytes(M);
    const bool tma = ((uintptr_t)F | (uintptr_t)model | (uintptr_t)time) % 16 == 0;
    if (N <= 0) grid = 1;
    // the ring also holds the solve's scaled entries (kCalSolveWords doubles a model)
    if (tma)
        k_calibrate<true><<<grid, kCalThreads, fixed + kCalStageBytes * nst, st>>>(N, F, model, time, M, D, nst, acc,
                                                                                  coef, ctl);
    else
        k_calibrate<false><<<grid, kCalThreads, fixed + solve_bytes(M), st>>>(N, F, model, time, M, D, nst, acc, coef,
                                                                               ctl);
    return cudaGetLastError();
}

cudaError_t set_calib_smem(int M) {
    const size_t fixed = cal_sums_bytes(M);
    cudaError_t e = cudaFuncSetAttribute(k_calibrate<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)(fixed + kCalStageBytes * calib_stages(M)));
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_calibrate<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(fixed + solve_bytes(M)));
    return e;
}

}  // namespace lr
