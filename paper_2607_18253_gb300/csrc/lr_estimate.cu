// K2: per-candidate SFS TTFT (Sec. 4.1, Eq. 7-9), utility (Eq. 2) and the
// per-query argmax (Eq. 3, Eq. 5).
//
// Each thread owns one instance j of its CTA's instance tile and walks the
// CTA's query rows; the instance's summary (written by K1) sits in shared
// memory, its scalars in registers.  For a query of prompt p:
//
//   k* = #{k : R_k < p}          cumulative budget after the admission batch;
//                                found with one bucket lookup (bucket width
//                                2^shift is below every budget increment, so a
//                                bucket holds at most one boundary)
//   F  = (la + k* + [separate first decode], F1tot + p, F2_k*,
//         F3_k* + [separate first decode] p, F4tot + p(p+1)/2)
//   TTFT = b0 F0 + b1d F2 + b1p F1 + b2 F3 + b3 F4   (fixed fp32 order)
//
// The first two terms depend on k* only and are precomputed as T_k.  The
// int64 -> fp32 roundings of F1, F3 and F4 are done exactly with fp32 adds:
// X + y with X = H + L (H a multiple of 2^20 below 2^44, L < 2^20) rounds as
// fadd(H, fadd(L, y)) because the inner sum is an exact integer below 2^24
// and the outer add rounds the exact total once.  This keeps the hot loop on
// the FMA pipe; instances whose totals reach 2^44 take the int64 path.
//
// The estimate matrix is write-only (4 bytes per candidate) and streamed out
// with evict-first stores; this kernel is bound by HBM bandwidth.
#include <math.h>

#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr long long kLowMask = (1LL << kSplitBits) - 1;

struct __align__(16) QRec {
    int p;     // prompt length, clamped into [1, pmax] for table lookups
    float fp;  // p as fp32, NaN if p was out of range
    float ph;  // p(p+1)/2 high part (multiple of 2^20)
    float pl;  // p(p+1)/2 low part
};

struct InstRegs {
    int jl, la, shift;
    float h1, l1, h4, l4, b1p, b2, b3;
    long long f1tot, f4tot;
};

__device__ __forceinline__ QRec make_qrec(int p, int pmax, bool *ok) {
    QRec q;
    *ok = p >= 1 && p <= pmax;
    if (!*ok) p = 1;
    const long long pp = ((long long)p * (p + 1)) / 2;
    const long long pl = pp & kLowMask;
    q.p = p;
    q.fp = *ok ? (float)p : __int_as_float(0x7fc00000);
    q.ph = __ll2float_rn(pp - pl);
    q.pl = __ll2float_rn(pl);
    return q;
}

__device__ __forceinline__ InstRegs load_inst(const DevConfig &c, const StateBuf &sb, int j, int jl) {
    InstRegs r;
    const InstParams ip = sb.inst[j];
    const int m = c.moi[j];
    r.jl = jl;
    r.la = ip.la;
    r.shift = ip.shift;
    r.h1 = ip.h1;
    r.l1 = ip.l1;
    r.h4 = ip.h4;
    r.l4 = ip.l4;
    r.f1tot = ip.f1tot;
    r.f4tot = ip.f4tot;
    r.b1p = c.coef[m * 5 + 1];
    r.b2 = c.coef[m * 5 + 3];
    r.b3 = c.coef[m * 5 + 4];
    return r;
}

// Index of the query's last prefill batch relative to the admission batch.
__device__ __forceinline__ int locate(const QRec &q, const InstRegs &r, const int2 *s_bkt, int IT) {
    const int2 bk = s_bkt[(q.p >> r.shift) * IT + r.jl];
    return bk.y + (q.p > bk.x ? 1 : 0);
}

template <int MODE>
__device__ __forceinline__ float ttft_fast(const QRec &q, const InstRegs &r, const float4 e) {
    const float f1 = __fadd_rn(r.h1, __fadd_rn(r.l1, q.fp));
    const float f3 = (MODE == 0) ? __fadd_rn(e.y, __fadd_rn(e.z, q.fp)) : e.w;
    const float f4 = __fadd_rn(__fadd_rn(r.h4, q.ph), __fadd_rn(r.l4, q.pl));
    float t = __fmaf_rn(r.b1p, f1, e.x);
    t = __fmaf_rn(r.b2, f3, t);
    t = __fmaf_rn(r.b3, f4, t);
    return t;
}

template <int MODE>
__device__ __forceinline__ float ttft_exact64(const QRec &q, const InstRegs &r, const float4 e, long long f3b) {
    if (q.fp != q.fp) return q.fp;
    const long long p = q.p;
    const float f1 = __ll2float_rn(r.f1tot + p);
    const float f3 = __ll2float_rn(f3b + (MODE == 0 ? p : 0));
    const float f4 = __ll2float_rn(r.f4tot + (p * (p + 1)) / 2);
    float t = __fmaf_rn(r.b1p, f1, e.x);
    t = __fmaf_rn(r.b2, f3, t);
    t = __fmaf_rn(r.b3, f4, t);
    return t;
}

// Stage the summary tables of instances [j0, j0 + IT) into shared memory.
__device__ __forceinline__ void stage_tables(const DevConfig &c, const StateBuf &sb, int j0, int IT,
                                             float4 *s_ent, int2 *s_bkt) {
    for (int idx = threadIdx.x; idx < c.kph * IT; idx += blockDim.x) {
        const int k = idx / IT;
        const int jg = j0 + (idx - k * IT);
        s_ent[idx] = jg < c.I ? sb.ent[(size_t)k * c.I + jg] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    for (int idx = threadIdx.x; idx < c.nbh * IT; idx += blockDim.x) {
        const int b = idx / IT;
        const int jg = j0 + (idx - b * IT);
        s_bkt[idx] = jg < c.I ? sb.bkt[(size_t)b * c.I + jg] : make_int2(kBig, 0);
    }
}

enum : int { kOutTtft = 0, kOutTtftIters = 1, kOutFeatures = 2 };

template <int MODE, int OUT>
__global__ void __launch_bounds__(256) k_estimate(const K2Launch a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const DevConfig &c = a.cfg;
    const int I = c.I, IT = a.IT, QS = a.QS, QT = a.QT;
    const int jl = threadIdx.x % IT;
    const int qs = threadIdx.x / IT;
    const int j = blockIdx.y * IT + jl;
    const bool jv = (qs < QS) && (j < I);
    const int rows_per = (a.Q + gridDim.x - 1) / gridDim.x;
    const int rb = blockIdx.x * rows_per;
    const int re = min(a.Q, rb + rows_per);
    if (rb >= re) return;
    const int active = *((volatile int32_t *)&a.ctl->active);
    if (active < 0) {
        if (threadIdx.x == 0) record_status(a.ctl, kENoState);
        if (jv) {
            for (int rr = rb + qs; rr < re; rr += QS) {
                const size_t o = (size_t)rr * I + j;
                if (OUT == kOutFeatures) {
                    for (int f = 0; f < 5; ++f) a.features[o * 5 + f] = -1;
                } else {
                    a.ttft[o] = __int_as_float(0x7fc00000);
                    if (OUT == kOutTtftIters) a.first_batch[o] = -1;
                }
            }
        }
        return;
    }
    const StateBuf sb = active ? a.buf1 : a.buf0;
    float4 *s_ent = reinterpret_cast<float4 *>(smem);                 // [kph][IT]
    QRec *s_q = reinterpret_cast<QRec *>(s_ent + c.kph * IT);          // [QT]
    int2 *s_bkt = reinterpret_cast<int2 *>(s_q + QT);                  // [nbh][IT]
    stage_tables(c, sb, blockIdx.y * IT, IT, s_ent, s_bkt);
    InstRegs r = {};
    if (jv) r = load_inst(c, sb, j, jl);
    const int fast = __syncthreads_and(!jv || sb.inst[j].fast);
    constexpr int off = (MODE == 0) ? 1 : 0;

    for (int q0 = rb; q0 < re; q0 += QT) {
        const int nrows = min(QT, re - q0);
        if ((int)threadIdx.x < nrows) {
            bool ok;
            s_q[threadIdx.x] = make_qrec(a.prompt[q0 + threadIdx.x], c.pmax, &ok);
            if (!ok && blockIdx.y == 0) record_status(a.ctl, kEInval);
        }
        __syncthreads();
        if (jv) {
            float *out = a.ttft + (size_t)q0 * I + j;
            for (int rr = qs; rr < nrows; rr += QS) {
                const QRec q = s_q[rr];
                const int k = locate(q, r, s_bkt, IT);
                const size_t o = (size_t)rr * I;
                if (OUT == kOutFeatures) {
                    long long *F = a.features + ((size_t)(q0 + rr) * I + j) * 5;
                    if (q.fp != q.fp) {
                        for (int f = 0; f < 5; ++f) F[f] = -1;
                    } else {
                        const long long p = q.p;
                        const size_t e = (size_t)k * I + j;
                        F[0] = r.la + k + off;
                        F[1] = r.f1tot + p;
                        F[2] = sb.f2[e];
                        F[3] = sb.f3[e] + (MODE == 0 ? p : 0);
                        F[4] = r.f4tot + (p * (p + 1)) / 2;
                    }
                } else {
                    const float4 e = s_ent[k * IT + jl];
                    const float t = fast ? ttft_fast<MODE>(q, r, e)
                                         : ttft_exact64<MODE>(q, r, e, sb.f3[(size_t)k * I + j]);
                    __stcs(out + o, t);
                    if (OUT == kOutTtftIters)
                        a.first_batch[(size_t)(q0 + rr) * I + j] = (q.fp != q.fp) ? -1 : r.la + k + off;
                }
            }
        }
        __syncthreads();
    }
}

// Route: phase 1 fills a [rows][instances] tile of TTFT in shared memory (and
// optionally streams it to the estimate matrix); phase 2 scores the tile for
// each (lambda, mu) pair with TPR threads per row and reduces to one instance
// per query, ties to the lowest index.
template <int MODE, bool CONSTRAINED, bool MATRIX>
__global__ void __launch_bounds__(1024) k_route(const K2Launch a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const DevConfig &c = a.cfg;
    const int I = c.I, M = c.M, IT = a.IT, QS = a.QS, QT = a.QT, TPR = a.TPR;
    const int ST = ((I + 31) & ~31) + TPR;  // padded row stride of the TTFT tile
    const int jl = threadIdx.x % IT;
    const int qs = threadIdx.x / IT;
    const int j = jl;
    const bool jv = (qs < QS) && (j < I);
    const int rows_per = (a.Q + gridDim.x - 1) / gridDim.x;
    const int rb = blockIdx.x * rows_per;
    const int re = min(a.Q, rb + rows_per);
    if (rb >= re) return;
    const int active = *((volatile int32_t *)&a.ctl->active);
    if (active < 0) {
        if (threadIdx.x == 0) record_status(a.ctl, kENoState);
        for (int pp = 0; pp < a.P; ++pp)
            for (int i = rb + threadIdx.x; i < re; i += blockDim.x) {
                a.assign[(size_t)pp * a.Q + i] = -1;
                a.util[(size_t)pp * a.Q + i] = __int_as_float(0x7fc00000);
                if (a.ttft_chosen) a.ttft_chosen[(size_t)pp * a.Q + i] = __int_as_float(0x7fc00000);
            }
        if (MATRIX && jv)
            for (int rr = rb + qs; rr < re; rr += QS) a.ttft[(size_t)rr * I + j] = __int_as_float(0x7fc00000);
        return;
    }
    const StateBuf sb = active ? a.buf1 : a.buf0;
    float4 *s_ent = reinterpret_cast<float4 *>(smem);                 // [kph][IT]
    QRec *s_q = reinterpret_cast<QRec *>(s_ent + c.kph * IT);          // [QT]
    int2 *s_bkt = reinterpret_cast<int2 *>(s_q + QT);                  // [nbh][IT]
    float2 *s_ca = reinterpret_cast<float2 *>(s_bkt + c.nbh * IT);     // [QT][M] (cost, acc)
    float *s_t = reinterpret_cast<float *>(s_ca + QT * M);             // [QT][ST]
    float *s_tau = s_t + QT * ST;                                      // [QT]
    int *s_moi = reinterpret_cast<int *>(s_tau + QT);                  // [I]
    stage_tables(c, sb, 0, IT, s_ent, s_bkt);
    for (int jj = threadIdx.x; jj < I; jj += blockDim.x) s_moi[jj] = c.moi[jj];
    InstRegs r = {};
    if (jv) r = load_inst(c, sb, j, jl);
    const int fast = __syncthreads_and(!jv || sb.inst[j].fast);

    const int rr2 = threadIdx.x / TPR;  // phase-2 row
    const int u = threadIdx.x % TPR;    // phase-2 lane within the row group

    for (int q0 = rb; q0 < re; q0 += QT) {
        const int nrows = min(QT, re - q0);
        if ((int)threadIdx.x < nrows) {
            bool ok;
            const int p = a.prompt[q0 + threadIdx.x];
            s_q[threadIdx.x] = make_qrec(p, c.pmax, &ok);
            if (!ok) record_status(a.ctl, kEInval);
            if (CONSTRAINED) s_tau[threadIdx.x] = a.tau[q0 + threadIdx.x];
        }
        // per (row, model): cost of App. B.4 and the predicted accuracy
        for (int idx = threadIdx.x; idx < nrows * M; idx += blockDim.x) {
            const int rr = idx / M;
            const int m = idx - rr * M;
            const size_t g = (size_t)(q0 + rr) * M + m;
            const float cost = __fmaf_rn((float)a.dec_hat[g], c.pout[m], __fmul_rn((float)a.prompt[q0 + rr], c.pin[m]));
            s_ca[idx] = make_float2(cost, a.acc[g]);
        }
        __syncthreads();
        if (jv) {
            for (int rr = qs; rr < nrows; rr += QS) {
                const QRec q = s_q[rr];
                const int k = locate(q, r, s_bkt, IT);
                const float4 e = s_ent[k * IT + jl];
                const float t = fast ? ttft_fast<MODE>(q, r, e)
                                     : ttft_exact64<MODE>(q, r, e, sb.f3[(size_t)k * I + j]);
                s_t[rr * ST + j] = t;
                if (MATRIX) __stcs(a.ttft + (size_t)(q0 + rr) * I + j, t);
            }
        }
        __syncthreads();
        const bool live = rr2 < nrows;
        const float *trow = s_t + (live ? rr2 : 0) * ST;
        const float2 *carow = s_ca + (live ? rr2 : 0) * M;
        for (int pp = 0; pp < a.P; ++pp) {
            const float lam = a.lam[pp];
            const float mu = a.mu[pp];
            float best = 0.f, bestu = 0.f, fastest = 0.f;
            int bj = kBig, bju = kBig, bjt = kBig;
            if (live) {
                const float tau = CONSTRAINED ? s_tau[rr2] : 0.f;
                for (int jj = u; jj < I; jj += TPR) {
                    const float t = trow[jj];
                    const float2 ca = carow[s_moi[jj]];
                    const float U = __fmaf_rn(-lam, ca.x, ca.y);
                    if (CONSTRAINED) {
                        if (t <= tau && (bju == kBig || U > bestu)) { bestu = U; bju = jj; }
                        if (t == t && (bjt == kBig || t < fastest)) { fastest = t; bjt = jj; }
                    } else {
                        const float J = __fmaf_rn(-mu, t, U);
                        if (J == J && (bj == kBig || J > best)) { best = J; bj = jj; }
                    }
                }
            }
            for (int o = TPR >> 1; o > 0; o >>= 1) {
                if (CONSTRAINED) {
                    const float ou = __shfl_xor_sync(kFull, bestu, o);
                    const int oj = __shfl_xor_sync(kFull, bju, o);
                    if (oj != kBig && (bju == kBig || ou > bestu || (ou == bestu && oj < bju))) { bestu = ou; bju = oj; }
                    const float ot = __shfl_xor_sync(kFull, fastest, o);
                    const int ojt = __shfl_xor_sync(kFull, bjt, o);
                    if (ojt != kBig && (bjt == kBig || ot < fastest || (ot == fastest && ojt < bjt))) { fastest = ot; bjt = ojt; }
                } else {
                    const float oJ = __shfl_xor_sync(kFull, best, o);
                    const int oj = __shfl_xor_sync(kFull, bj, o);
                    if (oj != kBig && (bj == kBig || oJ > best || (oJ == best && oj < bj))) { best = oJ; bj = oj; }
                }
            }
            if (live && u == 0) {
                const int pick = CONSTRAINED ? (bju != kBig ? bju : bjt) : bj;
                const size_t o = (size_t)pp * a.Q + q0 + rr2;
                if (pick == kBig) {
                    a.assign[o] = -1;
                    a.util[o] = __int_as_float(0x7fc00000);
                    if (a.ttft_chosen) a.ttft_chosen[o] = __int_as_float(0x7fc00000);
                } else {
                    const float2 ca = carow[s_moi[pick]];
                    a.assign[o] = pick;
                    a.util[o] = __fmaf_rn(-lam, ca.x, ca.y);
                    if (a.ttft_chosen) a.ttft_chosen[o] = trow[pick];
                }
            }
        }
        __syncthreads();
    }
}

// Per-pair means of (accuracy, cost, TTFT) of the chosen instances, fp64, fixed
// reduction order (one CTA per pair).
__global__ void __launch_bounds__(256) k_frontier(const K2Launch a, double *out) {
    __shared__ double red[3][256];
    const int pp = blockIdx.x;
    const DevConfig &c = a.cfg;
    double sa = 0.0, sc = 0.0, st = 0.0;
    for (int i = threadIdx.x; i < a.Q; i += blockDim.x) {
        const size_t o = (size_t)pp * a.Q + i;
        const int jj = a.assign[o];
        if (jj < 0) {
            sa = sc = st = __longlong_as_double(0x7ff8000000000000LL);
            continue;
        }
        const int m = c.moi[jj];
        const size_t g = (size_t)i * c.M + m;
        const float cost = __fmaf_rn((float)a.dec_hat[g], c.pout[m], __fmul_rn((float)a.prompt[i], c.pin[m]));
        sa += (double)a.acc[g];
        sc += (double)cost;
        st += (double)a.ttft_chosen[o];
    }
    red[0][threadIdx.x] = sa;
    red[1][threadIdx.x] = sc;
    red[2][threadIdx.x] = st;
    __syncthreads();
    for (int s = blockDim.x / 2; s > 0; s >>= 1) {
        if ((int)threadIdx.x < s)
            for (int f = 0; f < 3; ++f) red[f][threadIdx.x] += red[f][threadIdx.x + s];
        __syncthreads();
    }
    if (threadIdx.x < 3) out[pp * 3 + threadIdx.x] = red[threadIdx.x][0] / (double)a.Q;
}

template <int MODE>
cudaError_t launch_est_mode(const K2Launch &a, int kind, dim3 grid, int block, size_t smem, cudaStream_t st) {
    if (kind == kEstFeatures) {
        k_estimate<MODE, kOutFeatures><<<grid, block, smem, st>>>(a);
    } else if (a.first_batch) {
        k_estimate<MODE, kOutTtftIters><<<grid, block, smem, st>>>(a);
    } else {
        k_estimate<MODE, kOutTtft><<<grid, block, smem, st>>>(a);
    }
    return cudaGetLastError();
}

template <int MODE, bool CON>
cudaError_t launch_route_mode(const K2Launch &a, dim3 grid, int block, size_t smem, cudaStream_t st) {
    if (a.ttft) k_route<MODE, CON, true><<<grid, block, smem, st>>>(a);
    else k_route<MODE, CON, false><<<grid, block, smem, st>>>(a);
    return cudaGetLastError();
}

template <typename F>
cudaError_t set_attr(F f, size_t bytes) {
    return cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace

cudaError_t launch_estimate(const K2Launch &a, int kind, dim3 grid, int block, size_t smem, cudaStream_t st) {
    return a.cfg.mode == 0 ? launch_est_mode<0>(a, kind, grid, block, smem, st)
                           : launch_est_mode<1>(a, kind, grid, block, smem, st);
}

cudaError_t launch_route(const K2Launch &a, dim3 grid, int block, size_t smem, cudaStream_t st) {
    const bool con = a.tau != nullptr;
    if (a.cfg.mode == 0) return con ? launch_route_mode<0, true>(a, grid, block, smem, st)
                                    : launch_route_mode<0, false>(a, grid, block, smem, st);
    return con ? launch_route_mode<1, true>(a, grid, block, smem, st)
               : launch_route_mode<1, false>(a, grid, block, smem, st);
}

cudaError_t launch_frontier(const K2Launch &a, double *out, cudaStream_t st) {
    k_frontier<<<a.P, 256, 0, st>>>(a, out);
    return cudaGetLastError();
}

cudaError_t set_k2_smem(size_t est, size_t route) {
    cudaError_t e = cudaSuccess;
    const cudaError_t es[] = {
        set_attr(k_estimate<0, kOutTtft>, est), set_attr(k_estimate<0, kOutTtftIters>, est),
        set_attr(k_estimate<0, kOutFeatures>, est), set_attr(k_estimate<1, kOutTtft>, est),
        set_attr(k_estimate<1, kOutTtftIters>, est), set_attr(k_estimate<1, kOutFeatures>, est),
        set_attr(k_route<0, true, true>, route), set_attr(k_route<0, true, false>, route),
        set_attr(k_route<0, false, true>, route), set_attr(k_route<0, false, false>, route),
        set_attr(k_route<1, true, true>, route), set_attr(k_route<1, true, false>, route),
        set_attr(k_route<1, false, true>, route), set_attr(k_route<1, false, false>, route)};
    for (cudaError_t x : es)
        if (x != cudaSuccess) e = x;
    return e;
}

cudaError_t estimate_occupancy(int kind, int mode, int block, size_t smem, int *n) {
    (void)kind;
    return mode == 0 ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_estimate<0, kOutTtft>, block, smem)
                     : cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_estimate<1, kOutTtft>, block, smem);
}

cudaError_t route_occupancy(int mode, int block, size_t smem, int *n) {
    return mode == 0 ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_route<0, false, true>, block, smem)
                     : cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_route<1, false, true>, block, smem);
}

}  // namespace lr
