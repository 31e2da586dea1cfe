// K2: per-candidate SFS TTFT (Sec. 4.1, Eq. 7-9), utility (Eq. 2) and the
// per-query argmax (Eq. 3, Eq. 5).
//
// Each thread owns four consecutive instances of its CTA's instance tile and
// walks the CTA's query rows; the instances' summaries (written by K1) sit in
// shared memory, their scalars in registers.  For a query of prompt p:
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
// the FMA pipe; instances whose totals reach 2^44 take an int64 path.
//
// The estimate matrix is write-only (4 bytes per candidate) and leaves as one
// 16-byte evict-first store per thread and row.  Routing reduces each row with
// redux.sync over order-preserving integer keys of the objective: the lowest
// lane (lowest instance) among the maximal keys wins, as in a first-max scan.
#include <math.h>

#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr long long kLowMask = (1LL << kSplitBits) - 1;
constexpr float kNaN = __builtin_nanf("");

struct __align__(16) QRec {
    int p;     // prompt length, clamped into [1, pmax] for table lookups
    float fp;  // p as fp32, NaN if p was out of range
    float ph;  // p(p+1)/2 high part (multiple of 2^20)
    float pl;  // p(p+1)/2 low part
};

__device__ __forceinline__ QRec make_qrec(int p, int pmax, bool *ok) {
    QRec q;
    *ok = p >= 1 && p <= pmax;
    if (!*ok) p = 1;
    const long long pp = ((long long)p * (p + 1)) / 2;
    const long long pl = pp & kLowMask;
    q.p = p;
    q.fp = *ok ? (float)p : kNaN;
    q.ph = __ll2float_rn(pp - pl);
    q.pl = __ll2float_rn(pl);
    return q;
}

// Order-preserving key of a float (no NaN): larger float <-> larger key, and
// -0 and +0 share a key.  Zero is below every key.
__device__ __forceinline__ unsigned order_key(float x) {
    const unsigned u = __float_as_uint(__fadd_rn(x, 0.0f));
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// ---------------------------------------------------------------------------
// Integer features (exact, for verification): one thread per candidate.
__global__ void __launch_bounds__(256) k_features(const K2Launch a) {
    const DevConfig &c = a.cfg;
    const int active = *((volatile int32_t *)&a.ctl->active);
    const long long total = (long long)a.Q * c.I;
    const int off = (c.mode == 0) ? 1 : 0;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int i = (int)(idx / c.I);
        const int j = (int)(idx - (long long)i * c.I);
        long long *F = a.features + idx * 5;
        const int p = a.prompt[i];
        if (active < 0 || p < 1 || p > c.pmax) {
            record_status(a.ctl, active < 0 ? kENoState : kEInval);
            for (int f = 0; f < 5; ++f) F[f] = -1;
            continue;
        }
        const StateBuf sb = active ? a.buf1 : a.buf0;
        const InstParams ip = sb.inst[j];
        const int2 bk = sb.bkt[(size_t)(p >> ip.shift) * c.I + j];
        const int k = bk.y + (p > bk.x ? 1 : 0);
        const size_t e = (size_t)k * c.I + j;
        F[0] = ip.la + k + off;
        F[1] = ip.f1tot + p;
        F[2] = sb.f2[e];
        F[3] = sb.f3[e] + (c.mode == 0 ? p : 0);
        F[4] = ip.f4tot + ((long long)p * (p + 1)) / 2;
    }
}

// ---------------------------------------------------------------------------
// The candidate kernel.
enum : int {
    kOutMatrix = 1,   // write the TTFT matrix
    kOutIters = 2,    // write the first-token batch index
    kOutLag = 4,      // Lagrangian argmax (Eq. 5), one (lambda, mu) pair
    kOutCon = 8,      // constrained argmax (Eq. 3), one lambda
    kOutSweep = 16    // Lagrangian argmax for several pairs
};

struct Inst4 {
    int shift[4];
    float h1[4], l1[4], h4[4], l4[4], b1p[4], b2[4], b3[4];
};

// T = T_k (the first two terms, which depend on k* only), f3 = fp32(F3 of the candidate).
__device__ __forceinline__ float ttft_fast(const QRec &q, const Inst4 &r, int u, float T, float f3) {
    const float f1 = __fadd_rn(r.h1[u], __fadd_rn(r.l1[u], q.fp));
    const float f4 = __fadd_rn(__fadd_rn(r.h4[u], q.ph), __fadd_rn(r.l4[u], q.pl));
    float t = __fmaf_rn(r.b1p[u], f1, T);
    t = __fmaf_rn(r.b2[u], f3, t);
    t = __fmaf_rn(r.b3[u], f4, t);
    return t;
}

// Exact int64 path for instances whose totals do not split into fp32.
template <int MODE>
__device__ float ttft_exact64(const DevConfig &c, const StateBuf &sb, const QRec &q, int j, int k, const float T) {
    if (q.fp != q.fp) return q.fp;
    const InstParams ip = sb.inst[j];
    const int m = c.moi[j];
    const long long p = q.p;
    const float f1 = __ll2float_rn(ip.f1tot + p);
    const float f3 = __ll2float_rn(sb.f3[(size_t)k * c.I + j] + (MODE == 0 ? p : 0));
    const float f4 = __ll2float_rn(ip.f4tot + (p * (p + 1)) / 2);
    float t = __fmaf_rn(c.coef[m * 5 + 1], f1, T);
    t = __fmaf_rn(c.coef[m * 5 + 3], f3, t);
    t = __fmaf_rn(c.coef[m * 5 + 4], f4, t);
    return t;
}

// Reduce a key over the row's lanes; returns the winning lane's value of `v`
// (and its key) to every lane of the row group.  Rows of up to 32 groups sit in
// an aligned power-of-two lane group; wider rows use whole warps per row.
__device__ __forceinline__ unsigned group_mask(int Gp, int lane) {
    if (Gp >= 32) return kFull;
    const unsigned g = (Gp == 32) ? kFull : ((1u << Gp) - 1u);
    return g << (lane & ~(Gp - 1));
}

// A routing candidate: its key, instance, TTFT and utility.
struct Cand {
    unsigned key;  // order key of the objective, 0 = none
    int j;         // instance (the thread-local index before group_pick)
    float t, U;
};

__device__ __forceinline__ int4 pack(const Cand &c) {
    return make_int4((int)c.key, c.j, __float_as_int(c.t), __float_as_int(c.U));
}

__device__ __forceinline__ Cand unpack(const int4 v) {
    return Cand{(unsigned)v.x, v.y, __int_as_float(v.z), __int_as_float(v.w)};
}

__device__ __forceinline__ void write_pick(const K2Launch &a, size_t o, const Cand &w) {
    if (w.key == 0u) {  // invalid prompt: no instance
        a.assign[o] = -1;
        a.util[o] = kNaN;
        if (a.ttft_chosen) a.ttft_chosen[o] = kNaN;
    } else {
        a.assign[o] = w.j;
        a.util[o] = w.U;
        if (a.ttft_chosen) a.ttft_chosen[o] = w.t;
    }
}

// Table loads by 32-bit shared-memory address.  The tables are written once
// before the first barrier and only read afterwards.
__device__ __forceinline__ float2 lds_float2(uint32_t addr) {
    float2 v;
    asm("ld.shared.v2.f32 {%0, %1}, [%2];" : "=f"(v.x), "=f"(v.y) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint32_t lds_u32(uint32_t addr) {
    uint32_t v;
    asm("ld.shared.u32 %0, [%1];" : "=r"(v) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint4 lds_u32x4(uint32_t addr) {
    uint4 v;
    asm("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(addr));
    return v;
}

__device__ __forceinline__ float pick4(const float v[4], int u) {
    float x = v[0];
    x = (u == 1) ? v[1] : x;
    x = (u == 2) ? v[2] : x;
    x = (u == 3) ? v[3] : x;
    return x;
}

// Asynchronous 4-byte global -> shared copies (the staging of the next chunk of
// query rows overlaps the current chunk's compute).
__device__ __forceinline__ void cp_async4(void *smem_dst, const void *gmem_src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"((uint32_t)__cvta_generic_to_shared(smem_dst)),
                 "l"(gmem_src)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// One poll of an mbarrier's phase 0 (true once the bulk copy it tracks has landed).
__device__ __forceinline__ bool mbar_test(uint32_t mbar) {
    uint32_t done;
    asm volatile(
        "{\n .reg .pred P;\n mbarrier.try_wait.parity.shared::cta.b64 P, [%1], 0;\n selp.u32 %0, 1, 0, P;\n}"
        : "=r"(done)
        : "r"(mbar)
        : "memory");
    return done != 0;
}

template <bool B>
struct Flag {
    static constexpr bool value = B;
};

// The rows of a launch, per tile, as ranges (x, end) that a CTA works through QT rows
// at a time.  CTA b < first_ctas starts with the static range [b F, (b + 1) F)
// (F = first_rows, most of its share of the rows): those CTAs fit beside a snapshot
// load's CTAs running on another stream and start at once.  The remaining rows are
// claimed from the tile's counter, which counts the rows past the static ones: QT
// rows while many are left, down to 4 QS at the end (a claim's atomic still returns
// well within the chunk before it).  So CTAs that start late (their SM busy with the
// load) or run slower take less, and all finish at about the same time.  `seen` is
// a row index recently reached.
__device__ __forceinline__ int claim_size(const K2Launch &a, int seen) {
    const int n = (a.Q - seen) / (int)gridDim.x;
    return min(a.QT, max(4 * a.QS, n - n % a.QS));
}
__device__ __forceinline__ int static_rows(const K2Launch &a) { return min(a.Q, a.first_ctas * a.first_rows); }
// Every row of the launch lies in a static range: no CTA claims, and the counters stay
// untouched (and zero) -- a call that runs alone takes no atomic round trip at all.
__device__ __forceinline__ bool all_static(const K2Launch &a) { return (long long)a.first_ctas * a.first_rows >= a.Q; }
__device__ __forceinline__ int claim_rows(const K2Launch &a, int seen) {
    if (all_static(a)) return a.Q;
    return static_rows(a) + (int)atomicAdd(a.work + 1 + blockIdx.y, (unsigned)claim_size(a, seen));
}
__device__ __forceinline__ int2 first_range(const K2Launch &a) {
    if ((int)blockIdx.x < a.first_ctas)
        return make_int2((int)blockIdx.x * a.first_rows, ((int)blockIdx.x + 1) * a.first_rows);
    const int seen = static_rows(a) + (int)*(volatile uint32_t *)(a.work + 1 + blockIdx.y);
    const int x = claim_rows(a, seen);
    return make_int2(x, x + claim_size(a, seen));
}
// The range left after the chunk at the head of r, if any: no claim needed.
__device__ __forceinline__ bool has_rest(const K2Launch &a, int2 r) { return r.x + a.QT < min(r.y, a.Q); }
// The range that follows the chunk at the head of r (the claim x was made for it).
__device__ __forceinline__ int2 range_after(const K2Launch &a, int2 r, int x) {
    return has_rest(a, r) ? make_int2(r.x + a.QT, r.y) : make_int2(x, x + claim_size(a, r.x));
}

// End of a candidate-kernel CTA: the last of `ctas` to finish clears the row
// counters of the `tiles` tiles and the completion count for the next launch.
__device__ __forceinline__ void k2_finish(const K2Launch &a, uint32_t *work, unsigned ctas, unsigned tiles) {
    if (all_static(a)) return;  // no counter was touched
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        if (atomicAdd(work, 1u) == ctas - 1) {
            for (unsigned y = 0; y < tiles; ++y) atomicExch(work + 1 + y, 0u);
            atomicExch(work, 0u);
            __threadfence();
        }
    }
}

// MODE 0 / 1: SFS with the first output token in its own batch / with the last
// prompt chunk.  MODE 2: an average-case source (Sec. 4, App. E), affine in p:
// t = fma(p, g_j, C_j) with g_j = fp32(1/theta_j) and C_j = fp32(W_j + Tdec_j).
// Routing launches three 256-thread CTAs per SM, the estimate alone one 768-thread CTA
// (the same registers per thread either way).
template <int MODE, int OUT>
__global__ void __launch_bounds__((OUT & (kOutLag | kOutCon | kOutSweep)) ? kK2Block : kK2EstBlock,
                                  (OUT & (kOutLag | kOutCon | kOutSweep)) ? 3 : 1) k_cand(const K2Launch a) {
    extern __shared__ __align__(16) unsigned char smem[];
    constexpr bool AFF = MODE == 2;
    constexpr bool ROUTE = (OUT & (kOutLag | kOutCon | kOutSweep)) != 0;
    constexpr bool CON = (OUT & kOutCon) != 0;
    constexpr bool SWEEP = (OUT & kOutSweep) != 0;
    constexpr int off = (MODE == 0) ? 1 : 0;
    const DevConfig &c = a.cfg;
    const int I = c.I, M = c.M, Gp = a.Gp, QS = a.QS, QT = a.QT;
    const int lane = threadIdx.x & 31;
    const int g = threadIdx.x % Gp;
    const int qs = threadIdx.x / Gp;
    const int j0 = blockIdx.y * Gp * 4;
    const int jb = j0 + 4 * g;                         // first instance of this thread
    const int nv = max(0, min(4, I - jb));             // instances this thread owns
    // Query rows come in ranges (first_range, range_after): a static one, then claims
    // from this tile's counter, in the no-snapshot path as in the main one.
    __shared__ int s_active;
    __shared__ int2 s_claim[2];
    __shared__ __align__(8) unsigned long long s_mbar;
    const uint32_t mbar = (uint32_t)__cvta_generic_to_shared(&s_mbar);
    const size_t tb = tile_bytes(c);
    // Shared memory: the tile block (tables and per-instance scalars, exactly as K1
    // laid it out for this tile), query records, row partials, utility inputs,
    // targets and the raw query rows (route with one pair stages (U, cost) per row
    // and model, sweeps (cost, acc)).
    const int WPR = Gp > 32 ? Gp / 32 : 1;  // warps per row
    const int NP = SWEEP ? a.P : 1;
    QRec *s_q = reinterpret_cast<QRec *>(smem + tb);                                   // [QT]
    int4 *s_part = reinterpret_cast<int4 *>(s_q + QT);                                 // [NP][QT][WPR][2]
    float2 *s_ca = reinterpret_cast<float2 *>(s_part + (ROUTE && Gp > 32 ? 2 * NP * QT * WPR : 0));  // [QT][M]
    float *s_tau = reinterpret_cast<float *>(s_ca + (ROUTE ? QT * M : 0));             // [QT]
    // raw query rows as copied from global memory, two chunks in flight:
    // prompt [2][QT], and for routing tau [2][QT], dec_hat [2][QT][M], acc [2][QT][M]
    int32_t *r_p = reinterpret_cast<int32_t *>(s_tau + (ROUTE ? QT : 0));
    float *r_t = reinterpret_cast<float *>(r_p + 2 * QT);
    int32_t *r_d = reinterpret_cast<int32_t *>(r_t + (ROUTE ? 2 * QT : 0));
    float *r_a = reinterpret_cast<float *>(r_d + (ROUTE ? 2 * QT * M : 0));
    // copies of query rows [q0, q0 + nrows) into raw buffer b
    auto issue = [&](int q0, int nrows, int b) {
        for (int t = threadIdx.x; t < nrows; t += blockDim.x) {
            cp_async4(r_p + b * QT + t, a.prompt + q0 + t);
            if (CON) cp_async4(r_t + b * QT + t, a.tau + q0 + t);
        }
        if (ROUTE) {
            const size_t g0 = (size_t)q0 * M;
            for (int idx = threadIdx.x; idx < nrows * M; idx += blockDim.x) {
                cp_async4(r_d + b * QT * M + idx, a.dec_hat + g0 + idx);
                cp_async4(r_a + b * QT * M + idx, a.acc + g0 + idx);
            }
        }
        cp_async_commit();
    };
    // The tile block arrives with one bulk copy (TMA) completing on an mbarrier:
    // every CTA reads the same few tens of KB, and one large request per CTA is far
    // cheaper than thousands of scattered loads of the same lines.
    auto tile_copy = [&](const unsigned char *src, uint32_t dst_off) {
        asm volatile(
            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                (uint32_t)__cvta_generic_to_shared(smem) + dst_off),
            "l"(src), "r"((uint32_t)tb), "r"(mbar)
            : "memory");
    };
    // bounded wait for the tile block: a copy that never lands is reported, not waited out
    auto tile_wait = [&]() -> bool {
        bool landed = false;
        for (int it = 0; it < (1 << 22) && !landed; ++it) landed = mbar_test(mbar);
        return landed;
    };
    if (threadIdx.x == 0) {
        if (!AFF) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(mbar) : "memory");
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        }
        s_claim[0] = first_range(a);
    }
    __syncthreads();
    const int2 first = s_claim[0];
    // the first chunk of query rows travels while the live index is read and the tile
    // block lands; one read of the live-buffer index per CTA (every thread reading the
    // same word would queue them all on one L2 line)
    if (first.x < a.Q) issue(first.x, min(QT, min(first.y, a.Q) - first.x), 0);
    if (threadIdx.x == 0) s_active = load_live(a.ctl);
    __syncthreads();
    const int active = s_active;
    // the LPS source and a given matrix need no live snapshot; every other source does
    if (active < 0 && !(AFF && (a.src == kSrcLps || a.src == kSrcMatrix))) {
        if (threadIdx.x == 0) record_status(a.ctl, kENoState);
        cp_async_wait<0>();  // nothing may still be landing when the CTA leaves
        for (int k = 0;; ++k) {
            __syncthreads();  // the previous range has been read
            if (threadIdx.x == 0 && k > 0) {
                const int2 r = s_claim[0];
                s_claim[0] = range_after(a, r, has_rest(a, r) ? 0 : claim_rows(a, r.x));
            }
            __syncthreads();
            const int rb = s_claim[0].x, re = min(min(a.Q, s_claim[0].y), rb + QT);
            if (rb >= a.Q) break;
            for (int rr = rb + qs; rr < re; rr += QS) {
                for (int u = 0; u < nv; ++u) {
                    if (OUT & kOutMatrix) a.ttft[(size_t)rr * I + jb + u] = kNaN;
                    if (OUT & kOutIters) a.first_batch[(size_t)rr * I + jb + u] = -1;
                }
                if (ROUTE && g == 0)
                    for (int pp = 0; pp < a.P; ++pp) {
                        a.assign[(size_t)pp * a.Q + rr] = -1;
                        a.util[(size_t)pp * a.Q + rr] = kNaN;
                        if (a.ttft_chosen) a.ttft_chosen[(size_t)pp * a.Q + rr] = kNaN;
                    }
            }
        }
        k2_finish(a, a.work, gridDim.x * gridDim.y, gridDim.y);
        return;
    }
    {
    const StateBuf sb = active ? a.buf1 : a.buf0;
    // (Gp == c.tgp: the tile block's sections at the offsets K1 wrote them)
    const unsigned char *tile = smem;
    const unsigned char *s_ent = tile;                                                         // entA, entB
    const unsigned char *s_bkt = tile + tile_ent_bytes(c);                                     // [nbh][4][Gp]
    const int32_t *s_scal = reinterpret_cast<const int32_t *>(s_bkt + tile_bkt_bytes(c));    // [kScal][4][Gp]
    if (threadIdx.x == 0 && !AFF) {
        // the block was written by generic stores (possibly of a load on another
        // stream, acquired above); order them before the bulk copy's reads
        asm volatile("fence.proxy.async.global;" ::: "memory");
        asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(mbar), "r"((uint32_t)tb) : "memory");
        tile_copy(sb.tile + (size_t)blockIdx.y * tb, 0u);
    }
    // what follows the first chunk: found now, published once the tile block has landed
    int2 second = make_int2(a.Q, a.Q);
    if (threadIdx.x == 0 && first.x < a.Q) second = range_after(a, first, has_rest(a, first) ? 0 : claim_rows(a, first.x));
    if (!AFF) {
        if (__syncthreads_or(!tile_wait())) {
            if (threadIdx.x == 0) record_status(a.ctl, kECuda);
            for (int it = 0; it < (1 << 22) && !mbar_test(mbar); ++it) {
            }
            cp_async_wait<0>();
            goto finish;
        }
    }
    Inst4 r;
    int model[4], la[4];
    float ag[4], ac[4];  // average-case sources: t = fma(p, ag, ac)
    bool fast_mine = true, compact_mine = true;
    const int fs = 4 * Gp;  // scalar field stride
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        if (AFF) {
            const int j = min(jb + u, I - 1);
            model[u] = c.moi[j];
            const QueueDev qd = a.qd[j];
            ag[u] = qd.g;
            // throughput source: residents' remaining prefill tokens / theta + Tdec
            ac[u] = (a.src == kSrcLps)      ? qd.clps
                    : (a.src == kSrcMatrix) ? 0.f
                                            : __double2float_rn(__dadd_rn(__ddiv_rn((double)sb.inst[j].f1tot, qd.theta), qd.tdec));
            continue;
        }
        const int col = u * Gp + g;
        r.shift[u] = s_scal[kScShift * fs + col];
        r.h1[u] = __int_as_float(s_scal[kScH1 * fs + col]);
        r.l1[u] = __int_as_float(s_scal[kScL1 * fs + col]);
        r.h4[u] = __int_as_float(s_scal[kScH4 * fs + col]);
        r.l4[u] = __int_as_float(s_scal[kScL4 * fs + col]);
        r.b1p[u] = __int_as_float(s_scal[kScB1p * fs + col]);
        r.b2[u] = __int_as_float(s_scal[kScB2 * fs + col]);
        r.b3[u] = __int_as_float(s_scal[kScB3 * fs + col]);
        model[u] = s_scal[kScModel * fs + col];
        la[u] = s_scal[kScLa * fs + col];
        if (u < nv) fast_mine = fast_mine && s_scal[kScFast * fs + col] != 0;
        if (u < nv) compact_mine = compact_mine && s_scal[kScCompact * fs + col] != 0;
    }
    // the bucket width of the tile's first instance (SPEC needs one width per CTA)
    const int shift0 = AFF ? 0 : s_scal[kScShift * fs];
    if (threadIdx.x == 0) s_claim[1] = second;
    const bool fast = __syncthreads_and(fast_mine);
    const bool vec = a.vec_ok && nv == 4;
    const unsigned gmask = group_mask(Gp, lane);
    const int grp_lane0 = lane & ~(min(Gp, 32) - 1);  // first lane of this row group in the warp
    const int wrow = g / 32;                          // warp index within a wide row
    // shared addresses of this thread's table columns: entA (k, u) at
    // ecol + u * ecst + k * erow (entB ebofs further), bucket (b, u) at
    // bcol + 4 u + b * brow (formed at each use: the kernel is at its register limit)
    const uint32_t ecol = (uint32_t)__cvta_generic_to_shared(s_ent) + 8u * (uint32_t)g;
    const uint32_t bcol = (uint32_t)__cvta_generic_to_shared(s_bkt) + 16u * (uint32_t)g;
    const uint32_t ecst = 8u * (uint32_t)Gp;
    const uint32_t erow = 8u * 4u * (uint32_t)Gp, brow = 4u * 4u * (uint32_t)Gp;
    const uint32_t ebofs = (uint32_t)tile_enta_bytes(c);
    bool same_model = true;
#pragma unroll
    for (int u = 1; u < 4; ++u) same_model = same_model && model[u] == model[0];

    bool same_shift = true;
#pragma unroll
    for (int u = 0; u < 4; ++u) same_shift = same_shift && (AFF || r.shift[u] == shift0);
    // SPEC: every thread of the CTA has four compact instances of one model (the fp32
    // split path, F3 read from entA alone), every instance of the CTA the same bucket
    // width (a thread's four buckets are one 16-byte load) and aligned vector stores, so
    // none of the per-thread checks below is needed (an invalid prompt still gives NaN
    // times, which no comparison selects)
    const bool spec = __syncthreads_and(fast && compact_mine && nv == 4 && same_model && same_shift && a.vec_ok);
    auto run = [&](auto fast_tag, auto spec_tag) {
        constexpr bool FAST = decltype(fast_tag)::value;
        constexpr bool SPEC = decltype(spec_tag)::value;
        // chunk k: the first QT rows of the range in s_claim[k & 1], staged in raw buffer k & 1
        for (int buf = 0;; buf ^= 1) {
            int q0, nrows;
            {
                const int2 cur = s_claim[buf], nxt = s_claim[buf ^ 1];
                if (cur.x >= a.Q) break;
                q0 = cur.x;
                nrows = min(QT, min(cur.y, a.Q) - q0);
                if (nxt.x < a.Q) {
                    issue(nxt.x, min(QT, min(nxt.y, a.Q) - nxt.x), buf ^ 1);
                    cp_async_wait<1>();
                } else {
                    cp_async_wait<0>();
                }
            }
            __syncthreads();  // every thread's copies of this chunk have landed
            // the range after the next chunk: claimed now if needed, published when this chunk is done
            int ahead = a.Q;
            if (threadIdx.x == 0 && s_claim[buf ^ 1].x < a.Q && !has_rest(a, s_claim[buf ^ 1]))
                ahead = claim_rows(a, s_claim[buf ^ 1].x);
            const int32_t *bp = r_p + buf * QT;
            for (int t = threadIdx.x; t < nrows; t += blockDim.x) {
                bool ok;
                s_q[t] = make_qrec(bp[t], c.pmax, &ok);
                if (!ok && blockIdx.y == 0) record_status(a.ctl, kEInval);
                if (CON) s_tau[t] = r_t[buf * QT + t];
            }
            if (ROUTE) {
                const int32_t *bd = r_d + buf * QT * M;
                const float *ba = r_a + buf * QT * M;
                for (int idx = threadIdx.x; idx < nrows * M; idx += blockDim.x) {
                    const int rr = idx / M;
                    const int m = idx - rr * M;
                    const float cost = __fmaf_rn((float)bd[idx], c.pout[m], __fmul_rn((float)bp[rr], c.pin[m]));
                    const float acc = ba[idx];
                    // one pair: stage U itself (x), else (cost, acc)
                    s_ca[idx] = SWEEP ? make_float2(cost, acc) : make_float2(__fmaf_rn(-a.lam[0], cost, acc), cost);
                }
            }
            __syncthreads();
            float *orow = (OUT & kOutMatrix) ? a.ttft + (size_t)(q0 + qs) * I + jb : nullptr;
            const size_t ostep = (size_t)QS * I;
            for (int rr = qs; rr < nrows; rr += QS) {
                const QRec q = s_q[rr];
                const uint32_t p7 = (uint32_t)q.p << 7;
                float t[4];
                int kk[4];
                uint4 bw4 = make_uint4(0u, 0u, 0u, 0u);
                if (SPEC && !AFF) bw4 = lds_u32x4(bcol + (uint32_t)(q.p >> shift0) * brow);
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    if (AFF) {
                        if (a.src == kSrcMatrix)
                            t[u] = u < nv ? __ldcs(a.ttft_in + (size_t)(q0 + rr) * I + jb + u) : kNaN;
                        else t[u] = __fmaf_rn(q.fp, ag[u], ac[u]);
                        kk[u] = 0;
                        continue;
                    }
                    // bucket word (boundary << 7) | below: p > boundary iff (p << 7) > word
                    const uint32_t bw = SPEC ? (u == 0 ? bw4.x : u == 1 ? bw4.y : u == 2 ? bw4.z : bw4.w)
                                             : lds_u32(bcol + 4u * u + (uint32_t)(q.p >> r.shift[u]) * brow);
                    kk[u] = (int)(bw & 127u) + (p7 > bw ? 1 : 0);
                    const uint32_t ea = ecol + u * ecst + (uint32_t)kk[u] * erow;
                    const float2 e = lds_float2(ea);
                    if (SPEC) {
                        // compact: F3 + p below 2^31, one exact int -> fp32 rounding
                        const float f3 = MODE == 0 ? __int2float_rn(__float_as_int(e.y) + q.p) : e.y;
                        t[u] = ttft_fast(q, r, u, e.x, f3);
                    } else if (FAST) {
                        float f3 = e.y;
                        if (MODE == 0) {
                            const float2 hl = lds_float2(ea + ebofs);
                            f3 = __fadd_rn(hl.x, __fadd_rn(hl.y, q.fp));
                        }
                        t[u] = ttft_fast(q, r, u, e.x, f3);
                    } else {
                        t[u] = (u < nv) ? ttft_exact64<MODE>(c, sb, q, jb + u, kk[u], e.x) : 0.f;
                    }
                }
                if (OUT & kOutMatrix) {
                    if (SPEC || vec) {
                        __stcs(reinterpret_cast<float4 *>(orow), make_float4(t[0], t[1], t[2], t[3]));
                    } else {
                        for (int u = 0; u < nv; ++u) __stcs(orow + u, t[u]);
                    }
                    orow += ostep;
                }
                if (OUT & kOutIters) {
                    const bool bad = q.fp != q.fp;
                    const size_t o = (size_t)(q0 + rr) * I + jb;
                    for (int u = 0; u < nv; ++u) a.first_batch[o + u] = bad ? -1 : la[u] + kk[u] + off;
                }
                if (ROUTE) {
                    const bool row_ok = SPEC || q.fp == q.fp;
                    const float2 *carow = s_ca + rr * M;
                    const float tau = CON ? s_tau[rr] : 0.f;
#pragma unroll 1
                    for (int pp = 0; pp < (SWEEP ? NP : 1); ++pp) {
                        const float lam = SWEEP ? a.lam[pp] : 0.f;
                        const float mu = a.mu[pp];
                        float U[4];
                        if (SPEC || same_model) {
                            const float2 ca = carow[model[0]];
                            U[0] = U[1] = U[2] = U[3] = SWEEP ? __fmaf_rn(-lam, ca.x, ca.y) : ca.x;
                        } else {
#pragma unroll
                            for (int u = 0; u < 4; ++u) {
                                const float2 ca = carow[model[u]];
                                U[u] = SWEEP ? __fmaf_rn(-lam, ca.x, ca.y) : ca.x;
                            }
                        }
                        // this thread's best of its four instances (first max wins); NaN marks
                        // an invalid row or an instance beyond the pool
                        float best1, best2 = 0.f;
                        int u1 = 0, u2 = 0;
                        if (CON) {
                            best1 = ((SPEC || 0 < nv) && row_ok && t[0] <= tau) ? U[0] : kNaN;
                            best2 = ((SPEC || 0 < nv) && row_ok) ? t[0] : kNaN;
#pragma unroll
                            for (int u = 1; u < 4; ++u) {
                                if ((SPEC || u < nv) && t[u] <= tau && (U[u] > best1 || best1 != best1)) { best1 = U[u]; u1 = u; }
                                // a NaN time (no estimate, per candidate only from a matrix
                                // source) is never the least
                                if ((SPEC || u < nv) && (!AFF || t[u] == t[u]) && (t[u] < best2 || (AFF && best2 != best2))) {
                                    best2 = t[u];
                                    u2 = u;
                                }
                            }
                        } else {
                            best1 = ((SPEC || 0 < nv) && row_ok) ? __fmaf_rn(-mu, t[0], U[0]) : kNaN;
#pragma unroll
                            for (int u = 1; u < 4; ++u) {
                                // J is NaN exactly when the time is (no estimate): never chosen.
                                // Only a matrix source mixes NaN and finite times in a row.
                                const float J = __fmaf_rn(-mu, t[u], U[u]);
                                if ((SPEC || u < nv) && (!AFF || J == J) && (J > best1 || (AFF && best1 != best1))) {
                                    best1 = J;
                                    u1 = u;
                                }
                            }
                        }
                        const unsigned k1 = (best1 == best1) ? order_key(best1) : 0u;
                        const unsigned k2 = (CON && best2 == best2 && row_ok) ? order_key(-best2) : 0u;
                        // row group argmax: the lowest lane among the maximal keys
                        const unsigned w1 = __reduce_max_sync(gmask, k1);
                        const int src1 = __ffs(__ballot_sync(gmask, k1 == w1) & gmask) - 1;
                        unsigned w2 = 0u;
                        int src2 = 0;
                        if (CON) {
                            w2 = __reduce_max_sync(gmask, k2);
                            src2 = __ffs(__ballot_sync(gmask, k2 == w2) & gmask) - 1;
                        }
                        // the winner of each reduction describes itself
                        const Cand c1 = {w1, jb + u1, pick4(t, u1), pick4(U, u1)};
                        const Cand c2 = {w2, jb + u2, pick4(t, u2), pick4(U, u2)};
                        if (Gp <= 32) {
                            const bool use2 = CON && w1 == 0u;
                            if (lane == (use2 ? src2 : src1))
                                write_pick(a, (size_t)pp * a.Q + q0 + rr, use2 ? c2 : c1);
                        } else {
                            // wide rows: each warp leaves its partial; combined once per chunk
                            int4 *part = s_part + 2 * ((pp * QT + rr) * WPR + wrow);
                            if (lane == src1) part[0] = pack(c1);
                            if (CON && lane == src2) part[1] = pack(c2);
                        }
                    }
                }
            }
            if (ROUTE && Gp > 32) {
                // one thread per (row, pair) combines the warps of the row in instance order
                __syncthreads();
                for (int t2 = threadIdx.x; t2 < nrows * NP; t2 += blockDim.x) {
                    const int pp = t2 / nrows;
                    const int r2 = t2 - pp * nrows;
                    Cand c1 = {0u, 0, 0.f, 0.f}, c2 = {0u, 0, 0.f, 0.f};
                    for (int wi = 0; wi < WPR; ++wi) {
                        const Cand x1 = unpack(s_part[2 * ((pp * QT + r2) * WPR + wi)]);
                        if (x1.key > c1.key) c1 = x1;
                        if (CON) {
                            const Cand x2 = unpack(s_part[2 * ((pp * QT + r2) * WPR + wi) + 1]);
                            if (x2.key > c2.key) c2 = x2;
                        }
                    }
                    write_pick(a, (size_t)pp * a.Q + q0 + r2, (CON && c1.key == 0u) ? c2 : c1);
                }
            }
            if (threadIdx.x == 0) {  // into the slot this chunk was read from
                const int2 nxt = s_claim[buf ^ 1];
                s_claim[buf] = nxt.x < a.Q ? range_after(a, nxt, ahead) : make_int2(a.Q, a.Q);
            }
            __syncthreads();
        }
    };
    if (spec) run(Flag<true>{}, Flag<true>{});
    else if (fast) run(Flag<true>{}, Flag<false>{});
    else run(Flag<false>{}, Flag<false>{});
    (void)grp_lane0;
    }
finish:
    k2_finish(a, a.work, gridDim.x * gridDim.y, gridDim.y);
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
        if (jj < 0 || jj >= c.I) {
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
cudaError_t launch_cand_mode(const K2Launch &a, int out, dim3 grid, int block, size_t smem, cudaStream_t st) {
    switch (out) {
        case kOutMatrix: k_cand<MODE, kOutMatrix><<<grid, block, smem, st>>>(a); break;
        case kOutMatrix | kOutIters:
            if (MODE == 2) return cudaErrorInvalidValue;  // the batch index exists only for SFS
            k_cand<(MODE == 2 ? 0 : MODE), kOutMatrix | kOutIters><<<grid, block, smem, st>>>(a);
            break;
        case kOutLag: k_cand<MODE, kOutLag><<<grid, block, smem, st>>>(a); break;
        case kOutLag | kOutMatrix: k_cand<MODE, kOutLag | kOutMatrix><<<grid, block, smem, st>>>(a); break;
        case kOutCon: k_cand<MODE, kOutCon><<<grid, block, smem, st>>>(a); break;
        case kOutCon | kOutMatrix: k_cand<MODE, kOutCon | kOutMatrix><<<grid, block, smem, st>>>(a); break;
        case kOutSweep: k_cand<MODE, kOutSweep><<<grid, block, smem, st>>>(a); break;
        case kOutSweep | kOutMatrix: k_cand<MODE, kOutSweep | kOutMatrix><<<grid, block, smem, st>>>(a); break;
        default: return cudaErrorInvalidValue;
    }
    return cudaGetLastError();
}

template <typename F>
cudaError_t set_attr(F f, size_t bytes) {
    return cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

template <int MODE>
cudaError_t set_mode_attrs(size_t bytes) {
    const cudaError_t es[] = {
        set_attr(k_cand<MODE, kOutMatrix>, bytes), set_attr(k_cand<(MODE == 2 ? 0 : MODE), kOutMatrix | kOutIters>, bytes),
        set_attr(k_cand<MODE, kOutLag>, bytes), set_attr(k_cand<MODE, kOutLag | kOutMatrix>, bytes),
        set_attr(k_cand<MODE, kOutCon>, bytes), set_attr(k_cand<MODE, kOutCon | kOutMatrix>, bytes),
        set_attr(k_cand<MODE, kOutSweep>, bytes), set_attr(k_cand<MODE, kOutSweep | kOutMatrix>, bytes)};
    for (cudaError_t x : es)
        if (x != cudaSuccess) return x;
    return cudaSuccess;
}

}  // namespace

int cand_out_flags(bool matrix, bool iters, bool route, bool constrained, int P) {
    int f = 0;
    if (matrix) f |= kOutMatrix;
    if (iters) f |= kOutIters;
    if (route) f |= constrained ? kOutCon : (P > 1 ? kOutSweep : kOutLag);
    return f;
}

cudaError_t launch_cand(const K2Launch &a, int out, dim3 grid, int block, size_t smem, cudaStream_t st) {
    if (a.src != kSrcSfs) return launch_cand_mode<2>(a, out, grid, block, smem, st);
    return a.cfg.mode == 0 ? launch_cand_mode<0>(a, out, grid, block, smem, st)
                           : launch_cand_mode<1>(a, out, grid, block, smem, st);
}

namespace {

// x^k, k >= 0, by binary exponentiation (the bits of k from the least significant).
__device__ double pow_int(double x, int k) {
    double r = 1.0, b = x;
    while (k > 0) {
        if (k & 1) r = __dmul_rn(r, b);
        k >>= 1;
        if (k > 0) b = __dmul_rn(b, b);
    }
    return r;
}

// Per instance: the LPS expected wait of App. E, ((ca2 + cs2) / 2) rho^k / (mu - alpha)
// with rho = alpha / mu, and the fp32 constants of the affine TTFT.
__global__ void k_queue_params(int I, const QueueRaw *raw, QueueDev *qd) {
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    if (j >= I) return;
    const QueueRaw r = raw[j];
    double w = __longlong_as_double(0x7ff8000000000000LL);
    if (r.has_lps) {
        const double rho = __ddiv_rn(r.alpha, r.mu);
        const double c = __dmul_rn(__dadd_rn(r.ca2, r.cs2), 0.5);
        w = __ddiv_rn(__dmul_rn(c, pow_int(rho, r.k)), __dsub_rn(r.mu, r.alpha));
    }
    QueueDev o;
    o.theta = r.theta;
    o.tdec = r.tdec;
    o.wlps = w;
    o.g = __double2float_rn(__ddiv_rn(1.0, r.theta));
    o.clps = __double2float_rn(__dadd_rn(w, r.tdec));
    qd[j] = o;
}

// ---------------------------------------------------------------------------
// Baseline routing policies (Sec. 6, the baselines): the instance is chosen without the
// latency estimates, and the chosen candidate's utility (Eq. 2) and SFS TTFT estimate
// are reported beside it (the TTFT through the same exact path as the candidate
// kernel's, so the two agree bit for bit).  One thread per query.
//   Round Robin: (start + i) mod I.
//   Shortest Queue: the queries in order each join the instance with the fewest
//     resident requests, counting those routed before them, ties to the lowest index.
//     Query k therefore takes the k-th smallest slot (level, j) over the slots
//     instance j offers at levels c_j, c_j + 1, ...: the level L is the largest with
//     N(L) = sum_j max(0, L - c_j) <= k (N from the sorted counts and their prefix
//     sums), and the instance is the (k - N(L))-th, by index, of those with c_j <= L.
//   Latency-Agnostic: the largest utility, ties to the lowest index (utility depends
//     on the instance's model only, so the models are compared at their first instance).
template <int MODE>
__global__ void __launch_bounds__(256) k_baseline(const K2Launch a, int policy, long long rr_start, float lam) {
    extern __shared__ __align__(16) unsigned char bsm[];
    const DevConfig &c = a.cfg;
    const int I = c.I, M = c.M;
    __shared__ int s_active;
    if (threadIdx.x == 0) s_active = load_live(a.ctl);
    __syncthreads();
    const int active = s_active;
    const StateBuf sb = active > 0 ? a.buf1 : a.buf0;
    int P2 = 1;
    while (P2 < I) P2 <<= 1;
    int *cnt = reinterpret_cast<int *>(bsm);                              // [I] resident requests
    int *srt = cnt + I;                                                   // [P2] the counts, sorted
    long long *pre = reinterpret_cast<long long *>(bsm + 8 * ((I + P2 + 1) / 2));  // [I + 1] prefix sums
    int *firstj = reinterpret_cast<int *>(pre + I + 1);                   // [M] first instance of each model
    if (active >= 0 && policy == 1) {
        for (int j = threadIdx.x; j < P2; j += blockDim.x) {
            const int v = j < I ? sb.n_run[j] + sb.n_wait[j] : 0x7fffffff;
            if (j < I) cnt[j] = v;
            srt[j] = v;
        }
        __syncthreads();
        // bitonic sort of srt, ascending
        for (int k = 2; k <= P2; k <<= 1) {
            for (int h = k >> 1; h > 0; h >>= 1) {
                for (int t = threadIdx.x; t < P2; t += blockDim.x) {
                    const int u = t ^ h;
                    if (u > t) {
                        const int x = srt[t], y = srt[u];
                        if (((t & k) == 0) == (x > y)) {
                            srt[t] = y;
                            srt[u] = x;
                        }
                    }
                }
                __syncthreads();
            }
        }
        if (threadIdx.x == 0) {
            long long run = 0;
            for (int t = 0; t < I; ++t) {
                pre[t] = run;
                run += srt[t];
            }
            pre[I] = run;
        }
    }
    if (policy == 2) {
        for (int m = threadIdx.x; m < M; m += blockDim.x) firstj[m] = -1;
        __syncthreads();
        for (int j = threadIdx.x; j < I; j += blockDim.x) atomicMin(reinterpret_cast<unsigned *>(firstj) + c.moi[j], (unsigned)j);
    }
    __syncthreads();
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < a.Q; i += gridDim.x * blockDim.x) {
        const int p = a.prompt[i];
        bool ok;
        const QRec q = make_qrec(p, c.pmax, &ok);
        if (!ok || active < 0) {
            record_status(a.ctl, active < 0 ? kENoState : kEInval);
            a.assign[i] = -1;
            a.util[i] = kNaN;
            if (a.ttft_chosen) a.ttft_chosen[i] = kNaN;
            continue;
        }
        int j = 0;
        if (policy == 0) {
            j = (int)((rr_start + i) % I);
        } else if (policy == 1) {
            // N(L): slots below level L = (#counts below L) * L - (their sum)
            auto slots_below = [&](long long L) -> long long {
                int lo = 0, hi = I;  // first sorted count >= L
                while (lo < hi) {
                    const int mid = (lo + hi) >> 1;
                    if ((long long)srt[mid] < L) lo = mid + 1;
                    else hi = mid;
                }
                return (long long)lo * L - pre[lo];
            };
            long long lo = srt[0], hi = (long long)srt[0] + i + 1;  // N(lo) <= i < N(hi)
            while (hi - lo > 1) {
                const long long mid = (lo + hi) >> 1;
                if (slots_below(mid) <= i) lo = mid;
                else hi = mid;
            }
            long long r = i - slots_below(lo);  // < #{j : c_j <= lo}, so the scan finds it
            for (j = 0; j < I; ++j)
                if ((long long)cnt[j] <= lo && r-- == 0) break;
            j = min(j, I - 1);
        } else {
            float best = 0.f;
            int bj = -1;
            for (int m = 0; m < M; ++m) {
                const int fj = firstj[m];
                if (fj < 0) continue;
                const float cost = __fmaf_rn((float)a.dec_hat[(size_t)i * M + m], c.pout[m], __fmul_rn((float)p, c.pin[m]));
                const float U = __fmaf_rn(-lam, cost, a.acc[(size_t)i * M + m]);
                if (bj < 0 || U > best || (U == best && fj < bj)) {
                    best = U;
                    bj = fj;
                }
            }
            j = bj;
        }
        const int m = c.moi[j];
        const float cost = __fmaf_rn((float)a.dec_hat[(size_t)i * M + m], c.pout[m], __fmul_rn((float)p, c.pin[m]));
        const float U = __fmaf_rn(-lam, cost, a.acc[(size_t)i * M + m]);
        a.assign[i] = j;
        a.util[i] = U;
        if (a.ttft_chosen && a.ttft_in) {
            a.ttft_chosen[i] = a.ttft_in[(size_t)i * I + j];  // the KV-limited estimate
        } else if (a.ttft_chosen) {
            const InstParams ip = sb.inst[j];
            const int2 bk = sb.bkt[(size_t)(q.p >> ip.shift) * I + j];
            const int k = bk.y + (q.p > bk.x ? 1 : 0);
            const float T =
                reinterpret_cast<const float2 *>(sb.tile + tile_base(c, j))[(size_t)k * 4 * c.tgp + tile_col(c, j)].x;
            a.ttft_chosen[i] = ttft_exact64<MODE>(c, sb, q, j, k, T);
        }
    }
}

// OnTimeUtility (Eq. 4) and SLO attainment: CTA b sums the fixed row range
// [b R, (b + 1) R) in a fixed tree order into part[2 b .. 2 b + 1]; k_on_time_final
// adds the parts in index order.  The realized TTFT is the fp32 sum delay + ttft.
__global__ void __launch_bounds__(256) k_on_time_part(int Q, const float *util, const float *ttft, const float *tau,
                                                      const float *delay, double *part) {
    __shared__ double su[256], sn[256];
    const int R = (Q + gridDim.x - 1) / gridDim.x;
    const int lo = blockIdx.x * R, hi = min(Q, lo + R);
    double u = 0.0, n = 0.0;
    for (int i = lo + threadIdx.x; i < hi; i += blockDim.x) {
        const float realized = delay ? __fadd_rn(delay[i], ttft[i]) : ttft[i];
        if (realized <= tau[i]) {
            u += (double)util[i];
            n += 1.0;
        }
    }
    su[threadIdx.x] = u;
    sn[threadIdx.x] = n;
    __syncthreads();
    for (int h = 128; h > 0; h >>= 1) {
        if (threadIdx.x < h) {
            su[threadIdx.x] += su[threadIdx.x + h];
            sn[threadIdx.x] += sn[threadIdx.x + h];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        part[2 * blockIdx.x] = su[0];
        part[2 * blockIdx.x + 1] = sn[0];
    }
}

__global__ void k_on_time_final(int Q, int parts, const double *part, double *out) {
    if (threadIdx.x == 0 && blockIdx.x == 0) {
        double u = 0.0, n = 0.0;
        for (int b = 0; b < parts; ++b) {
            u += part[2 * b];
            n += part[2 * b + 1];
        }
        out[0] = u / Q;
        out[1] = n / Q;
    }
}

}  // namespace

cudaError_t launch_queue_params(int I, const QueueRaw *raw, QueueDev *qd, cudaStream_t st) {
    k_queue_params<<<(I + 127) / 128, 128, 0, st>>>(I, raw, qd);
    return cudaGetLastError();
}

cudaError_t launch_features(const K2Launch &a, int sms, cudaStream_t st) {
    const long long total = (long long)a.Q * a.cfg.I;
    const int grid = (int)std::min<long long>((total + 255) / 256, (long long)sms * 8);
    k_features<<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_frontier(const K2Launch &a, double *out, cudaStream_t st) {
    k_frontier<<<a.P, 256, 0, st>>>(a, out);
    return cudaGetLastError();
}

size_t baseline_smem(const DevConfig &c) {
    int P2 = 1;
    while (P2 < c.I) P2 <<= 1;
    return 8 * (size_t)((c.I + P2 + 1) / 2) + 8 * (size_t)(c.I + 1) + 4 * (size_t)c.M;
}

cudaError_t launch_baseline(const K2Launch &a, int policy, long long rr_start, float lam, int sms, cudaStream_t st) {
    const size_t smem = baseline_smem(a.cfg);
    const int grid = std::max(1, std::min((a.Q + 255) / 256, sms * 4));
    if (a.cfg.mode == 0) k_baseline<0><<<grid, 256, smem, st>>>(a, policy, rr_start, lam);
    else k_baseline<1><<<grid, 256, smem, st>>>(a, policy, rr_start, lam);
    return cudaGetLastError();
}

cudaError_t launch_on_time(int Q, const float *util, const float *ttft, const float *tau, const float *delay,
                           double *part, int max_parts, double *out, cudaStream_t st) {
    const int parts = std::max(1, std::min(max_parts, (Q + 2047) / 2048));
    k_on_time_part<<<parts, 256, 0, st>>>(Q, util, ttft, tau, delay, part);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_on_time_final<<<1, 32, 0, st>>>(Q, parts, part, out);
    return cudaGetLastError();
}

cudaError_t set_baseline_smem(size_t bytes) {
    cudaError_t e = cudaFuncSetAttribute(k_baseline<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_baseline<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    return e;
}

cudaError_t set_k2_smem(size_t bytes) {
    cudaError_t e = set_mode_attrs<0>(bytes);
    if (e == cudaSuccess) e = set_mode_attrs<1>(bytes);
    if (e == cudaSuccess) e = set_mode_attrs<2>(bytes);
    return e;
}

cudaError_t cand_occupancy(int mode, bool route, int block, size_t smem, int *n) {
    if (route)
        return mode == 0 ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_cand<0, kOutLag | kOutMatrix>, block, smem)
                         : cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_cand<1, kOutLag | kOutMatrix>, block, smem);
    return mode == 0 ? cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_cand<0, kOutMatrix>, block, smem)
                     : cudaOccupancyMaxActiveBlocksPerMultiprocessor(n, k_cand<1, kOutMatrix>, block, smem);
}

}  // namespace lr
