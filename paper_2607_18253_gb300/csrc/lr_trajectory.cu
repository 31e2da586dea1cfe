// K1: the query-independent part of the Serving Framework Simulation (Sec. 4.1).
//
// A new query q is appended at the FCFS tail of an instance's waiting queue
// and is served after every resident request in every batch, so it never
// changes what a resident receives.  The residents' trajectory is therefore
// the same for every query, and one warp per instance simulates it once:
//
//   * la  : the first batch whose scheduling leaves the waiting queue empty, a
//           token budget r0 > 0 and fewer than S_j requests running -- the
//           batch that admits any new query (admission is FCFS, Sec. 2);
//   * r_k : the budget left to the query in batch la + k (k >= 1); after la the
//           residents only decode, so r_k = B_j - (decoders in that batch);
//   * the residents' Eq. 9 features summed up to each batch the query's first
//           token can fall in (Eq. 7/8).
//
// The per-candidate kernel then only locates the query's last prefill batch
// among the cumulative budgets and adds the query's own features.
//
// Precondition (checked): at most one running request has remaining prefill
// and it is the last one, and n_run <= S_j.  Then every decoder receives its
// token in every batch (decoders come first and number fewer than B_j), so
// decode progress is lockstep: a request that starts decoding in batch s with
// d tokens to go decodes in batches s..s+d-1 at context cb + l.  The warp
// never touches individual decoders while it steps:
//
//   * every decoder is appended once to a list (s, f, cb); its Eq. 9 decode
//     features up to any batch L follow in closed form, summed over the list
//     by the whole warp after the loop;
//   * a calendar counts decoders by last decode batch f (with a bitmap to find
//     the next non-empty batch); decoders ending beyond the calendar are rare
//     and handled by scanning the list;
//   * the step loop itself -- a chain of dependent scheduling decisions --
//     is scalar code over shared memory (prompt prefix sums, calendar, list)
//     that every lane runs on the same values, with runs of batches that only
//     decode skipped in one step;
//   * where only the sequence cap limits admission (every freed seat is
//     refilled at once), up to 32 end batches are taken in one warp-wide step.
#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;

struct WarpSmem {
    int32_t *cal;    // [kCalendar] decoders by last decode batch
    uint32_t *bm;    // [kCalendar / 32] non-empty calendar batches
    int4 *dl;        // [capR + capW] decoder list: (first decode batch s, last decode
                     //   batch f, context offset cb: context at batch l is cb + l, 0)
    int32_t *P;      // [capW + 2] exclusive prefix sums of waiting prompts (+1 unread pad)
    int32_t *wdec;   // [capW + 1] waiting decode lengths (+1 unread pad)
    int32_t *rcum;   // [kph] cumulative budgets
    int32_t *scr;    // [32] a seat run's request-to-batch map, then the step loop's results
};

__device__ __forceinline__ WarpSmem carve(int32_t *base, const DevConfig &c) {
    WarpSmem w;
    w.cal = base;
    w.bm = reinterpret_cast<uint32_t *>(w.cal + kCalendar);
    w.dl = reinterpret_cast<int4 *>(w.bm + kCalendar / 32);  // 16-byte aligned
    w.P = reinterpret_cast<int32_t *>(w.dl + (c.capR + c.capW));
    w.wdec = w.P + (c.capW + 2);
    w.rcum = w.wdec + (c.capW + 1);
    w.scr = w.rcum + c.kph;
    return w;
}

__device__ void fail(DevCtl *ctl, int code, int lane) {
    if (lane == 0) {
        atomicCAS(&ctl->load_err, 0, code);
        record_status(ctl, code);
    }
}

__device__ __forceinline__ int warp_incl_sum(int x, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
    }
    return x;
}

// Exclusive prefix sum over the warp of values in [0, 63]: one ballot per bit,
// all independent of each other.
__device__ __forceinline__ int warp_excl_sum6(int v, unsigned lt) {
    int r = 0;
#pragma unroll
    for (int b = 0; b < 6; ++b) r += __popc(__ballot_sync(kFull, (v >> b) & 1) & lt) << b;
    return r;
}

// Shared-memory accesses of the step loop by 32-bit shared address: the loop is
// a chain of dependent decisions, so every address computation and every
// generic-to-shared translation sits on its critical path.  The volatile
// statements keep their program order, which the loop relies on.
__device__ __forceinline__ uint32_t saddr(const void *p) { return (uint32_t)__cvta_generic_to_shared(p); }
__device__ __forceinline__ int lds(uint32_t a) {
    int v;
    asm volatile("ld.shared.s32 %0, [%1];" : "=r"(v) : "r"(a));
    return v;
}
__device__ __forceinline__ void red_add(uint32_t a, int v) {
    asm volatile("red.shared.add.s32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ void red_or(uint32_t a, uint32_t v) {
    asm volatile("red.shared.or.b32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}

__device__ __forceinline__ void sts(uint32_t a, int v) {
    asm volatile("st.shared.s32 [%0], %1;" ::"r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ void sts4(uint32_t a, int x, int y, int z, int w) {
    asm volatile("st.shared.v4.s32 [%0], {%1, %2, %3, %4};" ::"r"(a), "r"(x), "r"(y), "r"(z), "r"(w) : "memory");
}
// The same updates taken by the leading lane only, for scalar code that every
// lane of the warp runs on the same values.
__device__ __forceinline__ void red_add_if(bool p, uint32_t a, int v) {
    asm volatile("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %0, 0;\n\t@q red.shared.add.s32 [%1], %2;\n\t}"
                 ::"r"((unsigned)p), "r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ void red_or_if(bool p, uint32_t a, uint32_t v) {
    asm volatile("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %0, 0;\n\t@q red.shared.or.b32 [%1], %2;\n\t}"
                 ::"r"((unsigned)p), "r"(a), "r"(v) : "memory");
}
__device__ __forceinline__ void sts4_if(bool p, uint32_t a, int x, int y, int z, int w) {
    asm volatile("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %0, 0;\n\t@q st.shared.v4.s32 [%1], {%2, %3, %4, %5};\n\t}"
                 ::"r"((unsigned)p), "r"(a), "r"(x), "r"(y), "r"(z), "r"(w) : "memory");
}

// Scalar view of one instance's trajectory state.  The step loop is a chain of
// dependent decisions: every lane runs it as the same scalar code over shared
// memory (loads broadcast), and only the leading lane stores.
struct Track {
    uint32_t cal, bm, dl;       // shared addresses of the calendar, its bitmap and the decoder list
    int nlist;                  // decoders in the list
    unsigned long long words;   // bit w set: calendar word w has a non-empty batch
    int lane;                   // lane 0 stores
    bool lead;

    // Smallest last-decode batch >= L of any decoder; ends beyond the calendar
    // (always later than every calendar end) are found in the list.
    __device__ int next_end(int L) const {
        __syncwarp();  // the leading lane's appends are visible to every lane
        if (L < kCalendar) {
            const int w = L >> 5;
            const uint32_t word = (uint32_t)lds(bm + 4u * w) & (~0u << (L & 31));
            if (word != 0u) return (w << 5) + __ffs(word) - 1;
            const unsigned long long rest = (w + 1 < 64) ? (words & (~0ull << (w + 1))) : 0ull;
            if (rest != 0ull) {
                const int w2 = __ffsll((long long)rest) - 1;
                return (w2 << 5) + __ffs(lds(bm + 4u * w2)) - 1;
            }
        }
        int mn = kBig;  // the lanes split the list
        for (int i = lane; i < nlist; i += 32) {
            const int f = lds(dl + 16u * i + 4u);
            if (f >= L && f < mn) mn = f;
        }
        return __reduce_min_sync(kFull, mn);
    }

    // Number of decoders whose last decode batch is fc.
    __device__ int ends_at(int fc) const {
        __syncwarp();
        if (fc < kCalendar) return lds(cal + 4u * fc);
        int eq = 0;
        for (int i = lane; i < nlist; i += 32) eq += (lds(dl + 16u * i + 4u) == fc) ? 1 : 0;
        return __reduce_add_sync(kFull, eq);
    }

    // A new decoder with first decode batch s and last decode batch f.  The
    // calendar updates are reductions whose results are not returned, so the
    // loop does not wait for a load-modify-store round trip.
    __device__ void append(int s, int f, int cb) {
        sts4_if(lead, dl + 16u * nlist, s, f, cb, 0);
        ++nlist;
        if (f < kCalendar) {
            red_add_if(lead, cal + 4u * f, 1);
            red_or_if(lead, bm + 4u * (f >> 5), 1u << (f & 31));
            words |= 1ull << (f >> 5);
        }
    }
};

// Last decode batch and context offset of a request that finished its prompt in
// batch e with ce tokens of context and d output tokens (Sec. 4.1: the decode
// stage starts after the prefill).  Returns false if it never decodes (first
// token sampled with the last chunk and d == 1).
template <int MODE>
__device__ __forceinline__ bool decoder_of(int e, int ce, int d, int *f, int *cb) {
    *cb = ce - (e + 1);
    *f = e + d - MODE;
    return MODE == 0 || d >= 2;
}

template <int MODE>
__device__ void summarize_instance(const K1Launch &a, const StateBuf &out, int j, int lane, int32_t *wbase) {
    const DevConfig &c = a.cfg;
    const size_t rrow = (size_t)j * c.capR;
    const size_t wrow = (size_t)j * c.capW;
    const int32_t *__restrict__ ic = a.in.run_ctx + rrow;
    const int32_t *__restrict__ ip = a.in.run_pre + rrow;
    const int32_t *__restrict__ id = a.in.run_dec + rrow;
    const int32_t *__restrict__ iwp = a.in.wait_pre + wrow;
    const int32_t *__restrict__ iwd = a.in.wait_dec + wrow;
    // The snapshot rows are read in blocks of 256 entries, all loads of a block issued
    // before any of them is used; the first block's loads go out before anything
    // waits on the counts, so that one memory round trip covers both.
    constexpr int kBlk = 8;  // entries per lane and block
    int xc[kBlk], xp[kBlk], xd[kBlk], yp[kBlk], yd[kBlk];
    auto load_block = [&](int base) {
#pragma unroll
        for (int k = 0; k < kBlk; ++k) {
            const int t = base + lane + 32 * k;
            xc[k] = t < c.capR ? __ldg(ic + t) : 0;
            xp[k] = t < c.capR ? __ldg(ip + t) : 0;
            xd[k] = t < c.capR ? __ldg(id + t) : 0;
            yp[k] = t < c.capW ? __ldg(iwp + t) : 0;
            yd[k] = t < c.capW ? __ldg(iwd + t) : 0;
        }
    };
    load_block(0);
    const int B = c.B[j];
    const int S = c.S[j];
    const int nr = a.in.n_run[j];
    const int nw = a.in.n_wait[j];
    if (lane == 0) {
        out.n_run[j] = nr;
        out.n_wait[j] = nw;
        out.clock[j] = a.in.clock ? a.in.clock[j] : 0.0;
    }
    WarpSmem m = carve(wbase, c);
    // Clear the calendar.
    for (int i = lane; i < kCalendar / 4; i += 32) reinterpret_cast<int4 *>(m.cal)[i] = make_int4(0, 0, 0, 0);
    for (int i = lane; i < kCalendar / 32; i += 32) m.bm[i] = 0u;
    if (!(nr >= 0 && nr <= c.capR && nr <= S && nw >= 0 && nw <= c.capW)) {
        fail(a.ctl, kEState, lane);
        return;
    }
    __syncwarp();

    // Copy the snapshot into library memory, validate it, total the prefill work
    // and list the running decoders (decoding from batch 1).
    bool bad = false;
    long long f1 = 0, f4 = 0, wsum = 0;
    int pf_pre = 0, pf_ctx = 0, pf_dec = 0;
    int32_t *__restrict__ oc = out.run_ctx + rrow;
    int32_t *__restrict__ op = out.run_pre + rrow;
    int32_t *__restrict__ od = out.run_dec + rrow;
    int32_t *__restrict__ owp = out.wait_pre + wrow;
    int32_t *__restrict__ owd = out.wait_dec + wrow;
    for (int base = 0; base < max(c.capR, c.capW); base += 32 * kBlk) {
        if (base > 0) load_block(base);
#pragma unroll
        for (int k = 0; k < kBlk; ++k) {
            const int t = base + lane + 32 * k;
            const int ctx = xc[k], pre = xp[k], dec = xd[k];
            if (t < c.capR) {
                oc[t] = ctx;
                op[t] = pre;
                od[t] = dec;
            }
            if (t < nr) {
                bad |= ctx < 0 || ctx > (1 << 28) || pre < 0 || pre > (1 << 24) || dec < 1 || dec > (1 << 24);
                bad |= pre > 0 && t != nr - 1;
                f1 += pre;
                f4 += (long long)pre * ctx + ((long long)pre * (pre + 1)) / 2;
                if (t == nr - 1) {
                    pf_pre = pre;
                    pf_ctx = ctx;
                    pf_dec = dec;
                }
                if (pre == 0 && !bad) {
                    m.dl[t] = make_int4(1, dec, ctx - 1, 0);
                    if (dec < kCalendar) {
                        atomicAdd(&m.cal[dec], 1);
                        atomicOr(&m.bm[dec >> 5], 1u << (dec & 31));
                    }
                }
            }
        }
#pragma unroll
        for (int k = 0; k < kBlk; ++k) {
            const int t = base + lane + 32 * k;
            if (t >= c.capW) continue;
            const int pre = yp[k], dec = yd[k];
            owp[t] = pre;
            owd[t] = dec;
            m.wdec[t] = dec;
            const bool live = t < nw;
            if (live) {
                bad |= pre < 1 || pre > (1 << 24) || dec < 1 || dec > (1 << 24);
                f1 += pre;
                f4 += ((long long)pre * (pre + 1)) / 2;
                wsum += pre;
            }
            m.P[t + 1] = live ? min(max(pre, 0), 1 << 24) : 0;
        }
    }
    __syncwarp();
    // exclusive prefix sums of the prompts, in place (valid while the total stays below
    // 2^30): each lane sums the consecutive entries it owns, the lane totals are scanned
    // once, and each lane then writes its entries' sums
    {
        const int seg = (c.capW + 31) >> 5;
        const int t0 = lane * seg, t1 = min(t0 + seg, c.capW);
        int own = 0;
        for (int t = t0; t < t1; ++t) own += m.P[t + 1];
        int run = warp_incl_sum(own, lane) - own;
        for (int t = t0; t < t1; ++t) {
            run += m.P[t + 1];
            m.P[t + 1] = run;
        }
        if (lane == 0) m.P[0] = 0;
    }
    wsum = warp_sum64(wsum);
    f1 = warp_sum64(f1);
    f4 = warp_sum64(f4);
    if (__any_sync(kFull, bad) || wsum > (1LL << 30)) {
        fail(a.ctl, kEState, lane);
        return;
    }
    __syncwarp();

    // the request still in prefill, if any, is the last running one
    int pfR = 0, pfC = 0, pfD = 0;
    if (nr > 0) {
        const int src = (nr - 1) & 31;
        pfR = __shfl_sync(kFull, pf_pre, src);
        pfC = __shfl_sync(kFull, pf_ctx, src);
        pfD = __shfl_sync(kFull, pf_dec, src);
    }
    const int n0 = nr - (pfR > 0 ? 1 : 0);

    // non-empty calendar words after the running decoders were entered
    const unsigned long long words0 =
        (unsigned long long)__ballot_sync(kFull, m.bm[lane] != 0u) |
        ((unsigned long long)__ballot_sync(kFull, m.bm[lane + 32] != 0u) << 32);

    // Step the scheduler until a query appended now would be admitted.  Every
    // lane runs the loop on the same values; the whole warp joins in for runs of
    // end batches in which only seats limit admission.
    {
        Track tr;
        tr.cal = saddr(m.cal);
        tr.bm = saddr(m.bm);
        tr.dl = saddr(m.dl);
        tr.nlist = n0;
        tr.words = words0;
        tr.lane = lane;
        tr.lead = lane == 0;
        const uint32_t sP = saddr(m.P), sW = saddr(m.wdec), sE = saddr(m.scr);
        bool pf = pfR > 0;
        int n = n0;  // decoders alive at the start of batch l
        int l = 1, head = 0, iters = 0;
        int ph = 0;  // prompt prefix sum at the waiting head
        int fnext = tr.next_end(1);
        int la = 0, r0 = 0;

        // A seat-limited run.  Precondition: after batch e0 every seat is held by
        // a decoder, no prompt is part-way, and decoders end in batch
        // e0 < kCalendar.  If c_b decoders end in batch b, batch b + 1 then runs
        // S - c_b decoders and admits exactly the next c_b waiting requests, as
        // long as (a) the queue holds them, (b) their prompts fit the budget
        // B - (S - c_b) whole and (c) no request admitted after an earlier batch
        // of the run ends by batch b (in the first-token-on-prefill mode a
        // one-token request ends in its prefill batch, so (c) excludes those
        // too); batches in which no decoder ends admit nobody.  Lane k takes
        // batch e0 + k, lane i the i-th request admitted in the run (32 at most).
        // The run moves to the last batch e0 + K with ends before the first that
        // breaks (a)-(c): the admissions after batches e0 .. e0 + K - 1 are
        // appended in FCFS order, and the scalar step takes those of batch
        // e0 + K + 1.  Returns false if there is no such K > 0.
        auto seat_run = [&](int e0) -> bool {
            __syncwarp();
            const unsigned lt = (1u << lane) - 1u;
            // waiting request head + lane: its decode length and the prompt sum through it
            const int rq = head + lane;
            const int dq = rq < nw ? lds(sW + 4u * rq) : 0;
            const int pq = rq < nw ? lds(sP + 4u * (rq + 1)) : 0;
            const bool incal = e0 + lane < kCalendar;
            const int ck = incal ? lds(tr.cal + 4u * (e0 + lane)) : 0;
            const int cc = min(ck, 33);                 // more than 32 never fit the lanes
            const int x0 = warp_excl_sum6(cc, lt);      // requests admitted before batch e0 + k + 1
            const int x1 = x0 + cc;
            const int phi = __shfl_sync(kFull, pq, (x1 - 1) & 31);  // prompt sums at the ends
            const int plo = __shfl_sync(kFull, pq, (x0 - 1) & 31);
            const bool ok = incal && (ck == 0 || (x1 <= 32 && head + x1 <= nw &&
                                                  (x1 > 0 ? phi : ph) - (x0 > 0 ? plo : ph) <= B - (S - ck)));
            const unsigned bad = __ballot_sync(kFull, !ok);
            const unsigned em = __ballot_sync(kFull, ck > 0);  // batches with ends (lane 0 among them)
            const int kmax = min(bad ? __ffs(bad) - 1 : 32, 31);  // (a) and (b) hold below it
            if (kmax <= 0 || (em & ((2u << kmax) - 1u) & ~1u) == 0u) return false;
            // request lane i: the lane of its batch (the run's request starts, by rank) and its last batch
            const int nreq = __shfl_sync(kFull, x0, kmax);
            // each batch lane below kmax writes its index into its requests' slots (those
            // requests fit the 32 lanes: x1 <= 32), and request lane i reads slot i
            if (lane < kmax)
                for (int t = x0; t < x1; ++t) sts(sE + 4u * t, lane);
            __syncwarp();
            const int kq = lane < nreq ? lds(sE + 4u * lane) : 0;
            const int fi = lane < nreq ? e0 + kq + 1 + dq - MODE : kBig;
            // (c): a request of lane kq ending in batch f rules out every K > kq with e0 + K >= f
            int K = kmax;
            for (unsigned sh = __ballot_sync(kFull, fi <= e0 + kmax); sh != 0u; sh &= sh - 1u) {
                const int i = __ffs(sh) - 1;
                const int f = __shfl_sync(kFull, fi, i);
                K = min(K, max(__shfl_sync(kFull, kq, i) + 1, f - e0) - 1);
            }
            if (K <= 0) return false;
            const unsigned cand = em & ((2u << K) - 1u) & ~1u;
            if (cand == 0u) return false;
            K = 31 - __clz(cand);
            // every request admitted in the run decodes: (c) excludes the one-token ones
            const int taken = __shfl_sync(kFull, x0, K);  // >= c_e0 >= 1
            int pprev = __shfl_up_sync(kFull, pq, 1);
            if (lane == 0) pprev = ph;
            unsigned wlo = 0u, whi = 0u;
            int fmin = kBig;
            if (lane < taken) {
                const int e = e0 + kq;  // the admission batch is e + 1
                fmin = fi;
                sts4(tr.dl + 16u * (tr.nlist + lane), e + 2, fi, pq - pprev - (e + 2), 0);
                if (fi < kCalendar) {
                    red_add(tr.cal + 4u * fi, 1);
                    red_or(tr.bm + 4u * (fi >> 5), 1u << (fi & 31));
                    if (fi < kCalendar / 2) wlo |= 1u << (fi >> 5);
                    else whi |= 1u << ((fi >> 5) - 32);
                }
            }
            tr.words |= ((unsigned long long)__reduce_or_sync(kFull, whi) << 32) | __reduce_or_sync(kFull, wlo);
            const int fK = __reduce_min_sync(kFull, fmin);  // > e0 + K
            const int cK = __shfl_sync(kFull, ck, K);
            const int pK = __shfl_sync(kFull, pq, taken - 1);
            const unsigned later = em & ~((2u << K) - 1u);  // end batches after e0 + K in the window
            __syncwarp();  // the appended decoders are visible to every lane
            tr.nlist += taken;
            head += taken;
            ph = pK;
            n = S - cK;
            l = e0 + K + 1;
            fnext = later ? min(e0 + __ffs(later) - 1, fK) : tr.next_end(l);
            return true;
        };

        // A window of up to 32 batches l .. l + 31 stepped without touching shared memory
        // per batch, while only the token budget and free sequence slots limit admission.
        // In FCFS order the prefill tokens form one stream: the carried prefill, then the
        // waiting prompts.  Batch b serves its decoders one token each and gives the stream
        // min(B - n_b, the end of the last prompt a free sequence slot lets start); the
        // prompts completed in batch b become decoders from b + 1; n_{b+1} = n_b + (new
        // decoders) - (decoders ending in batch b: the calendar's and those created in
        // this window).  Lane k holds stream entry k (start, end, context at completion,
        // decode length, completion batch) and lane w the calendar count of batch l + w;
        // each batch is a few ballots and shuffles, one shuffle and one ballot on the
        // chain from n_b to n_{b+1}.  The window stops before a batch with every slot taken
        // by decoders (the seat-limited path takes those), one that would need an entry
        // beyond the lanes, one at or past the calendar's end, one in which the queue could
        // run out (the admission batch is the scalar step's), or after 32 batches.
        // Returns the batches taken (0: none).
        auto window = [&]() -> int {
            __syncwarp();  // the leading lane's appends are visible to every lane
            const int pfo = pf ? 1 : 0;
            const int base = pf ? pfR : 0;
            const int q = head + lane - pfo;  // waiting request of this lane's entry
            bool valid;
            int st0, en, ce, d;
            if (pf && lane == 0) {
                valid = true;
                st0 = -1;
                en = pfR;
                ce = pfC + pfR;
                d = pfD;
            } else {
                valid = q < nw;
                const int a0 = valid ? lds(sP + 4u * q) : 0;
                const int a1 = valid ? lds(sP + 4u * (q + 1)) : 0;
                st0 = base + a0 - ph;
                en = valid ? base + a1 - ph : kBig;
                ce = a1 - a0;
                d = valid ? lds(sW + 4u * q) : 0;
            }
            const bool dc = valid && (MODE == 0 || d >= 2);  // becomes a decoder when it completes
            const int fl0 = d - MODE;                        // last decode batch - completion batch
            const unsigned dcm = __ballot_sync(kFull, dc);
            const int nent = __popc(__ballot_sync(kFull, valid));
            const int last_end = __shfl_sync(kFull, en, max(nent - 1, 0));
            const int total_left = base + lds(sP + 4u * nw) - ph;
            const int lb = l + lane;
            const int calw = lb < kCalendar ? lds(tr.cal + 4u * lb) : -1;
            const unsigned calok = __ballot_sync(kFull, calw >= 0);
            int T = 0, nn = n, w = 0, ndone = 0;
            bool ip = pf;            // a prompt is part-way at the start of the batch
            int dn = -1, fl = kBig;  // this lane's completion batch and last decode batch
            while (w < 32 && ((calok >> w) & 1u)) {
                const int lw = l + w;
                // decoders ending in batch lw: the calendar's and this window's (off the chain)
                const int ecal = __shfl_sync(kFull, calw, w);
                const int ewin = __popc(__ballot_sync(kFull, dn >= 0 && fl == lw) & dcm);
                const int freeseats = S - nn - (ip ? 1 : 0);
                if (freeseats <= 0 && !ip) break;  // every slot holds a decoder
                const int budget = B - nn;
                if (budget <= 0) break;
                int T2 = T + budget;
                if (T2 >= total_left) break;  // the queue could run out in this batch
                if (freeseats > 0) {
                    const int kl = ndone + (ip ? 1 : 0) + freeseats - 1;  // last entry a free slot lets start
                    const int lim = __shfl_sync(kFull, en, min(kl, 31));
                    if (kl < nent) T2 = min(T2, lim);
                    else if (T2 > last_end) break;  // beyond the lanes
                } else {
                    T2 = min(T2, __shfl_sync(kFull, en, ndone & 31));  // only the prefill in progress advances
                }
                const bool nd = valid && dn < 0 && en <= T2;
                if (nd) {
                    dn = lw;
                    fl = lw + fl0;
                }
                const unsigned ndm = __ballot_sync(kFull, nd);
                ip = __ballot_sync(kFull, valid && st0 < T2 && T2 < en) != 0u;
                ndone += __popc(ndm);
                nn += __popc(ndm & dcm) - ecal - ewin;
                T = T2;
                ++w;
            }
            if (w == 0) return 0;
            // the window's new decoders, in completion (stream) order
            const bool ap = dn >= 0 && dc;
            const unsigned apm = __ballot_sync(kFull, ap);
            unsigned wlo = 0u, whi = 0u;
            if (ap) {
                sts4(tr.dl + 16u * (tr.nlist + __popc(apm & lanemask_lt())), dn + 1, fl, ce - (dn + 1), 0);
                if (fl < kCalendar) {
                    red_add(tr.cal + 4u * fl, 1);
                    red_or(tr.bm + 4u * (fl >> 5), 1u << (fl & 31));
                    if (fl < kCalendar / 2) wlo |= 1u << (fl >> 5);
                    else whi |= 1u << ((fl >> 5) - 32);
                }
            }
            tr.words |= ((unsigned long long)__reduce_or_sync(kFull, whi) << 32) | __reduce_or_sync(kFull, wlo);
            tr.nlist += __popc(apm);
            // the new stream position: started prompts leave the queue; the entry in progress
            // at T, if any, is the prefill carried into batch l + w
            head += __popc(__ballot_sync(kFull, valid && lane >= pfo && st0 < T));
            ph = lds(sP + 4u * head);
            const int snd = __shfl_sync(kFull, st0, ndone & 31);
            const int end_nd = __shfl_sync(kFull, en, ndone & 31);
            const int ce_nd = __shfl_sync(kFull, ce, ndone & 31);
            const int d_nd = __shfl_sync(kFull, d, ndone & 31);
            if (ndone < nent && snd < T) {
                pf = true;
                pfR = end_nd - T;
                pfC = ce_nd - pfR;
                pfD = d_nd;
            } else {
                pf = false;
            }
            n = nn;
            // the next end: the calendar's within the lanes' batches, or one of the window's
            // new decoders, else a search
            const unsigned cm = __ballot_sync(kFull, calw > 0) & (w < 32 ? (~0u << w) : 0u);
            const int fc = cm ? l + __ffs(cm) - 1 : kBig;
            const int fm = __reduce_min_sync(kFull, (ap && fl >= l + w) ? fl : kBig);
            l += w;
            fnext = (fc < kBig) ? min(fc, fm) : tr.next_end(l);
            return w;
        };

        while (iters < c.max_iters && l < (1 << 30)) {
            ++iters;
            int cnt = n + (pf ? 1 : 0);  // requests running in batch l
            if (pf || cnt < S) {
                const int wt = window();  // every batch of a window counts against max_iters
                if (wt > 0) {
                    iters += wt - 1;
                    continue;
                }
            }
            if (!pf && cnt >= S) {
                // Every sequence slot is taken: nothing but decoding until one frees.
                if (fnext == kBig) break;  // excluded: a decoder is running
                if (fnext < kCalendar && seat_run(fnext)) continue;
                n -= tr.ends_at(fnext);
                l = fnext + 1;
                fnext = tr.next_end(l);
                continue;
            }
            int budget = B - n;  // every decoder takes one token first
            const int nl0 = tr.nlist;  // decoders appended in this batch start in batch l + 1
            if (pf) {
                if (budget <= 0) break;  // excluded by the preconditions
                if (pfR > budget) {
                    // The prefill continues; skip the batches in which it cannot
                    // finish and the number of decoders stays the same.
                    const int step = min((pfR - 1) / budget, fnext == kBig ? kBig : fnext + 1 - l);
                    pfR -= step * budget;
                    pfC += step * budget;
                    l += step;
                    if (l - 1 == fnext) {
                        n -= tr.ends_at(fnext);
                        fnext = tr.next_end(l);
                    }
                    continue;
                }
                budget -= pfR;
                pfC += pfR;
                pf = false;
                int f, cb;
                if (decoder_of<MODE>(l, pfC, pfD, &f, &cb)) {
                    tr.append(l + 1, f, cb);
                    fnext = min(fnext, f);
                }
            }
            // FCFS admission while budget and a sequence slot remain, up to 32
            // requests at a time: the prompt prefix sums increase, so the requests
            // that fit whole are a prefix of the queue (lane i tests head + i).
            const int lim = min(nw, head + (S - cnt));  // the queue and the free seats
            const int head0 = head;
            while (budget > 0 && head < lim) {
                const int r = head + lane;
                const int pe = r < lim ? lds(sP + 4u * (r + 1)) : 0;  // prompt sum through request r
                const int dr = r < lim ? lds(sW + 4u * r) : 0;        // and its decode length
                const bool whole = r < lim && pe - ph <= budget;
                const int k = __popc(__ballot_sync(kFull, whole));
                if (k > 0) {
                    int before = __shfl_up_sync(kFull, pe, 1);
                    if (lane == 0) before = ph;
                    int f = kBig, cb = 0;
                    const bool dec = whole && decoder_of<MODE>(l, pe - before, dr, &f, &cb);
                    const unsigned dm = __ballot_sync(kFull, dec);
                    unsigned wlo = 0u, whi = 0u;
                    if (dec) {
                        sts4(tr.dl + 16u * (tr.nlist + __popc(dm & lanemask_lt())), l + 1, f, cb, 0);
                        if (f < kCalendar) {
                            red_add(tr.cal + 4u * f, 1);
                            red_or(tr.bm + 4u * (f >> 5), 1u << (f & 31));
                            if (f < kCalendar / 2) wlo |= 1u << (f >> 5);
                            else whi |= 1u << ((f >> 5) - 32);
                        }
                    }
                    tr.words |= ((unsigned long long)__reduce_or_sync(kFull, whi) << 32) | __reduce_or_sync(kFull, wlo);
                    fnext = min(fnext, __reduce_min_sync(kFull, f));
                    tr.nlist += __popc(dm);
                    const int pk = __shfl_sync(kFull, pe, k - 1);
                    budget -= pk - ph;
                    ph = pk;
                    head += k;
                }
                if (k < 32 && budget > 0 && head < lim) {
                    // the next prompt does not fit whole: it continues in later batches
                    const int pn = lds(sP + 4u * (head + 1));
                    pf = true;
                    pfR = pn - ph - budget;
                    pfC = budget;
                    pfD = lds(sW + 4u * head);
                    budget = 0;
                    ++head;
                    ph = pn;
                }
            }
            cnt += head - head0;  // every request taken from the queue holds a seat
            if (!pf && head == nw && budget > 0 && cnt < S) {
                la = l;
                r0 = budget;
                break;
            }
            n += tr.nlist - nl0;
            if (l == fnext) {
                // all seats held by decoders after this batch: a seat-limited run may follow
                if (!pf && n == S && fnext < kCalendar && seat_run(l)) continue;
                n -= tr.ends_at(l);
                fnext = tr.next_end(l + 1);
            }
            ++l;
        }
        __syncwarp();  // the run's scratch is read before it is overwritten
        if (lane == 0) {
            m.scr[0] = la;
            m.scr[1] = r0;
            m.scr[2] = tr.nlist;
            m.scr[3] = iters;
        }
    }
    __syncwarp();
    const int la = m.scr[0];
    const int r0 = m.scr[1];
    const int iters = m.scr[3];  // simulation steps taken
    (void)iters;
    if (la == 0) {
        fail(a.ctl, kETraj, lane);
        return;
    }
    struct {
        int nlist;
    } sim = {m.scr[2]};

    // Budgets left to the query after its admission batch, and the residents' decode
    // features up to each batch its first token can fall in.  One pass over the
    // decoder list serves eight table rows k: the decoders alive in batch la + k (so
    // r_k = B - alive) and the decode tokens and context they contribute up to batch
    // L_k = la + k + off.  A decoder alive over the whole window of a pass adds to
    // row q in closed form (u + q tokens, and context sum up to L_0 plus
    // q cb + q L_0 + q(q+1)/2, with u its tokens up to L_0), so only decoders that
    // start or end inside the window take the per-row loop (one finished before it
    // adds the same to every row).  Lane partials are
    // reduced through shared memory (the calendar is free after the step loop).
    constexpr int off = (MODE == 0) ? 1 : 0;
    constexpr int kRows = 8;
    constexpr int kCols = 3 * kRows + 4;  // per-row partials of window decoders, then N, A2, A3, CB
    const int nl = sim.nlist;
    long long *red = reinterpret_cast<long long *>(m.cal);  // [kCols][32] lane partials (7 KB)
    // after them, up to the end of the calendar bitmap: the window decoders' indices
    constexpr int kWinList = (int)((kCalendar * 4 + kCalendar / 8 - kCols * 32 * 8) / 4);
    int32_t *wlist = reinterpret_cast<int32_t *>(red + kCols * 32);
    const int m_j = c.moi[j];
    const float b0 = c.coef[m_j * 5 + 0];
    const float b1d = c.coef[m_j * 5 + 2];
    const long long ppmax = ((long long)c.pmax * (c.pmax + 1)) / 2;
    bool fast = (f1 + c.pmax < kFastLimit) && (f4 + ppmax < kFastLimit);
    bool compact = true;  // every F3_k + pmax below 2^31 (first token in its own batch)
    const long long lowmask = (1LL << kSplitBits) - 1;
    int kp = 0;          // table rows kept
    long long rc = r0;   // cumulative budget R_k
    bool more = true;
    for (int k0 = 0; more && k0 < c.kph; k0 += kRows) {
        const int lk0 = la + k0;             // first batch of the alive counts
        const int L0 = lk0 + off;            // first feature horizon
        const int Lend = lk0 + kRows - 1 + off;
        int nd[kRows];
        long long a2[kRows], a3[kRows];
#pragma unroll
        for (int q = 0; q < kRows; ++q) {
            nd[q] = 0;
            a2[q] = 0;
            a3[q] = 0;
        }
        int nreg = 0;                        // decoders alive over the whole window
        long long A2 = 0, A3 = 0, CB = 0;    // their tokens and context sums up to L0 (plus those of
                                             // decoders finished before the window), and their cb sum
        // a decoder that starts or ends inside the window adds to each row separately
        auto rows = [&](const int4 dd) {
            const int s = dd.x;
#pragma unroll
            for (int q = 0; q < kRows; ++q) {
                const int lk = lk0 + q;
                nd[q] += (s <= lk && lk <= dd.y) ? 1 : 0;
                const int L = lk + off;
                if (s <= L) {
                    const int e = min(dd.y, L);
                    const long long cnt = (long long)e - s + 1;
                    a2[q] += cnt;
                    a3[q] += cnt * (long long)dd.z + (((long long)s + e) * cnt) / 2;
                }
            }
        };
        // Window decoders are few but scattered, so they are first gathered into a
        // list (stable ballot compaction) and then taken 32 at a time: a warp would
        // otherwise run the per-row path in almost every step over the list.  Each
        // lane classifies two decoders per step, loaded together.
        // Branch-free: a decoder alive over the whole window contributes its tokens up to
        // L0, one finished before it all of its tokens; both are the same closed form
        // (u tokens at contexts cb + s .. cb + e: u cb + (s + e) u / 2, where (s + e) u
        // is twice a sum of consecutive integers, so the halving is exact).
        auto classify = [&](const int4 dd) -> bool {
            const int s = dd.x;
            const bool reg = s <= lk0 && dd.y >= Lend;
            const bool fin = dd.y < lk0;
            const int e = reg ? L0 : dd.y;
            const int u = (reg || fin) ? e - s + 1 : 0;
            nreg += reg ? 1 : 0;
            A2 += u;
            A3 += (long long)u * dd.z + (((long long)s + e) * u >> 1);
            CB += reg ? dd.z : 0;
            return !(reg || fin);
        };
        const unsigned lt = lanemask_lt();
        int nwin = 0;
        for (int base = 0; base < nl; base += 64) {
            const int i0 = base + lane, i1 = i0 + 32;
            const int4 d0 = m.dl[min(i0, nl - 1)], d1 = m.dl[min(i1, nl - 1)];
            const bool w0 = i0 < nl && classify(d0);
            const bool w1 = i1 < nl && classify(d1);
            const unsigned b0 = __ballot_sync(kFull, w0), b1 = __ballot_sync(kFull, w1);
            const int s0 = nwin + __popc(b0 & lt), s1 = nwin + __popc(b0) + __popc(b1 & lt);
            if (w0 && s0 < kWinList) wlist[s0] = i0;
            if (w1 && s1 < kWinList) wlist[s1] = i1;
            nwin += __popc(b0) + __popc(b1);
        }
        if (nwin > kWinList) {
            // the list is full: the window decoders beyond it take the per-row path here
            // (the same compaction finds them again, without accumulating anything)
            int seen = 0;
            for (int base = 0; base < nl; base += 32) {
                const int i = base + lane;
                bool win = false;
                if (i < nl) {
                    const int4 dd = m.dl[i];
                    win = !(dd.x <= lk0 && dd.y >= Lend) && !(dd.y < lk0);
                }
                const unsigned bal = __ballot_sync(kFull, win);
                if (win && seen + __popc(bal & lt) >= kWinList) rows(m.dl[i]);
                seen += __popc(bal);
            }
        }
        __syncwarp();
        for (int t = lane; t < min(nwin, kWinList); t += 32) rows(m.dl[wlist[t]]);
        __syncwarp();
#pragma unroll
        for (int q = 0; q < kRows; ++q) {
            red[(0 * kRows + q) * 32 + lane] = nd[q];
            red[(1 * kRows + q) * 32 + lane] = a2[q];
            red[(2 * kRows + q) * 32 + lane] = a3[q];
        }
        red[(3 * kRows + 0) * 32 + lane] = nreg;
        red[(3 * kRows + 1) * 32 + lane] = A2;
        red[(3 * kRows + 2) * 32 + lane] = A3;
        red[(3 * kRows + 3) * 32 + lane] = CB;
        __syncwarp();
        // lane c sums column c, starting at its own offset so that the 28 lanes read
        // different banks (a column's 32 partials share one bank group), with four
        // independent partial sums
        long long tot = 0;
        if (lane < kCols) {
            long long t4[4] = {0, 0, 0, 0};
#pragma unroll
            for (int l = 0; l < 32; ++l) t4[l & 3] += red[lane * 32 + ((l + lane) & 31)];
            tot = (t4[0] + t4[1]) + (t4[2] + t4[3]);
        }
        __syncwarp();
        if (lane < kCols) red[lane * 32] = tot;  // each column's head holds its sum
        __syncwarp();
        const long long Nw = red[(3 * kRows + 0) * 32], A2w = red[(3 * kRows + 1) * 32];
        const long long A3w = red[(3 * kRows + 2) * 32], CBw = red[(3 * kRows + 3) * 32];
        // the rows of this pass in order; row k >= 1 is needed while R_{k-1} < pmax
        for (int q = 0; q < kRows && more; ++q) {
            const int k = k0 + q;
            if (k >= c.kph || (k >= 1 && rc >= c.pmax)) {
                more = false;
                break;
            }
            if (k >= 1) rc += B - (Nw + red[(0 * kRows + q) * 32]);
            const int rk = (int)min(rc, (long long)kBig - 1);
            if (lane == 0) m.rcum[k] = rk;
            kp = k + 1;
            const int L = la + k + off;
            // + the query's own first decode token
            const long long F2 = A2w + Nw * q + red[(1 * kRows + q) * 32] + off;
            const long long F3 = A3w + q * CBw + Nw * ((long long)q * L0 + (long long)q * (q + 1) / 2) +
                                 red[(2 * kRows + q) * 32];
            fast = fast && (F3 + c.pmax < kFastLimit);
            compact = compact && (MODE == 1 || F3 + c.pmax < (1LL << 31));
            if (lane == (k & 31)) {
                const float t = __fmaf_rn(b1d, __ll2float_rn(F2), __fmul_rn(b0, __int2float_rn(L)));
                const long long lo = F3 & lowmask;
                // entA: (T_k, X_k); entB: (H3_k, L3_k)
                const int x = MODE == 1 ? __float_as_int(__ll2float_rn(F3))
                                        : (F3 + c.pmax < (1LL << 31) ? (int)F3 : 0);
                const size_t slot = (size_t)k * 4 * c.tgp + tile_col(c, j);
                unsigned char *tb = out.tile + tile_base(c, j);
                reinterpret_cast<float2 *>(tb)[slot] = make_float2(t, __int_as_float(x));
                reinterpret_cast<float2 *>(tb + tile_enta_bytes(c))[slot] =
                    make_float2(__ll2float_rn(F3 - lo), __ll2float_rn(lo));
                const size_t o = (size_t)k * c.I + j;
                out.f2[o] = F2;
                out.f3[o] = F3;
                out.rcum[o] = rk;
            }
        }
        __syncwarp();
    }
    if (rc < c.pmax) {
        fail(a.ctl, kETraj, lane);
        return;
    }

    // Prompt-length buckets of width 2^shift <= B_j - S_j + 1 <= every r_k (k >= 1):
    // each holds at most one boundary, so k*(p) = below[b] + (p > boundary[b]).
    const int sh = c.shift[j];
    const int nb = c.nb[j];
    for (int b = lane; b < nb; b += 32) {
        const long long lo = (long long)b << sh;
        const long long hi = lo + (1LL << sh) - 1;
        int below = 0, bnd = kBig;
        for (int k = 0; k < kp; ++k) {
            const long long rk = m.rcum[k];
            if (rk < lo) ++below;
            else if (rk <= hi) bnd = (int)rk;
        }
        out.bkt[(size_t)b * c.I + j] = make_int2(bnd, below);
        // packed word: a boundary at or above kBktNone (> every allowed prompt, 2^20) reads
        // as none; below is at most kKMax < 128
        reinterpret_cast<uint32_t *>(out.tile + tile_base(c, j) + tile_ent_bytes(c))[(size_t)b * 4 * c.tgp +
                                                                                   j % (4 * c.tgp)] =
            (min((uint32_t)bnd, kBktNone) << 7) | (uint32_t)below;
    }
    if (lane == 0) {
        InstParams ip;
        ip.la = la;
        ip.kp = kp;
        ip.shift = sh;
        ip.fast = fast ? 1 : 0;
        ip.f1tot = f1;
        ip.f4tot = f4;
        ip.h1 = __ll2float_rn(f1 - (f1 & lowmask));
        ip.l1 = __ll2float_rn(f1 & lowmask);
        ip.h4 = __ll2float_rn(f4 - (f4 & lowmask));
        ip.l4 = __ll2float_rn(f4 & lowmask);
        ip.r0 = r0;
        ip.pad[0] = ip.pad[1] = ip.pad[2] = 0;
        out.inst[j] = ip;
        // the candidate kernel's per-instance scalars
        int32_t *sc = reinterpret_cast<int32_t *>(out.tile + tile_base(c, j) + tile_ent_bytes(c) + tile_bkt_bytes(c)) +
                      tile_col(c, j);
        const size_t fs = 4 * (size_t)c.tgp;  // field stride
        const float *cf = c.coef + 5 * m_j;
        sc[kScShift * fs] = sh;
        sc[kScH1 * fs] = __float_as_int(ip.h1);
        sc[kScL1 * fs] = __float_as_int(ip.l1);
        sc[kScH4 * fs] = __float_as_int(ip.h4);
        sc[kScL4 * fs] = __float_as_int(ip.l4);
        sc[kScB1p * fs] = __float_as_int(cf[1]);
        sc[kScB2 * fs] = __float_as_int(cf[3]);
        sc[kScB3 * fs] = __float_as_int(cf[4]);
        sc[kScModel * fs] = m_j;
        sc[kScLa * fs] = la;
        sc[kScFast * fs] = ip.fast;
        sc[kScCompact * fs] = (fast && compact) ? 1 : 0;
    }
}

template <int MODE>
__global__ void __launch_bounds__(kK1Warps * 32) k_trajectory(const K1Launch a) {
    extern __shared__ __align__(16) int32_t k1_smem[];
    const int lane = threadIdx.x & 31;
    const int wid = threadIdx.x >> 5;
    const int j = blockIdx.x * kK1Warps + wid;
    // one read of the live-buffer index per CTA (every thread reading the same word
    // would queue them all on one L2 line)
    __shared__ int s_active;
    if (threadIdx.x == 0) s_active = load_acquire(&a.ctl->active);
    __syncthreads();
    const int active = s_active;
    const int dst = (active == 0) ? 1 : 0;
    const StateBuf out = dst ? a.buf1 : a.buf0;
    const size_t per_warp = trajectory_smem_per_warp(a.cfg) / sizeof(int32_t);
    if (j < a.cfg.I) summarize_instance<MODE>(a, out, j, lane, k1_smem + wid * per_warp);

    // The last CTA to finish publishes the new snapshot if every instance succeeded.
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const unsigned prev = atomicAdd(&a.ctl->done_ctas, 1u);
        if (prev == gridDim.x - 1) {
            __threadfence();
            const int err = atomicExch(&a.ctl->load_err, 0);
            if (err == 0) publish_live(a.ctl, dst);
            atomicExch(&a.ctl->done_ctas, 0u);
            __threadfence();
        }
    }
}

}  // namespace

namespace {

// Padding columns of the last tile: no boundary in any bucket, zero tables, an
// exact ("fast", compact) instance of model 0, and a bucket shift of 30 so that every
// allowed prompt (at most 2^20 tokens) looks up bucket 0 and entry 0.
__global__ void k_tile_pad(const DevConfig c, unsigned char *tile) {
    const int first = c.I;
    const int last = tile_count(c) * 4 * c.tgp;
    for (int j = first + blockIdx.x * blockDim.x + threadIdx.x; j < last; j += gridDim.x * blockDim.x) {
        unsigned char *base = tile + tile_base(c, j);
        const int col = tile_col(c, j);
        for (int k = 0; k < c.kph; ++k) {
            reinterpret_cast<float2 *>(base)[(size_t)k * 4 * c.tgp + col] = make_float2(0.f, 0.f);
            reinterpret_cast<float2 *>(base + tile_enta_bytes(c))[(size_t)k * 4 * c.tgp + col] = make_float2(0.f, 0.f);
        }
        for (int b = 0; b < c.nbh; ++b)
            reinterpret_cast<uint32_t *>(base + tile_ent_bytes(c))[(size_t)b * 4 * c.tgp + j % (4 * c.tgp)] =
                kBktNone << 7;
        int32_t *sc = reinterpret_cast<int32_t *>(base + tile_ent_bytes(c) + tile_bkt_bytes(c)) + col;
        for (int f = 0; f < kScal; ++f)
            sc[(size_t)f * 4 * c.tgp] = (f == kScFast || f == kScCompact) ? 1 : (f == kScShift) ? 30 : 0;
    }
}

}  // namespace

cudaError_t launch_tile_pad(const DevConfig &c, unsigned char *tile, cudaStream_t st) {
    k_tile_pad<<<1, 256, 0, st>>>(c, tile);
    return cudaGetLastError();
}

cudaError_t launch_trajectory(const K1Launch &a, int grid, int block, size_t smem, cudaStream_t st) {
    if (a.cfg.mode == 0) k_trajectory<0><<<grid, block, smem, st>>>(a);
    else k_trajectory<1><<<grid, block, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t set_k1_smem(size_t bytes) {
    cudaError_t e = cudaFuncSetAttribute(k_trajectory<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_trajectory<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    return e;
}

}  // namespace lr
