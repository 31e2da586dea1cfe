// K3: online stream step (Sec. 5: queries arrive by a Poisson process and are
// routed as they come; App. F: every instance keeps executing token batches
// and publishes its state after each one).
//
// One warp per instance: the queries routed to it join its waiting tail in
// query order (a stable ballot compaction over the assignment vector), then
// the instance executes whole token batches -- the same scheduler step the
// estimator simulates -- as long as each ends by t_now.  Each batch takes the
// Eq. 9 time of its own composition, evaluated in the same fp32 order as the
// estimate and accumulated into an fp64 clock.  An instance with nothing to
// run jumps to t_now.  The advanced snapshot goes to a scratch buffer, which
// K1 then summarizes and publishes like any snapshot.
//
// Unlike K1 this kernel does not rely on decode being lockstep: every batch
// serves the running list in order with a prefix sum of the token needs, so
// any list (including prefills ahead of decoders) advances exactly.
//
// Under KV-cache limits a second kernel (k_advance_kv) executes the KV step rule
// and hands its snapshot to the KV load instead of K1.
#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ long long warp_incl_sum64(long long x, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
    }
    return x;
}

__device__ void fail3(DevCtl *ctl, int code, int lane) {
    if (lane == 0) {
        atomicCAS(&ctl->load_err, 0, code);
        record_status(ctl, code);
    }
}

// First-token tracking (Sec. 4.1: the TTFT ends with the first output token; Eq. 4
// scores the realized TTFT): a tracked request (id >= 0) that emits its first output
// token in an executed batch -- its first decode token, or the token sampled with its
// last prompt chunk in that mode -- records the batch's end time and drops its id.
__device__ __forceinline__ int emit_first(const K3Launch &a, int id, bool emitted, double t_end) {
    if (emitted && id >= 0) {
        a.ftt[id] = t_end;
        return -1;
    }
    return id;
}

// src: the live snapshot; idst: the buffer K1 publishes next (it receives the ids)
__device__ void advance_instance(const K3Launch &a, const StateBuf &src, const StateBuf &idst, int j, int lane,
                                 int32_t *wbase) {
    const DevConfig &c = a.cfg;
    const StateBuf &dst = a.scratch;
    const int B = c.B[j];
    const int S = c.S[j];
    const int capR = c.capR, capW = c.capW;
    int32_t *rc0 = wbase, *rp0 = rc0 + capR, *rd0 = rp0 + capR;
    int32_t *rc1 = rd0 + capR, *rp1 = rc1 + capR, *rd1 = rp1 + capR;
    int32_t *wp = rd1 + capR, *wd = wp + capW;
    int32_t *ri0 = wd + capW, *ri1 = ri0 + capR, *wi = ri1 + capR;  // ids (tracking only)
    const bool track = a.track != 0;
    const size_t rrow = (size_t)j * capR, wrow = (size_t)j * capW;
    int nr = src.n_run[j];
    int nw = src.n_wait[j];
    for (int t = lane; t < nr; t += 32) {
        rc0[t] = src.run_ctx[rrow + t];
        rp0[t] = src.run_pre[rrow + t];
        rd0[t] = src.run_dec[rrow + t];
        if (track) ri0[t] = src.run_id[rrow + t];
    }
    for (int t = lane; t < nw; t += 32) {
        wp[t] = src.wait_pre[wrow + t];
        wd[t] = src.wait_dec[wrow + t];
        if (track) wi[t] = src.wait_id[wrow + t];
    }
    // routed queries join the waiting tail in query order
    for (int base = 0; base < a.Q; base += 32) {
        const int i = base + lane;
        const bool mine = i < a.Q && a.assign[i] == j;
        const unsigned bal = __ballot_sync(kFull, mine);
        if (mine) {
            const int pos = nw + __popc(bal & lanemask_lt());
            if (pos < capW) {
                wp[pos] = a.prompt[i];
                wd[pos] = a.dec[(size_t)i * a.dec_cols + (a.dec_cols == 1 ? 0 : c.moi[j])];
                if (track) wi[pos] = a.id_base >= 0 ? (int)(a.id_base + i) : -1;
            }
        }
        nw += __popc(bal);
    }
    const bool over = nw > capW;
    bool bad = false;
    for (int t = lane; t < min(nw, capW); t += 32)
        bad |= wp[t] < 1 || wp[t] > (1 << 24) || wd[t] < 1 || wd[t] > (1 << 24);
    if (over) {
        fail3(a.ctl, kECapacity, lane);
        return;
    }
    if (__any_sync(kFull, bad)) {
        fail3(a.ctl, kEInval, lane);
        return;
    }
    __syncwarp();

    const float *cf = c.coef + 5 * c.moi[j];
    const float b0 = cf[0], b1p = cf[1], b1d = cf[2], b2 = cf[3], b3 = cf[4];
    double t = src.clock[j];
    int wh = 0, iters = 0;
    bool ok = true;
    int32_t *rc = rc0, *rp = rp0, *rd = rd0, *nc = rc1, *np = rp1, *nd = rd1, *ri = ri0, *ni = ri1;
    while (true) {
        if (nr == 0 && wh == nw) {  // nothing to run: idle until t_now (never backwards)
            t = fmax(t, a.t_now);
            break;
        }
        // A run of decode-only batches: with no request in prefill and no admission
        // possible (waiting queue empty, or every seat taken), every batch decodes one
        // token of each running request, so consecutive batches differ only in their
        // context sum until the first request finishes.  Each batch is still timed on
        // its own, with the general path's fp32 expression.
        {
            bool pre = false;
            int dmin = kBig;
            long long csum = 0;
            for (int r = lane; r < nr; r += 32) {
                pre |= rp[r] > 0;
                dmin = min(dmin, rd[r]);
                csum += rc[r];
            }
            if (!__any_sync(kFull, pre) && nr > 0 && (wh == nw || nr >= S) && iters < c.max_iters) {
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) dmin = min(dmin, __shfl_xor_sync(kFull, dmin, o));
                csum = warp_sum64(csum);
                const int run = (int)min((long long)dmin, (long long)c.max_iters - iters);
                const float f1 = 0.0f, f2 = __int2float_rn(nr), f4 = 0.0f;
                int done = 0;
                double t_first = t;  // end of the run's first batch, where every request decodes
                for (; done < run; ++done) {
                    float T = __fmul_rn(b0, 1.0f);
                    T = __fmaf_rn(b1d, f2, T);
                    T = __fmaf_rn(b1p, f1, T);
                    T = __fmaf_rn(b2, __ll2float_rn(csum + (long long)done * nr), T);
                    T = __fmaf_rn(b3, f4, T);
                    if (t + (double)T > a.t_now) break;
                    t += (double)T;
                    if (done == 0) t_first = t;
                }
                iters += done;
                if (done > 0) {
                    int kept = 0;
                    for (int base = 0; base < nr; base += 32) {
                        const int r = base + lane;
                        const bool live = r < nr;
                        const int dec = live ? rd[r] - done : 0;
                        // every request decodes in the run's first batch: that is the first
                        // token of a tracked one when the first token has its own batch
                        const int id = (track && live) ? emit_first(a, ri[r], c.mode == 0, t_first) : -1;
                        const bool keep = live && dec > 0;
                        const unsigned bal = __ballot_sync(kFull, keep);
                        if (keep) {
                            const int pos = kept + __popc(bal & lanemask_lt());
                            nc[pos] = rc[r] + done;
                            np[pos] = 0;
                            nd[pos] = dec;
                            if (track) ni[pos] = id;
                        }
                        kept += __popc(bal);
                    }
                    __syncwarp();
                    int32_t *x0 = rc, *x1 = rp, *x2 = rd, *x3 = ri;
                    rc = nc;
                    rp = np;
                    rd = nd;
                    ri = ni;
                    nc = x0;
                    np = x1;
                    nd = x2;
                    ni = x3;
                    nr = kept;
                }
                if (done < run) break;  // the next batch would end after t_now
                continue;               // a request finished (or max_iters is reached)
            }
        }
        if (++iters > c.max_iters) {
            ok = false;
            break;
        }
        // Plan the batch: the running list in order, each request taking
        // min(need, budget left) where need is its remaining prompt or one
        // decode token; then FCFS admission while budget and a slot remain.
        long long used = 0;  // tokens given to the running list so far
        long long f1 = 0, f2 = 0, f3 = 0, f4 = 0;
        for (int base = 0; base < nr; base += 32) {
            const int r = base + lane;
            const bool live = r < nr;
            const int need = live ? (rp[r] > 0 ? rp[r] : 1) : 0;
            const long long incl = used + warp_incl_sum64(need, lane);
            const long long excl = incl - need;
            const long long x = live ? max(0LL, min((long long)need, (long long)B - excl)) : 0;
            if (live && x > 0) {
                if (rp[r] > 0) {
                    f1 += x;
                    f4 += x * rc[r] + x * (x + 1) / 2;
                } else {
                    f2 += 1;
                    f3 += rc[r];
                }
            }
            used = __shfl_sync(kFull, incl, 31);
        }
        const long long budget = max(0LL, (long long)B - used);
        // admissions: the k-th waiting request is admitted if its prompt starts
        // inside the budget and a sequence slot is free
        int na = 0;
        long long wused = 0;
        for (int base = 0; budget - wused > 0 && wh + base < nw && nr + base < S; base += 32) {
            const int k = base + lane;
            const bool cand = wh + k < nw && nr + k < S;
            const int p = cand ? wp[wh + k] : 0;
            const long long incl = wused + warp_incl_sum64(p, lane);
            const long long st = incl - p;
            const bool adm = cand && st < budget;
            const long long x = adm ? min((long long)p, budget - st) : 0;
            f1 += x;
            f4 += x * (x + 1) / 2;
            const int nadm = __popc(__ballot_sync(kFull, adm));
            na += nadm;
            wused = __shfl_sync(kFull, incl, 31);
            if (nadm < 32) break;
        }
        f1 = warp_sum64(f1);
        f2 = warp_sum64(f2);
        f3 = warp_sum64(f3);
        f4 = warp_sum64(f4);
        // Eq. 9 for this batch, in the estimator's fp32 order
        float T = __fmul_rn(b0, 1.0f);
        T = __fmaf_rn(b1d, __ll2float_rn(f2), T);
        T = __fmaf_rn(b1p, __ll2float_rn(f1), T);
        T = __fmaf_rn(b2, __ll2float_rn(f3), T);
        T = __fmaf_rn(b3, __ll2float_rn(f4), T);
        if (t + (double)T > a.t_now) break;  // still running at t_now
        if (nr + na > capR) {
            ok = false;
            break;
        }
        // Execute it: update the running list and the admitted requests, then
        // keep (in order) every request with decode tokens left.
        int kept = 0;
        used = 0;
        const int total = nr + na;
        long long wst = 0;
        for (int base = 0; base < total; base += 32) {
            const int r = base + lane;
            int ctx = 0, pre = 0, dec = 0, id = -1;
            long long need = 0;
            const bool live = r < total;
            if (live) {
                if (r < nr) {
                    ctx = rc[r];
                    pre = rp[r];
                    dec = rd[r];
                    need = pre > 0 ? pre : 1;
                    if (track) id = ri[r];
                } else {
                    pre = wp[wh + r - nr];
                    dec = wd[wh + r - nr];
                    need = pre;
                    if (track) id = wi[wh + r - nr];
                }
            }
            const long long inr = (live && r < nr) ? need : 0;
            const long long incl_r = used + warp_incl_sum64(inr, lane);
            const long long inw = (live && r >= nr) ? need : 0;
            const long long incl_w = wst + warp_incl_sum64(inw, lane);
            long long x = 0;
            if (live && r < nr) x = max(0LL, min(need, (long long)B - (incl_r - inr)));
            if (live && r >= nr) x = min(need, budget - (incl_w - inw));
            if (live && x > 0) {
                if (pre > 0) {
                    ctx += (int)x;
                    pre -= (int)x;
                    if (pre == 0 && c.mode == 1) {
                        dec -= 1;  // first token with the last chunk
                        if (track) id = emit_first(a, id, true, t + (double)T);
                    }
                } else {
                    ctx += 1;
                    dec -= 1;
                    if (track) id = emit_first(a, id, c.mode == 0, t + (double)T);
                }
            }
            const bool keep = live && dec > 0;
            const unsigned bal = __ballot_sync(kFull, keep);
            if (keep) {
                const int pos = kept + __popc(bal & lanemask_lt());
                nc[pos] = ctx;
                np[pos] = pre;
                nd[pos] = dec;
                if (track) ni[pos] = id;
            }
            kept += __popc(bal);
            used = __shfl_sync(kFull, incl_r, 31);
            wst = __shfl_sync(kFull, incl_w, 31);
        }
        __syncwarp();
        int32_t *x0 = rc, *x1 = rp, *x2 = rd, *x3 = ri;
        rc = nc;
        rp = np;
        rd = nd;
        ri = ni;
        nc = x0;
        np = x1;
        nd = x2;
        ni = x3;
        nr = kept;
        wh += na;
        t += (double)T;
    }
    if (!ok) {
        fail3(a.ctl, kETraj, lane);
        return;
    }
    const int nw2 = nw - wh;
    for (int q = lane; q < capR; q += 32) {
        dst.run_ctx[rrow + q] = q < nr ? rc[q] : 0;
        dst.run_pre[rrow + q] = q < nr ? rp[q] : 0;
        dst.run_dec[rrow + q] = q < nr ? rd[q] : 0;
    }
    for (int q = lane; q < capW; q += 32) {
        dst.wait_pre[wrow + q] = q < nw2 ? wp[wh + q] : 0;
        dst.wait_dec[wrow + q] = q < nw2 ? wd[wh + q] : 0;
    }
    if (track) {
        for (int q = lane; q < capR; q += 32) idst.run_id[rrow + q] = q < nr ? ri[q] : -1;
        for (int q = lane; q < capW; q += 32) idst.wait_id[wrow + q] = q < nw2 ? wi[wh + q] : -1;
    }
    if (lane == 0) {
        dst.n_run[j] = nr;
        dst.n_wait[j] = nw2;
        dst.clock[j] = t;
    }
}

// ---- The stream step under KV-cache limits (App. F: KV-cache allocation, context
// limits and preemption; the same step rule as the KV estimate) ----
//
// One warp per instance, every batch planned in two warp passes: the running list in
// order (each request's tokens within the budget, its new blocks, the blocks it holds),
// then FCFS admission from the waiting head while the budget, a seat and the first
// chunk's blocks allow.  When the running scan's new blocks exceed the free ones, lane
// 0 replays the scan request by request, preempting the last running request (possibly
// the one being served) until each finds its blocks; that case is rare and keeps the
// exact order of the rule.  A preempted request returns its blocks, its whole context
// becomes prefill again and it goes to the front of the waiting ring, in running order.
// A request whose context reaches the limit ends.  Each batch takes the Eq. 9 time of
// its own composition in the estimator's fp32 order, and runs only if it ends by t_now.

__device__ __forceinline__ int kv_blk(int c, int bs) { return (int)(((unsigned)c + (unsigned)bs - 1u) / (unsigned)bs); }

__device__ void advance_instance_kv(const K3Launch &a, const StateBuf &src, const StateBuf &idst, int j, int lane,
                                    int32_t *wbase) {
    const DevConfig &c = a.cfg;
    const StateBuf &dst = a.scratch;
    const int B = c.B[j];
    const int S = c.S[j];
    const int bs = a.kv.bs[j];
    const long long nbk = a.kv.nb[j], mctx = a.kv.mctx[j];
    const int capR = c.capR, capW = c.capW;
    const int Wc = capW + capR;  // the waiting ring
    int32_t *rc0 = wbase, *rp0 = rc0 + capR, *rd0 = rp0 + capR;
    int32_t *rc1 = rd0 + capR, *rp1 = rc1 + capR, *rd1 = rp1 + capR;
    int32_t *ri0 = rd1 + capR, *ri1 = ri0 + capR;
    int32_t *wp = ri1 + capR, *wd = wp + Wc, *wi = wd + Wc;
    const bool track = a.track != 0;
    const size_t rrow = (size_t)j * capR, wrow = (size_t)j * capW;
    int nr = src.n_run[j];
    int nw = src.n_wait[j];
    for (int t = lane; t < nr; t += 32) {
        rc0[t] = src.run_ctx[rrow + t];
        rp0[t] = src.run_pre[rrow + t];
        rd0[t] = src.run_dec[rrow + t];
        ri0[t] = track ? src.run_id[rrow + t] : -1;
    }
    for (int t = lane; t < nw; t += 32) {
        wp[t] = src.wait_pre[wrow + t];
        wd[t] = src.wait_dec[wrow + t];
        wi[t] = track ? src.wait_id[wrow + t] : -1;
    }
    // routed queries join the waiting tail in query order; one that could never run
    // (its prompt at the context limit, or its whole context capped at the limit needing
    // more blocks than the instance has) is refused
    bool bad = false;
    for (int base = 0; base < a.Q; base += 32) {
        const int i = base + lane;
        const bool mine = i < a.Q && a.assign[i] == j;
        const unsigned bal = __ballot_sync(kFull, mine);
        if (mine) {
            const int pos = nw + __popc(bal & lanemask_lt());
            const int p = a.prompt[i];
            const int d = a.dec[(size_t)i * a.dec_cols + (a.dec_cols == 1 ? 0 : c.moi[j])];
            bad |= p < 1 || p > (1 << 24) || d < 1 || d > (1 << 24);
            bad |= (long long)p >= mctx;
            bad |= (long long)(((unsigned long long)min((long long)p + d, mctx) + bs - 1) / bs) > nbk;
            if (pos < capW) {
                wp[pos] = p;
                wd[pos] = d;
                wi[pos] = (track && a.id_base >= 0) ? (int)(a.id_base + i) : -1;
            }
        }
        nw += __popc(bal);
    }
    if (nw > capW) {
        fail3(a.ctl, kECapacity, lane);
        return;
    }
    if (__any_sync(kFull, bad)) {
        fail3(a.ctl, kEInval, lane);
        return;
    }
    __syncwarp();

    const float *cf = c.coef + 5 * c.moi[j];
    const float b0 = cf[0], b1p = cf[1], b1d = cf[2], b2 = cf[3], b3 = cf[4];
    double t = src.clock[j];
    int wh = 0, iters = 0;  // the waiting ring holds nw requests from wh on
    int err = kOk;
    int32_t *rc = rc0, *rp = rp0, *rd = rd0, *ri = ri0, *nc = rc1, *np = rp1, *nd = rd1, *ni = ri1;
    while (true) {
        if (nr == 0 && nw == 0) {  // nothing to run: idle until t_now (never backwards)
            t = fmax(t, a.t_now);
            break;
        }
        if (++iters > c.max_iters) {
            err = kETraj;
            break;
        }
        // 1. the running scan: each request's tokens within the budget (a prefix of the
        //    list is served), the new blocks they need and the blocks every request holds
        long long used = 0, held = 0, nblk = 0;
        long long f1 = 0, f2 = 0, f3 = 0, f4 = 0;
        int rend = 0;
        for (int base = 0; base < nr; base += 32) {
            const int r = base + lane;
            const bool live = r < nr;
            const int ctx = live ? rc[r] : 0, pre = live ? rp[r] : 0;
            const int need = live ? (pre > 0 ? pre : 1) : 0;
            const long long incl = used + warp_incl_sum64(need, lane);
            const long long x = live ? max(0LL, min((long long)need, (long long)B - (incl - need))) : 0;
            if (live) held += kv_blk(ctx, bs);
            if (x > 0) {
                nblk += kv_blk(ctx + (int)x, bs) - kv_blk(ctx, bs);
                if (pre > 0) {
                    f1 += x;
                    f4 += x * ctx + x * (x + 1) / 2;
                } else {
                    f2 += 1;
                    f3 += ctx;
                }
            }
            rend += __popc(__ballot_sync(kFull, x > 0));
            used = __shfl_sync(kFull, incl, 31);
        }
        held = warp_sum64(held);
        nblk = warp_sum64(nblk);
        long long freeb = nbk - held;
        long long budget = max(0LL, (long long)B - used);
        int pnr = nr;  // running requests left after preemptions
        if (nblk > freeb) {
            // Not every served request finds its blocks: lane 0 replays the scan in the
            // rule's order, preempting from the tail, and the served prefix's features
            // are summed again.
            long long pf = freeb, bud = B;
            int r = 0, n = nr;
            if (lane == 0) {
                while (r < n && bud > 0) {
                    const long long x = rp[r] > 0 ? min((long long)rp[r], bud) : 1LL;
                    const int nb1 = kv_blk(rc[r] + (int)x, bs) - kv_blk(rc[r], bs);
                    while (pf < nb1 && n - 1 >= r) {
                        --n;
                        pf += kv_blk(rc[n], bs);
                    }
                    if (r >= n) break;  // r preempted itself
                    pf -= nb1;
                    bud -= x;
                    ++r;
                }
            }
            rend = __shfl_sync(kFull, r, 0);
            pnr = __shfl_sync(kFull, n, 0);
            freeb = __shfl_sync(kFull, pf, 0);
            budget = __shfl_sync(kFull, bud, 0);
            f1 = f2 = f3 = f4 = 0;
            used = 0;
            for (int base = 0; base < rend; base += 32) {
                const int r2 = base + lane;
                const bool live = r2 < rend;
                const int ctx = live ? rc[r2] : 0, pre = live ? rp[r2] : 0;
                const int need = live ? (pre > 0 ? pre : 1) : 0;
                const long long incl = used + warp_incl_sum64(need, lane);
                const long long x = live ? max(0LL, min((long long)need, (long long)B - (incl - need))) : 0;
                if (x > 0) {
                    if (pre > 0) {
                        f1 += x;
                        f4 += x * ctx + x * (x + 1) / 2;
                    } else {
                        f2 += 1;
                        f3 += ctx;
                    }
                }
                used = __shfl_sync(kFull, incl, 31);
            }
        } else {
            freeb -= nblk;
        }
        // the preempted tail [pnr, nr) goes to the ring's front in running order, its
        // whole context prefill again (the slots before the head are free; the head
        // moves only if the batch runs)
        const int k = nr - pnr;
        int wh2 = wh - k;
        if (wh2 < 0) wh2 += Wc;
        for (int i = lane; i < k; i += 32) {
            int pos = wh2 + i;
            if (pos >= Wc) pos -= Wc;
            wp[pos] = rc[pnr + i] + rp[pnr + i];
            wd[pos] = rd[pnr + i];
            wi[pos] = ri[pnr + i];
        }
        __syncwarp();
        const int nw2 = nw + k;
        // 2. admission from the ring's head while the budget, a seat and the first
        //    chunk's blocks allow (each condition holds for a prefix of the queue)
        int na = 0;
        long long wused = 0, bused = 0;
        for (int base = 0; budget - wused > 0 && base < nw2 && pnr + base < S; base += 32) {
            const int q = base + lane;
            int pos = wh2 + q;
            if (pos >= Wc) pos -= Wc;
            const bool in = q < nw2 && pnr + q < S;
            const int p = in ? wp[pos] : 0;
            const long long incl = wused + warp_incl_sum64(p, lane);
            const long long st = incl - p;
            const bool cand = in && st < budget;
            const long long x = cand ? min((long long)p, budget - st) : 0;
            const int nb1 = cand ? kv_blk((int)x, bs) : 0;
            const long long binc = bused + warp_incl_sum64(nb1, lane);
            const bool adm = cand && binc <= freeb;
            if (adm) {
                f1 += x;
                f4 += x * (x + 1) / 2;
            }
            const int nadm = __popc(__ballot_sync(kFull, adm));
            na += nadm;
            wused = __shfl_sync(kFull, incl, 31);
            bused = __shfl_sync(kFull, binc, 31);
            if (nadm < 32) break;
        }
        f1 = warp_sum64(f1);
        f2 = warp_sum64(f2);
        f3 = warp_sum64(f3);
        f4 = warp_sum64(f4);
        // Eq. 9 for this batch, in the estimator's fp32 order
        float T = __fmul_rn(b0, 1.0f);
        T = __fmaf_rn(b1d, __ll2float_rn(f2), T);
        T = __fmaf_rn(b1p, __ll2float_rn(f1), T);
        T = __fmaf_rn(b2, __ll2float_rn(f3), T);
        T = __fmaf_rn(b3, __ll2float_rn(f4), T);
        if (t + (double)T > a.t_now) break;  // still running at t_now
        if (pnr + na > capR) {
            err = kETraj;
            break;
        }
        // 3. execute it: the served prefix and the admitted requests advance; a request
        //    with no decode token left, or whose context reached the limit, ends
        int kept = 0;
        long long rused = 0, wst = 0;
        const int total = pnr + na;
        for (int base = 0; base < total; base += 32) {
            const int r = base + lane;
            const bool isr = r < pnr, isw = r >= pnr && r < total;
            int ctx = 0, pre = 0, dec = 0, id = -1;
            if (isr) {
                ctx = rc[r];
                pre = rp[r];
                dec = rd[r];
                id = ri[r];
            } else if (isw) {
                int pos = wh2 + (r - pnr);
                if (pos >= Wc) pos -= Wc;
                pre = wp[pos];
                dec = wd[pos];
                id = wi[pos];
            }
            const long long inr = isr ? (pre > 0 ? pre : 1) : 0;
            const long long incl_r = rused + warp_incl_sum64(inr, lane);
            const long long inw = isw ? pre : 0;
            const long long incl_w = wst + warp_incl_sum64(inw, lane);
            long long x = 0;
            if (isr && r < rend) x = max(0LL, min(inr, (long long)B - (incl_r - inr)));
            if (isw) x = min(inw, budget - (incl_w - inw));
            if (x > 0) {
                if (pre > 0) {
                    ctx += (int)x;
                    pre -= (int)x;
                    if (pre == 0 && c.mode == 1) {
                        dec -= 1;  // first token with the last chunk
                        if (track) id = emit_first(a, id, true, t + (double)T);
                    }
                } else {
                    ctx += 1;
                    dec -= 1;
                    if (track) id = emit_first(a, id, c.mode == 0, t + (double)T);
                }
            }
            if (pre == 0 && (long long)ctx >= mctx) dec = 0;  // the context limit
            const bool keep = (isr || isw) && dec > 0;
            const unsigned bal = __ballot_sync(kFull, keep);
            if (keep) {
                const int pos = kept + __popc(bal & lanemask_lt());
                nc[pos] = ctx;
                np[pos] = pre;
                nd[pos] = dec;
                ni[pos] = id;
            }
            kept += __popc(bal);
            rused = __shfl_sync(kFull, incl_r, 31);
            wst = __shfl_sync(kFull, incl_w, 31);
        }
        __syncwarp();
        int32_t *x0 = rc, *x1 = rp, *x2 = rd, *x3 = ri;
        rc = nc;
        rp = np;
        rd = nd;
        ri = ni;
        nc = x0;
        np = x1;
        nd = x2;
        ni = x3;
        nr = kept;
        wh = wh2 + na;
        if (wh >= Wc) wh -= Wc;
        nw = nw2 - na;
        t += (double)T;
        if (nw > capW) {
            err = kECapacity;
            break;
        }
    }
    if (err != kOk) {
        fail3(a.ctl, err, lane);
        return;
    }
    for (int q = lane; q < capR; q += 32) {
        dst.run_ctx[rrow + q] = q < nr ? rc[q] : 0;
        dst.run_pre[rrow + q] = q < nr ? rp[q] : 0;
        dst.run_dec[rrow + q] = q < nr ? rd[q] : 0;
        if (track) idst.run_id[rrow + q] = q < nr ? ri[q] : -1;
    }
    for (int q = lane; q < capW; q += 32) {
        int pos = wh + q;
        if (pos >= Wc) pos -= Wc;
        dst.wait_pre[wrow + q] = q < nw ? wp[pos] : 0;
        dst.wait_dec[wrow + q] = q < nw ? wd[pos] : 0;
        if (track) idst.wait_id[wrow + q] = q < nw ? wi[pos] : -1;
    }
    if (lane == 0) {
        dst.n_run[j] = nr;
        dst.n_wait[j] = nw;
        dst.clock[j] = t;
    }
}

__global__ void __launch_bounds__(kK3Warps * 32) k_advance(const K3Launch a) {
    extern __shared__ __align__(16) int32_t k3_smem[];
    const int lane = threadIdx.x & 31;
    const int wid = threadIdx.x >> 5;
    const int j = blockIdx.x * kK3Warps + wid;
    const int active = *((volatile int32_t *)&a.ctl->active);
    if (j >= a.cfg.I) return;
    if (active < 0) {
        fail3(a.ctl, kENoState, lane);
        return;
    }
    const StateBuf src = active ? a.buf1 : a.buf0;
    // the buffer the summary (K1) publishes next, as K1 chooses it from the same index
    const StateBuf idst = active ? a.buf0 : a.buf1;
    const size_t per_warp = advance_smem_per_warp(a.cfg) / sizeof(int32_t);
    advance_instance(a, src, idst, j, lane, k3_smem + wid * per_warp);
}

__global__ void __launch_bounds__(kK3Warps * 32) k_advance_kv(const K3Launch a) {
    extern __shared__ __align__(16) int32_t k3_smem[];
    const int lane = threadIdx.x & 31;
    const int wid = threadIdx.x >> 5;
    const int j = blockIdx.x * kK3Warps + wid;
    const int active = *((volatile int32_t *)&a.ctl->active);
    if (j >= a.cfg.I) return;
    if (active < 0) {
        fail3(a.ctl, kENoState, lane);
        return;
    }
    const StateBuf src = active ? a.buf1 : a.buf0;
    // the buffer the KV load publishes next, as it chooses it from the same index
    const StateBuf idst = active ? a.buf0 : a.buf1;
    const size_t per_warp = advance_kv_smem_per_warp(a.cfg) / sizeof(int32_t);
    advance_instance_kv(a, src, idst, j, lane, k3_smem + wid * per_warp);
}

// Copy of the live snapshot into caller arrays (the live buffer is known only on
// the device).
__global__ void k_read_state(const DevConfig c, const StateBuf b0, const StateBuf b1, const DevCtl *ctl,
                             const StateOut o) {
    const int active = *((volatile const int32_t *)&ctl->active);
    const StateBuf s = active == 1 ? b1 : b0;
    const size_t R = (size_t)c.I * c.capR, W = (size_t)c.I * c.capW;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < R + W + c.I;
         i += (size_t)gridDim.x * blockDim.x) {
        if (i < R) {
            if (o.run_ctx) o.run_ctx[i] = s.run_ctx[i];
            if (o.run_pre) o.run_pre[i] = s.run_pre[i];
            if (o.run_dec) o.run_dec[i] = s.run_dec[i];
        } else if (i < R + W) {
            if (o.wait_pre) o.wait_pre[i - R] = s.wait_pre[i - R];
            if (o.wait_dec) o.wait_dec[i - R] = s.wait_dec[i - R];
        } else {
            const size_t k = i - R - W;
            if (o.n_run) o.n_run[k] = s.n_run[k];
            if (o.n_wait) o.n_wait[k] = s.n_wait[k];
            if (o.clock) o.clock[k] = s.clock[k];
        }
    }
}

}  // namespace

cudaError_t launch_read_state(const DevConfig &c, const StateBuf &b0, const StateBuf &b1, DevCtl *ctl,
                              const StateOut &o, cudaStream_t st) {
    k_read_state<<<128, 256, 0, st>>>(c, b0, b1, ctl, o);
    return cudaGetLastError();
}

cudaError_t launch_advance(const K3Launch &a, int grid, size_t smem, cudaStream_t st) {
    k_advance<<<grid, kK3Warps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t set_k3_smem(size_t bytes) {
    return cudaFuncSetAttribute(k_advance, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

cudaError_t launch_advance_kv(const K3Launch &a, int grid, size_t smem, cudaStream_t st) {
    k_advance_kv<<<grid, kK3Warps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t set_k3_kv_smem(size_t bytes) {
    return cudaFuncSetAttribute(k_advance_kv, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace lr
