// KV-limited Serving Framework Simulation (Sec. 4.1; App. F names context limits,
// the KV-cache allocation state and preemption among what the simulation models).
//
// Reading of the step rule: instance j has nb_j blocks of bs_j tokens and a request
// with c tokens in the cache holds ceil(c / bs_j) of them.  The running list is
// served in order; a request whose tokens of the batch need blocks that are not
// free preempts the last running request (its blocks return, its whole context
// becomes prefill again and it goes to the front of the waiting queue), itself if it
// is the last.  The waiting head is admitted only if its first chunk's blocks are
// free.  A request whose context reaches mctx_j ends there.
//
// The query q appended at the waiting tail never changes the residents' batches:
// it is admitted only once no resident waits, and while it runs it is the last
// running request, so it is the first preemption victim and no resident ever waits
// for its blocks.  So the load (k_kv_load) simulates each instance's residents
// alone, once, and records for every batch from the first in which q could be
// admitted what q's fate depends on: the budget left to it, the largest prompt it
// could be admitted with, the free blocks and the least block slack of the
// residents' scan (q, holding h blocks, is preempted in a batch whose slack is
// below h), and the residents' Eq. 9 features summed so far.  The estimate
// (k_kv_estimate) then finds each (query, instance) candidate's admission batch by
// a binary search over the running maximum of the admission bounds and follows it
// from there, record by record, through prefill chunks, preemptions and
// readmissions, to its first token.  A candidate depends only on the instance and
// the prompt length, so each call first counting-sorts its queries by length
// (k_kv_count, k_kv_scan, k_kv_scatter), walks once per distinct length, and
// copies those rows to the other queries of the same length (k_kv_expand).
#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr long long kHuge = 1LL << 62;

__device__ __forceinline__ long long kv_blocks(long long c, long long bs) { return (c + bs - 1) / bs; }
// ceil(c / bs) for 0 <= c < 2^31 (32-bit division)
__device__ __forceinline__ int kv_blocks32(int c, int bs) {
    return (int)(((unsigned)c + (unsigned)bs - 1u) / (unsigned)bs);
}

__device__ void kv_fail(DevCtl *ctl, int code, int lane) {
    if (lane == 0) {
        atomicCAS(&ctl->load_err, 0, code);
        record_status(ctl, code);
    }
}

__device__ __forceinline__ long long warp_incl_sum64(long long x, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const long long y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
    }
    return x;
}
__device__ __forceinline__ int warp_incl_sum32(int x, int lane) {
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(kFull, x, o);
        if (lane >= o) x += y;
    }
    return x;
}
__device__ __forceinline__ long long warp_sum64(long long x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
    return x;
}
__device__ __forceinline__ int warp_sum32(int x) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(kFull, x, o);
    return x;
}

// End calendar of the KV load: a decoder that ends in batch E (>= the current
// batch G) waits in list E mod kKvCal if E < G + kKvCal, else in the overflow list,
// whose nodes are re-filed at every multiple of kKvCal.  Pushes from several lanes
// at once are safe.
__device__ __forceinline__ void kv_cal_push(int32_t *head, int32_t *nxt, int32_t *ovf, int s, long long E, int G) {
    int32_t *h = E < (long long)G + kKvCal ? &head[E & (kKvCal - 1)] : ovf;
    nxt[s] = atomicExch(h, s);
}
// the batch (as a value of G) in which a decoder held as (context - G, decode + G) ends
__device__ __forceinline__ long long kv_end(const int4 &q, long long mctx) {
    return min((long long)q.z - 1, mctx - 1 - q.x);
}
// Division by an instance's block size, which the load repeats many times a batch:
// unsigned n / d for any 32-bit n as a multiply-high and shifts (Granlund and
// Montgomery's method for invariant divisors: l = ceil(log2 d), m = floor(2^32 (2^l - d)
// / d) + 1, q = (t + ((n - t) >> 1)) >> (l - 1) with t = mulhi(m, n); d = 1 takes
// shifts of 0).
struct Div32 {
    unsigned d, m;
    int s1, s2;
};
__device__ __forceinline__ Div32 make_div32(int d) {
    const unsigned ud = (unsigned)d;
    const int l = ud <= 1u ? 0 : 32 - __clz((int)(ud - 1u));
    Div32 v;
    v.d = ud;
    v.m = (unsigned)((((1ull << 32) * ((1ull << l) - ud)) / ud) + 1ull);
    v.s1 = min(l, 1);
    v.s2 = max(l - 1, 0);
    return v;
}
__device__ __forceinline__ unsigned udiv32(const Div32 &v, unsigned n) {
    const unsigned t = __umulhi(v.m, n);
    return (t + ((n - t) >> v.s1)) >> v.s2;
}
// ceil(c / d) for 0 <= c < 2^31
__device__ __forceinline__ int dblk(const Div32 &v, int c) { return (int)udiv32(v, (unsigned)c + v.d - 1u); }
// x mod d in [0, d) for any int x
__device__ __forceinline__ int dres(const Div32 &v, int x) {
    if (x >= 0) return (int)((unsigned)x - udiv32(v, (unsigned)x) * v.d);
    const unsigned ax = (unsigned)(-(long long)x);
    const unsigned r = ax - udiv32(v, ax) * v.d;
    return r == 0u ? 0 : (int)(v.d - r);
}

// One instance's residents alone, batch by batch, from the snapshot.  Every lane
// holds the same scalar state.
//
// Running request in slot s: rq[s] = (context, prefill, decode, blocks held) for
// the prefill request, (context - G, 0, decode + G, context residue mod bs) for a
// decoder, whose blocks at its end wait in eb[s].  Slots keep the list's order; a
// request that leaves becomes a hole (prefill -1) until a compaction.  Only the
// last running request may be in prefill (slot pfs).  The others decode one token
// a batch (G = batches done), so no word of theirs changes until they end.  The
// decoders crossing into a new block in batch G are those whose context is a
// multiple of bs, counted by a histogram of stored contexts mod bs; their context
// sum (Eq. 9's F3 term) is a running total; the batch each one ends in (decode
// count or context limit) waits in the end calendar.  A request that ends frees
// ceil(context / bs) blocks after its last batch.
template <int MODE>
__device__ void kv_instance(const KvLoad &a, const StateBuf &out, int j, int lane, int32_t *wb) {
    const DevConfig &c = a.cfg;
    const int B = c.B[j];
    const int S = c.S[j];
    const long long nbk = a.kv.nb[j], mctx = a.kv.mctx[j];
    const int bs = a.kv.bs[j];
    const Div32 dv = make_div32(bs);
    const int C = c.capR + c.capW;  // at most this many residents
    int4 *rq = reinterpret_cast<int4 *>(wb);               // running list slots
    int2 *wq = reinterpret_cast<int2 *>(rq + C);           // waiting ring (prefill, decode)
    int32_t *nxt = reinterpret_cast<int32_t *>(wq + C);    // [C] calendar links
    int32_t *eb = nxt + C;                                 // [C] a decoder's blocks at its end
    int32_t *head = eb + C;                                // [kKvCal] calendar lists
    int32_t *hist = head + kKvCal;                         // [bs] residue histogram
    int32_t *ovf = hist + a.kv.hist;                       // overflow list head
    const int nr0 = a.in.n_run[j];
    const int nw0 = a.in.n_wait[j];
    if (lane == 0) {
        out.n_run[j] = nr0;
        out.n_wait[j] = nw0;
        out.clock[j] = a.in.clock ? a.in.clock[j] : 0.0;
    }
    if (!(nr0 >= 0 && nr0 <= c.capR && nr0 <= S && nw0 >= 0 && nw0 <= c.capW)) {
        kv_fail(a.ctl, kEState, lane);
        return;
    }
    for (int b = lane; b < kKvCal; b += 32) head[b] = -1;
    for (int b = lane; b < bs; b += 32) hist[b] = 0;
    if (lane == 0) *ovf = -1;
    // file decoder slot s, held as q (fourth word: residue) at batch G
    auto file = [&](int s, const int4 &q, int G_) {
        const long long E = kv_end(q, mctx);
        eb[s] = dblk(dv, (int)(q.x + E + 1));
        kv_cal_push(head, nxt, ovf, s, E, G_);
    };
    // Copy and validate the snapshot: only the last running request may still be in
    // prefill, no context reaches the limit, every request's whole context fits the
    // instance's blocks, and the running requests' blocks fit together.
    const size_t rrow = (size_t)j * c.capR, wrow = (size_t)j * c.capW;
    bool bad = false;
    long long held = 0, wsum = 0, src = 0;
    int nd = 0;
    for (int t = lane; t < c.capR; t += 32) {
        const int ctx = a.in.run_ctx[rrow + t], pre = a.in.run_pre[rrow + t], dec = a.in.run_dec[rrow + t];
        out.run_ctx[rrow + t] = ctx;
        out.run_pre[rrow + t] = pre;
        out.run_dec[rrow + t] = dec;
        if (t < nr0) {
            const bool ok = ctx >= 0 && ctx <= (1 << 28) && pre >= 0 && pre <= (1 << 24) && dec >= 1 &&
                            dec <= (1 << 24);
            bad |= !ok;
            bad |= pre > 0 && t != nr0 - 1;
            bad |= (long long)ctx + pre >= mctx;
            bad |= ok && kv_blocks(min((long long)ctx + pre + dec, mctx), bs) > nbk;
            const int h = ok ? dblk(dv, ctx) : 0;
            held += h;
            if (pre == 0) {
                src += ctx;
                ++nd;
            }
            rq[t] = pre > 0 ? make_int4(ctx, pre, dec, h) : make_int4(ctx, 0, dec, dres(dv, ctx));
        }
    }
    for (int t = lane; t < c.capW; t += 32) {
        const int pre = a.in.wait_pre[wrow + t], dec = a.in.wait_dec[wrow + t];
        out.wait_pre[wrow + t] = pre;
        out.wait_dec[wrow + t] = dec;
        if (t < nw0) {
            bad |= pre < 1 || pre > (1 << 24) || dec < 1 || dec > (1 << 24);
            bad |= (long long)pre >= mctx;
            bad |= kv_blocks(min((long long)pre + dec, mctx), bs) > nbk;
            wsum += pre;
            wq[t] = make_int2(pre, dec);
        }
    }
    held = warp_sum64(held);
    wsum = warp_sum64(wsum);
    src = warp_sum64(src);
    nd = warp_sum32(nd);
    if (__any_sync(kFull, bad) || held > nbk || wsum > (1LL << 30)) {
        kv_fail(a.ctl, kEState, lane);
        return;
    }
    __syncwarp();
    // the decoders into the histogram and the calendar (G = 0)
    for (int t = lane; t < nr0; t += 32) {
        const int4 q = rq[t];
        if (q.y == 0) {
            atomicAdd(&hist[q.w], 1);
            file(t, q, 0);
        }
    }
    __syncwarp();

    long long freeb = nbk - held;
    int nr = nr0, ne = nr0;                             // running requests; slots in use
    int pfs = (nr0 > 0 && rq[nr0 - 1].y > 0) ? nr0 - 1 : -1;  // the prefill request's slot
    int wh = 0, wc = nw0;                               // waiting ring head and count
    int G = 0, gr = 0;                                  // batches done; G mod bs
    long long f4c = 0;                                  // this lane's part of F4 before the first record
    long long fcum[5] = {0, 0, 0, 0, 0};
    long long cf1 = 0, cf2 = 0, cf3 = 0, cf4 = 0;  // features summed over the records
    int la0 = 0, nrec = 0, done = 0, pmx = 0;
    KvRec *rec = out.kvr + (size_t)j * a.kv.horizon;
    int32_t *pmxo = out.kvp + (size_t)j * a.kv.horizon;

    // live slots to [0, nr) in order, and the calendar rebuilt
    auto compact = [&]() {
        int kept = 0;
        for (int base = 0; base < ne; base += 32) {
            const int s = base + lane;
            const int4 q = s < ne ? rq[s] : make_int4(0, -1, 0, 0);
            const int e = s < ne ? eb[s] : 0;
            const bool live = q.y >= 0;
            const unsigned m = __ballot_sync(kFull, live);
            __syncwarp();
            if (live) {
                const int d = kept + __popc(m & ((1u << lane) - 1u));
                rq[d] = q;
                eb[d] = e;
            }
            kept += __popc(m);
            __syncwarp();
        }
        ne = kept;
        for (int b = lane; b < kKvCal; b += 32) head[b] = -1;
        if (lane == 0) *ovf = -1;
        __syncwarp();
        for (int s = lane; s < ne; s += 32) {
            const int4 q = rq[s];
            if (q.y == 0) kv_cal_push(head, nxt, ovf, s, kv_end(q, mctx), G);
        }
        pfs = (ne > 0 && rq[ne - 1].y > 0) ? ne - 1 : -1;
        __syncwarp();
    };

    // Up to 32 batches at once, lane k taking batch G + k, while no resident waits
    // (after the first record): then a batch admits nobody, and all it depends on is
    // known at the window's start -- the decoders ending in it (the calendar), those
    // crossing into a new block (the histogram, less the earlier ends of the
    // window), the prefill request's chunk (the budget the decoders leave, summed)
    // and the free blocks (needs and returns, summed).  The window stops before a
    // batch that preempts or in which the prefill request finishes (both taken by
    // the batch step), at a re-file boundary, at the horizon, and after the batch
    // that empties the instance.  The window's ends are listed in the idle waiting
    // ring.  Returns the batches done (0: none).
    int32_t *evn = ovf + 1;  // the window's ends
    auto window = [&]() -> int {
        const int W = min(min(32, a.kv.horizon - nrec), kKvCal - (G & (kKvCal - 1)));
        if (lane == 0) *evn = 0;
        __syncwarp();
        const int k = lane;
        int cntk = 0;
        long long rck = 0, ebk = 0;
        if (k < W) {
            for (int s = head[(G + k) & (kKvCal - 1)]; s >= 0;) {
                const int ns = nxt[s];
                const int4 q = rq[s];
                if (q.y == 0) {
                    ++cntk;
                    rck += q.x;
                    ebk += eb[s];
                    wq[atomicAdd(evn, 1)] = make_int2(k, s);
                }
                s = ns;
            }
        }
        __syncwarp();
        const int nev = *evn;
        const int endsb = warp_incl_sum32(cntk, lane) - cntk;  // ends before batch k
        const long long rcb = warp_incl_sum64(rck, lane) - rck;
        const int ndk = nd - endsb, nrk = nr - endsb;
        const long long srck = src - rcb;
        // decoders at a block boundary in batch G + k, the window's earlier ends removed
        const int gk = dres(dv, gr + k);
        const int rk = gk == 0 ? 0 : bs - gk;
        int sub = 0;
        for (int e = 0; e < nev; ++e) {
            const int2 ev = wq[e];
            if (ev.x < k && rq[ev.y].w == rk) ++sub;
        }
        const int need_d = ndk > 0 ? hist[rk] - sub : 0;
        // the prefill request's chunk: what the decoders leave, until it finishes
        int x = 0, pneed = 0, ctxp = 0, remk = 0;
        bool pf_ends = false;
        const int4 pq = pfs >= 0 ? rq[pfs] : make_int4(0, 0, 0, 0);
        if (pfs >= 0) {
            const int avail = B - ndk;
            const int before = warp_incl_sum32(k < W ? avail : 0, lane) - (k < W ? avail : 0);
            remk = max(0, pq.y - before);
            x = min(remk, avail);
            pf_ends = remk - x == 0;
            ctxp = pq.x + (pq.y - remk);
            pneed = dblk(dv, ctxp + x) - dblk(dv, ctxp);
        }
        const int need_all = need_d + pneed;
        const long long dl = k < W ? ebk - need_all : 0;       // free blocks gained over batch k
        const long long fb = freeb + warp_incl_sum64(dl, lane) - dl;  // free blocks before batch k
        const unsigned okm = __ballot_sync(kFull, k < W && !pf_ends && need_all <= fb);
        int n = okm == kFull ? 32 : __ffs(~okm) - 1;
        const unsigned em = __ballot_sync(kFull, k < n && nrk - cntk == 0);  // the instance empties
        if (em) n = __ffs(em);
        if (n == 0) return 0;
        const bool in = k < n;
        const long long fa = fb - need_all;
        const int bar = B - ndk - x;
        const long long c1 = cf1 + warp_incl_sum64(in ? x : 0, lane);
        const long long c2 = cf2 + warp_incl_sum64(in ? ndk : 0, lane);
        const long long c3 = cf3 + warp_incl_sum64(in ? srck + (long long)ndk * (G + k) : 0, lane);
        const long long c4 = cf4 + warp_incl_sum64(in ? (long long)x * ctxp + (long long)x * (x + 1) / 2 : 0, lane);
        long long thr = 0;
        if (in && bar > 0 && nrk < S) thr = ((long long)bar <= fa * bs) ? kHuge : fa * bs;
        int pm = max(pmx, (int)min(thr, (long long)INT32_MAX));
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(kFull, pm, o);
            if (lane >= o) pm = max(pm, y);
        }
        if (in) {
            KvRec R;
            R.cf[0] = c1;
            R.cf[1] = c2;
            R.cf[2] = c3;
            R.cf[3] = c4;
            R.slack = fa;  // nrk > 0: the window never starts on an empty instance
            R.far = fa;
            R.thr = thr;
            R.bar = bar;
            R.bl = bar;
            rec[nrec + k] = R;
            pmxo[nrec + k] = pm;
        }
        // the state after batch n - 1
        const int L = n - 1;
        const int ndL = __shfl_sync(kFull, ndk, L), nrL = __shfl_sync(kFull, nrk, L), cntL = __shfl_sync(kFull, cntk, L);
        const long long srcL = __shfl_sync(kFull, srck, L), rckL = __shfl_sync(kFull, rck, L);
        const long long fbL = __shfl_sync(kFull, fb, L), dlL = __shfl_sync(kFull, dl, L);
        const int xL = __shfl_sync(kFull, x, L), ctxpL = __shfl_sync(kFull, ctxp, L), remL = __shfl_sync(kFull, remk, L);
        cf1 = __shfl_sync(kFull, c1, L);
        cf2 = __shfl_sync(kFull, c2, L);
        cf3 = __shfl_sync(kFull, c3, L);
        cf4 = __shfl_sync(kFull, c4, L);
        pmx = __shfl_sync(kFull, pm, L);
        __syncwarp();
        for (int e = lane; e < nev; e += 32) {  // the window's ends leave
            const int2 ev = wq[e];
            if (ev.x < n) {
                atomicSub(&hist[rq[ev.y].w], 1);
                reinterpret_cast<int *>(rq + ev.y)[1] = -1;
            }
        }
        if (in) head[(G + k) & (kKvCal - 1)] = -1;
        if (pfs >= 0 && lane == 0) rq[pfs] = make_int4(ctxpL + xL, remL - xL, pq.z, dblk(dv, ctxpL + xL));
        nd = ndL - cntL;
        nr = nrL - cntL;
        src = srcL - rckL;
        freeb = fbL + dlL;
        nrec += n;
        G += n;
        gr = dres(dv, G);
        if (nr == 0) done = 1;
        __syncwarp();
        return n;
    };

    for (int l = 1;; ++l) {
        if (l > c.max_iters) {
            kv_fail(a.ctl, kETraj, lane);
            return;
        }
        if (G > 0 && (G & (kKvCal - 1)) == 0) {
            // re-file the overflow list
            if (lane == 0) {
                int s = *ovf, keep = -1;
                while (s >= 0) {
                    const int ns = nxt[s];
                    const int4 q = rq[s];
                    if (q.y == 0) {
                        const long long E = kv_end(q, mctx);
                        int32_t *h = E < (long long)G + kKvCal ? &head[E & (kKvCal - 1)] : &keep;
                        nxt[s] = *h;
                        *h = s;
                    }
                    s = ns;
                }
                *ovf = keep;
            }
            __syncwarp();
        }
        if (la0 != 0 && wc == 0) {
            const int n = window();
            if (n > 0) {
                l += n - 1;
                if (done || nrec == a.kv.horizon) break;
                if (ne - nr >= max(32, nr)) compact();
                continue;
            }
        }
        // 1. The running scan.  n_run <= S <= B and only the last request may be in
        //    prefill, so every request gets its tokens if the blocks suffice: one per
        //    decoder, and the last one's chunk from what the decoders leave.
        const int4 pq = pfs >= 0 ? rq[pfs] : make_int4(0, 0, 0, 0);
        const int need_d = nd > 0 ? hist[gr == 0 ? 0 : bs - gr] : 0;  // decoders at a block boundary
        int px = 0, pneed = 0;
        if (pfs >= 0) {
            px = min(pq.y, B - nd);
            pneed = dblk(dv, pq.x + px) - pq.w;
        }
        const int need_all = need_d + pneed;
        long long slack, f1, f2, f3, f4;
        int budget;
        bool pf_run = pfs >= 0;  // the prefill request still runs after the scan
        int dying = 0;           // requests leaving after this batch
        long long back = 0;      // and their blocks
        if (need_all <= freeb) {
            slack = nr > 0 ? freeb - need_all : kHuge;
            freeb -= need_all;
            budget = B - nd - px;
            f1 = px;
            f2 = nd;
            f3 = src + (long long)nd * G;
            f4 = (long long)px * pq.x + (long long)px * (px + 1) / 2;
        } else {
            // a request runs out of blocks.  Preempting the tail until each request, in
            // order, has its blocks leaves the longest prefix of the list whose blocks
            // after the batch fit in the instance (what the rest held is what was free
            // to them): those run, the rest go, in order, to the front of the waiting
            // queue.  The prefill request, last, goes first, so the survivors are
            // decoders.
            // Every request's blocks after the batch sum to what is held plus what the
            // batch needs, so the cut is found from the tail: the first slot cut (from the
            // end) whose suffix of post-batch blocks reaches the excess over nb_j.  Usually
            // few requests go, and the walk stops in the first 32 slots.
            const long long total = (nbk - freeb) + need_all, excess = total - nbk;
            long long acc = 0, fitb = -1;  // post-batch blocks: of the suffix so far; of the survivors
            int cut = 0;
            for (int top = ne - 1; top >= 0; top -= 32) {
                const int s = top - lane;
                long long wv = 0;
                if (s >= 0) {
                    const int4 q = rq[s];
                    if (q.y == 0) wv = dblk(dv, q.x + G + 1);
                    else if (q.y > 0) wv = dblk(dv, q.x + px);
                }
                const long long suf = acc + warp_incl_sum64(wv, lane);
                const unsigned hit = __ballot_sync(kFull, s >= 0 && suf >= excess);
                if (hit) {
                    const int l0 = __ffs(hit) - 1;
                    cut = top - l0;
                    fitb = total - __shfl_sync(kFull, suf, l0);
                    break;
                }
                acc = __shfl_sync(kFull, suf, 31);
            }
            if (fitb < 0) fitb = total - acc;  // (unreachable: the whole list reaches the excess)
            int m = 0;
            for (int base = cut; base < ne; base += 32) {
                const int s = base + lane;
                m += __popc(__ballot_sync(kFull, s < ne && rq[s].y >= 0));
            }
            const int wh2 = (wh - m + C) % C;
            int k0 = 0, gd = 0;
            long long gone = 0;
            for (int base = cut; base < ne; base += 32) {
                const int s = base + lane;
                const int4 q = s < ne ? rq[s] : make_int4(0, -1, 0, 0);
                const bool live = q.y >= 0;
                const unsigned bl = __ballot_sync(kFull, live);
                if (live) {
                    int slot = wh2 + k0 + __popc(bl & ((1u << lane) - 1u));
                    if (slot >= C) slot -= C;
                    if (q.y == 0) {
                        wq[slot] = make_int2(q.x + G, q.z - G);
                        atomicSub(&hist[q.w], 1);
                        gone += q.x;
                        ++gd;
                    } else {
                        wq[slot] = make_int2(q.x + q.y, q.z);
                    }
                    reinterpret_cast<int *>(rq + s)[1] = -1;
                }
                k0 += __popc(bl);
            }
            src -= warp_sum64(gone);
            nd -= warp_sum32(gd);
            if (pfs >= cut) pfs = -1;
            wh = wh2;
            wc += m;
            nr -= m;
            freeb = nbk - fitb;
            budget = B - nr;
            f1 = 0;
            f2 = nd;
            f3 = src + (long long)nd * G;
            f4 = 0;
            slack = -1;
            pf_run = false;
        }
        __syncwarp();
        if (pf_run) {
            // the prefill request's chunk; at its last chunk it turns decoder
            const int r = pfs;
            const int cx = pq.x + px, pre = pq.y - px;
            int dec = pq.z;
            if (pre == 0 && MODE == 1) dec -= 1;
            if (pre > 0) {
                if (lane == 0) rq[r] = make_int4(cx, pre, dec, pq.w + pneed);
            } else if (dec <= 0 || (long long)cx >= mctx) {
                if (lane == 0) reinterpret_cast<int *>(rq + r)[1] = -1;
                back += pq.w + pneed;
                ++dying;
                pfs = -1;
            } else {
                const int4 q = make_int4(cx - (G + 1), 0, dec + (G + 1), dres(dv, cx - (G + 1)));
                if (lane == 0) {
                    rq[r] = q;
                    hist[q.w] += 1;
                    file(r, q, G);
                }
                src += q.x;
                ++nd;
                pfs = -1;
            }
        }
        __syncwarp();
        const int bar = budget;
        const long long far = freeb;
        long long f4l = 0;      // this lane's whole admissions' F4 terms
        bool admitted = false;  // any whole admission this batch
        // 2. Admission from the waiting front while budget, a seat and the first chunk's
        //    blocks allow: the prompts that fit whole are a prefix (lane i tests the
        //    i-th waiting request), then possibly one partial chunk.  An admitted
        //    request's chunk is applied at once; one that prefills whole decodes from
        //    the next batch.
        // FCFS: a head whose first chunk's blocks are not free admits nobody (the
        // usual case while a queue waits on a full cache)
        bool adm = budget > 0 && wc > 0 && nr < S;
        if (adm) adm = dblk(dv, min(wq[wh].x, budget)) <= freeb;
        while (adm && budget > 0 && wc > 0 && nr < S) {
            if (ne + 32 > C) compact();
            const bool in = lane < wc && lane < S - nr;
            int slot = wh + lane;
            if (slot >= C) slot -= C;
            const int2 wv = in ? wq[slot] : make_int2(0, 0);
            const int hb_i = in ? dblk(dv, wv.x) : 0;
            const int cp = warp_incl_sum32(wv.x, lane);  // 32 prompts of at most 2^24 tokens
            const int cb = warp_incl_sum32(hb_i, lane);
            const bool whole = in && cp <= budget && (long long)cb <= freeb;
            const int k = __popc(__ballot_sync(kFull, whole));
            const int dec_a = wv.y - (MODE == 1 ? 1 : 0);
            const bool ends = whole && (dec_a <= 0 || (long long)wv.x >= mctx);
            if (whole) {
                const int s = ne + lane;
                const int4 q = make_int4(wv.x - (G + 1), ends ? -1 : 0, dec_a + (G + 1), dres(dv, wv.x - (G + 1)));
                rq[s] = q;
                if (!ends) {
                    atomicAdd(&hist[q.w], 1);
                    file(s, q, G);
                }
                f4l += (long long)wv.x * (wv.x + 1) / 2;
            }
            const unsigned em = __ballot_sync(kFull, ends);
            if (k > 0) {
                const int sp = __shfl_sync(kFull, cp, k - 1), sb = __shfl_sync(kFull, cb, k - 1);
                f1 += sp;
                admitted = true;
                src += sp - (long long)k * (G + 1);
                nd += k;
                if (em) {
                    src -= warp_sum64(ends ? (long long)wv.x - (G + 1) : 0);
                    back += warp_sum64(ends ? (long long)hb_i : 0);
                    dying += __popc(em);
                    nd -= __popc(em);
                }
                budget -= sp;
                freeb -= sb;
                nr += k;
                ne += k;
                wh = wh + k >= C ? wh + k - C : wh + k;
                wc -= k;
            }
            __syncwarp();
            if (k < 32) {
                if (budget > 0 && wc > 0 && nr < S) {
                    const int2 hv = wq[wh];
                    const int x = min(hv.x, budget);
                    const int nb1 = dblk(dv, x);
                    if (x < hv.x && nb1 <= freeb) {
                        if (lane == 0) rq[ne] = make_int4(x, hv.x - x, hv.y, nb1);
                        pfs = ne;
                        f1 += x;
                        f4 += (long long)x * (x + 1) / 2;
                        ++nr;
                        ++ne;
                        wh = wh + 1 >= C ? wh + 1 - C : wh + 1;
                        --wc;
                        budget -= x;
                        freeb -= nb1;
                    }
                }
                break;
            }
        }
        __syncwarp();
        const bool qcan = wc == 0;
        if (la0 == 0 && qcan && budget > 0 && nr < S) la0 = l;
        // 3. The batch's record, or the features before the first record.
        if (la0 != 0 && admitted) f4 += warp_sum64(f4l);
        if (la0 != 0) {
            cf1 += f1;
            cf2 += f2;
            cf3 += f3;
            cf4 += f4;
            // the largest prompt p admitted now: min(p, bl) tokens need at most fa blocks
            long long thr = 0;
            if (qcan && budget > 0 && nr < S) thr = ((long long)budget <= freeb * bs) ? kHuge : freeb * bs;
            pmx = (int)max((long long)pmx, min(thr, (long long)INT32_MAX));
            if (lane == 0) {
                KvRec R;
                R.cf[0] = cf1;
                R.cf[1] = cf2;
                R.cf[2] = cf3;
                R.cf[3] = cf4;
                R.slack = slack;
                R.far = far;
                R.thr = thr;
                R.bar = bar;
                R.bl = budget;
                rec[nrec] = R;
                pmxo[nrec] = pmx;
            }
            ++nrec;
        } else {
            fcum[0] += 1;
            fcum[1] += f1;
            fcum[2] += f2;
            fcum[3] += f3;
            fcum[4] += f4;
            f4c += f4l;  // summed over the warp at the end
        }
        // 4. The decoders whose last batch this is leave and return their blocks.
        {
            int s = head[G & (kKvCal - 1)];
            while (s >= 0) {
                const int ns = nxt[s];
                const int4 q = rq[s];
                if (q.y == 0) {  // a hole is a request preempted after it was filed
                    back += eb[s];
                    ++dying;
                    src -= q.x;
                    --nd;
                    if (lane == 0) {
                        hist[q.w] -= 1;
                        reinterpret_cast<int *>(rq + s)[1] = -1;
                    }
                }
                s = ns;
            }
            __syncwarp();
            if (lane == 0) head[G & (kKvCal - 1)] = -1;
        }
        nr -= dying;
        freeb += back;
        G = G + 1;
        gr = gr + 1 == bs ? 0 : gr + 1;
        __syncwarp();
        if (nr == 0 && wc == 0) {  // no resident left: every later batch is empty
            if (la0 == 0) la0 = l + 1;
            done = 1;
            break;
        }
        if (nrec == a.kv.horizon) break;
        if (ne - nr >= max(32, nr)) compact();
    }
    fcum[4] += warp_sum64(f4c);
    if (lane == 0) {
        KvInst hd;
        for (int k = 0; k < 5; ++k) hd.fcum[k] = fcum[k];
        hd.la0 = la0;
        hd.nrec = nrec;
        hd.done = done;
        hd.pad = 0;
        out.kvi[j] = hd;
    }
}

template <int MODE>
__global__ void __launch_bounds__(kKvWarps * 32) k_kv_load(const KvLoad a) {
    extern __shared__ __align__(16) int32_t kv_smem[];
    const int lane = threadIdx.x & 31;
    const int wid = threadIdx.x >> 5;
    const int j = blockIdx.x * (int)(blockDim.x >> 5) + wid;
    __shared__ int s_active;
    if (threadIdx.x == 0) s_active = load_acquire(&a.ctl->active);
    __syncthreads();
    const int dst = (s_active == 0) ? 1 : 0;
    const StateBuf out = dst ? a.buf1 : a.buf0;
    const size_t per_warp = kv_smem_per_warp(a.cfg, a.kv.hist) / sizeof(int32_t);
    if (j < a.cfg.I) kv_instance<MODE>(a, out, j, lane, kv_smem + wid * per_warp);
    // the last CTA to finish publishes the new snapshot if every instance succeeded
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

constexpr float kNaN = __builtin_nanf("");
constexpr int kEstGroup = 32;   // instances per CTA
constexpr int kEstWarps = 8;    // warps per CTA
// leading records of each instance staged in shared memory: on pool256, 99.3% of the
// candidates reach their first token within 64 records (88% within 16)
constexpr int kEstStage = 52;
// the staged fields of the walk: slack, far, thr (8 bytes), bar, bl, admission maximum (4)
constexpr size_t kEstStageBytes = (size_t)kEstGroup * kEstStage * (3 * 8 + 3 * 4);
// and each warp's tile of 32 later records (slack, far, thr, bar, bl); three CTAs with
// their views fit an SM
constexpr size_t kEstTileBytes = 32 * (3 * 8 + 2 * 4);
constexpr size_t kEstSmem = kEstStageBytes + kEstWarps * kEstTileBytes;

// The walk's fields of an instance's leading records, in shared memory.
struct KvStage {
    long long *slack, *far, *thr;
    int32_t *bar, *bl, *pmx;
};
__device__ __forceinline__ KvStage kv_stage(unsigned char *smem, int g) {
    KvStage st;
    long long *b64 = reinterpret_cast<long long *>(smem) + (size_t)g * 3 * kEstStage;
    st.slack = b64;
    st.far = b64 + kEstStage;
    st.thr = b64 + 2 * kEstStage;
    int32_t *b32 = reinterpret_cast<int32_t *>(reinterpret_cast<long long *>(smem) + (size_t)kEstGroup * 3 * kEstStage) +
                   (size_t)g * 3 * kEstStage;
    st.bar = b32;
    st.bl = b32 + kEstStage;
    st.pmx = b32 + 2 * kEstStage;
    return st;
}

// One instance as the estimate reads it: the first `ns` records (with their admission
// maxima) from shared memory; later records through the warp's tile, and their
// admission maxima and the residents' features from global memory.
struct KvView {
    const KvRec *rec;
    const int32_t *pmx;
    long long fcum[5];
    long long nb, mctx;
    float b[5];
    int la0, nrec, ns, done, B, bs;
    Div32 dv;  // division by bs
};

// A warp's tile of 32 consecutive records past the staged ones (the walk's fields).
struct KvTile {
    long long *slack, *far, *thr;
    int32_t *bar, *bl;
};
__device__ __forceinline__ KvTile kv_tile(unsigned char *smem, int w) {
    KvTile tl;
    tl.slack = reinterpret_cast<long long *>(smem + kEstStageBytes + (size_t)w * kEstTileBytes);
    tl.far = tl.slack + 32;
    tl.thr = tl.far + 32;
    tl.bar = reinterpret_cast<int32_t *>(tl.thr + 32);
    tl.bl = tl.bar + 32;
    return tl;
}

// first index in [lo, lo + n) whose value is >= p, in a nondecreasing array
__device__ __forceinline__ int kv_lower_bound(const int32_t *a, int lo, int n, int p) {
    while (n > 0) {
        const int half = n >> 1;
        if (a[lo + half] < p) {
            lo += half + 1;
            n -= half + 1;
        } else {
            n = half;
        }
    }
    return lo;
}

// A candidate's walk: whether it runs, its prefill left, its context, the blocks it
// holds and its own Eq. 9 features so far.
struct KvWalk {
    bool run;
    int pre, ctx, held;
    long long o1, o2, o3, o4;
};

// One batch (record) of a candidate's walk; true if its first token falls in it.  A
// running query is preempted if the residents' scan leaves a slack below its blocks,
// or if its own tokens need more blocks than are free to it (it is the last running
// request: it preempts itself); a preempted query recomputes its whole context and may
// be readmitted in the same batch.  Token counts stay below p + 2 <= 2^31.
template <int MODE>
__device__ __forceinline__ bool kv_step(KvWalk &w, const Div32 &dv, long long slack, long long far, long long thr,
                                        int bar, int bl) {
    if (w.run) {
        if (slack < w.held) {  // a resident needs the query's blocks
            w.pre += w.ctx;
            w.ctx = 0;
            w.held = 0;
            w.run = false;
        } else if (bar > 0) {
            const int x = w.pre > 0 ? min(w.pre, bar) : 1;
            const int nh = dblk(dv, w.ctx + x);
            if (nh > far) {  // its own tokens do not fit: it preempts itself
                w.pre += w.ctx;
                w.ctx = 0;
                w.held = 0;
                w.run = false;
            } else {
                w.held = nh;
                if (w.pre > 0) {
                    w.o1 += x;
                    w.o4 += (long long)x * w.ctx + (long long)x * (x + 1) / 2;
                    w.ctx += x;
                    w.pre -= x;
                    return w.pre == 0 && MODE == 1;
                }
                w.o2 += 1;
                w.o3 += w.ctx;
                return true;
            }
        } else {
            return false;  // no budget reached the query this batch
        }
    }
    if (w.pre <= thr) {  // admission (pre == p while waiting)
        const int x = min(w.pre, bl);
        w.held = dblk(dv, x);
        w.o1 += x;
        w.o4 += (long long)x * (x + 1) / 2;
        w.ctx = x;
        w.pre -= x;
        w.run = true;
        return w.pre == 0 && MODE == 1;
    }
    return false;
}

// The (query, instance) candidates of a warp's lanes (one instance, `live`: the lane
// has one), called by all 32 lanes: each candidate's features and first-token record,
// or an error.  The query waits (pre = p) until the first record whose admission bound
// reaches p, found by binary search over the bounds' running maximum (the staged part
// in shared memory, the rest in global memory), and is followed from there record by
// record to its first token: through the staged records alone, then through the warp's
// tile, which holds the 32 records from the least one a lane still needs (one load of
// 32 records for the warp instead of one dependent load per record and lane).
template <int MODE>
__device__ int kv_candidate(const KvView &v, const KvStage &st, const KvTile &tl, int lane, bool live, int p,
                            long long F[5], int &lt) {
    int err = 0, t = 0;
    KvWalk w = {false, p, 0, 0, 0, 0, 0, 0};
    bool fin = !live;
    if (live) {
        int lo;
        if (v.ns > 0 && st.pmx[v.ns - 1] >= p) lo = kv_lower_bound(st.pmx, 0, v.ns, p);
        else lo = kv_lower_bound(v.pmx, v.ns, v.nrec - v.ns, p);
        if (lo == v.nrec && !v.done) {
            err = kETraj;
            fin = true;
        }
        for (t = lo; !fin && t < v.ns;) {
            if (kv_step<MODE>(w, v.dv, st.slack[t], st.far[t], st.thr[t], st.bar[t], st.bl[t])) fin = true;
            else ++t;
        }
    }
    // after the records the instance is empty; the query then needs at most
    // ceil(p / B) + 2 batches
    const int limit = live ? v.nrec + (v.done ? (p / v.B + 3) : 0) : 0;
    for (;;) {
        if (__ballot_sync(kFull, !fin) == 0u) break;
        const int base = __reduce_min_sync(kFull, fin ? 0x7fffffff : t);  // >= ns
        {
            const int r = base + lane;
            long long sl = kHuge, fa = v.nb, th = kHuge;  // past the records: an empty batch
            int ba = v.B, bb = v.B;
            if (r < v.nrec) {
                const KvRec *rr = v.rec + r;
                sl = __ldg(&rr->slack);
                fa = __ldg(&rr->far);
                th = __ldg(&rr->thr);
                ba = __ldg(&rr->bar);
                bb = __ldg(&rr->bl);
            }
            tl.slack[lane] = sl;
            tl.far[lane] = fa;
            tl.thr[lane] = th;
            tl.bar[lane] = ba;
            tl.bl[lane] = bb;
        }
        __syncwarp();
        while (!fin && t < base + 32) {
            if (t >= limit) {
                err = kETraj;
                fin = true;
                break;
            }
            const int k = t - base;
            if (kv_step<MODE>(w, v.dv, tl.slack[k], tl.far[k], tl.thr[k], tl.bar[k], tl.bl[k])) fin = true;
            else ++t;
        }
        __syncwarp();  // the tile is read before the next one is written
    }
    if (!live || err) return err;
    lt = t;
    const int tc = min(t, v.nrec - 1);
    long long cf[4] = {0, 0, 0, 0};
    if (tc >= 0) {
        const KvRec *r = v.rec + tc;
        for (int k = 0; k < 4; ++k) cf[k] = __ldg(&r->cf[k]);
    }
    F[0] = v.fcum[0] + t + 1;
    F[1] = v.fcum[1] + cf[0] + w.o1;
    F[2] = v.fcum[2] + cf[1] + w.o2;
    F[3] = v.fcum[3] + cf[2] + w.o3;
    F[4] = v.fcum[4] + cf[3] + w.o4;
    return 0;
}

// The call's queries sorted by prompt length, by a counting sort over buckets:
// bucket 0 holds the invalid lengths, bucket 1 + ((p - 1) >> shift) the valid ones.
// A candidate depends on the instance and p alone, so with shift 0 (one bucket per
// length) the estimate runs once per distinct length, on the bucket's first query
// (its leader), and k_kv_expand copies the leader's rows to the bucket's other
// queries; with a coarser shift every query is estimated, in sorted order, which
// keeps the lanes of a warp on near-equal walks through the records.
__device__ __forceinline__ int kv_bucket(int p, int pmax, int shift) {
    return (p >= 1 && p <= pmax) ? 1 + ((p - 1) >> shift) : 0;
}

__global__ void __launch_bounds__(256) k_kv_count(const int32_t *prompt, int Q, int pmax, int shift, int32_t *cnt) {
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < Q; i += gridDim.x * blockDim.x) {
        const int b = kv_bucket(prompt[i], pmax, shift);
        const unsigned m = __match_any_sync(__activemask(), b);
        if ((threadIdx.x & 31) == __ffs(m) - 1) atomicAdd(&cnt[b], __popc(m));
    }
}

// One CTA: start = run = exclusive prefix sums of the counts, uid = the number of
// non-empty buckets before each one, nu = their total; the counts are cleared for
// the next call, and the estimate's block counters too.  Tiles of 4096 buckets,
// four per thread as one 16-byte word.
constexpr int kScanThreads = 1024;
static_assert(kKvBuckets == kKvScanTiles * 4 * kScanThreads, "scan tiles cover the buckets");
// The bucket scan in two launches, one CTA per tile of 4,096 buckets: the tiles'
// sums (count and non-empty buckets), then each tile's exclusive scan from the sums of
// the tiles before it.  (One CTA over every bucket was bound by one SM's bandwidth.)
__global__ void __launch_bounds__(kScanThreads) k_kv_tile_sums(const int32_t *cnt, int32_t *tsum, int32_t *claim,
                                                               int groups) {
    __shared__ int ws[2][kScanThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    if (blockIdx.x == 0)
        for (int g = tid; g < groups; g += kScanThreads) claim[g] = 0;
    const int4 v = reinterpret_cast<const int4 *>(cnt)[blockIdx.x * kScanThreads + tid];
    int sc = v.x + v.y + v.z + v.w;
    int su = (v.x > 0) + (v.y > 0) + (v.z > 0) + (v.w > 0);
    sc = warp_sum32(sc);
    su = warp_sum32(su);
    if (lane == 0) {
        ws[0][w] = sc;
        ws[1][w] = su;
    }
    __syncthreads();
    if (w == 0) {
        const int xc = warp_sum32(ws[0][lane]), xu = warp_sum32(ws[1][lane]);
        if (lane == 0) {
            tsum[2 * blockIdx.x] = xc;
            tsum[2 * blockIdx.x + 1] = xu;
        }
    }
}

__global__ void __launch_bounds__(kScanThreads) k_kv_scan(int32_t *cnt, int32_t *start, int32_t *run, int32_t *uid,
                                                          int32_t *nu, const int32_t *tsum) {
    __shared__ int ws[2][kScanThreads / 32];
    __shared__ int base[2];
    const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
    if (tid == 0) {  // the tiles before this one
        int c = 0, u = 0;
        for (int t = 0; t < (int)blockIdx.x; ++t) {
            c += tsum[2 * t];
            u += tsum[2 * t + 1];
        }
        base[0] = c;
        base[1] = u;
        if (blockIdx.x == gridDim.x - 1) *nu = u + tsum[2 * blockIdx.x + 1];
    }
    const int b = (blockIdx.x * kScanThreads + tid) * 4;
    const int4 v = reinterpret_cast<const int4 *>(cnt)[b / 4];
    const int sc = v.x + v.y + v.z + v.w;
    const int su = (v.x > 0) + (v.y > 0) + (v.z > 0) + (v.w > 0);
    const int ic = warp_incl_sum32(sc, lane), iu = warp_incl_sum32(su, lane);
    if (lane == 31) {
        ws[0][w] = ic;
        ws[1][w] = iu;
    }
    __syncthreads();
    if (w == 0) {
        const int xc = ws[0][lane], xu = ws[1][lane];
        const int yc = warp_incl_sum32(xc, lane), yu = warp_incl_sum32(xu, lane);
        ws[0][lane] = yc - xc;
        ws[1][lane] = yu - xu;
    }
    __syncthreads();
    int oc = base[0] + ws[0][w] + ic - sc, ou = base[1] + ws[1][w] + iu - su;
    int4 so, uo;
    so.x = oc;
    uo.x = ou;
    oc += v.x;
    ou += v.x > 0;
    so.y = oc;
    uo.y = ou;
    oc += v.y;
    ou += v.y > 0;
    so.z = oc;
    uo.z = ou;
    oc += v.z;
    ou += v.z > 0;
    so.w = oc;
    uo.w = ou;
    reinterpret_cast<int4 *>(start)[b / 4] = so;
    reinterpret_cast<int4 *>(run)[b / 4] = so;
    reinterpret_cast<int4 *>(uid)[b / 4] = uo;
    reinterpret_cast<int4 *>(cnt)[b / 4] = make_int4(0, 0, 0, 0);
}

__global__ void __launch_bounds__(256) k_kv_scatter(const int32_t *prompt, int Q, int pmax, int shift, int32_t *run,
                                                    const int32_t *start, const int32_t *uid, int32_t *order,
                                                    int32_t *leaders) {
    const int lane = threadIdx.x & 31;
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < Q; i += gridDim.x * blockDim.x) {
        const int b = kv_bucket(prompt[i], pmax, shift);
        const unsigned act = __activemask();
        const unsigned m = __match_any_sync(act, b);
        const int lead = __ffs(m) - 1;
        int base = 0;
        if (lane == lead) base = atomicAdd(&run[b], __popc(m));
        base = __shfl_sync(m, base, lead);
        const int pos = base + __popc(m & ((1u << lane) - 1u));
        order[pos] = i;
        if (pos == start[b]) leaders[uid[b]] = i;
    }
}

// One warp per query row: a query that is not its bucket's leader copies the
// leader's rows (times, and first batches and features if asked for).
__global__ void __launch_bounds__(256) k_kv_expand(const KvEst a) {
    const int I = a.cfg.I, lane = threadIdx.x & 31;
    const int warps = gridDim.x * (blockDim.x >> 5);
    const bool v4 = I % 4 == 0 && (reinterpret_cast<uintptr_t>(a.ttft) & 15) == 0;
    const bool f2 = I % 2 == 0 && (reinterpret_cast<uintptr_t>(a.features) & 15) == 0;
    for (int i = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); i < a.Q; i += warps) {
        const int L = a.order[a.start[kv_bucket(a.prompt[i], a.cfg.pmax, 0)]];
        if (L == i) continue;
        const size_t ri = (size_t)i * I, rl = (size_t)L * I;
        if (a.ttft) {
            if (v4) {
                const float4 *src = reinterpret_cast<const float4 *>(a.ttft + rl);
                float4 *dst = reinterpret_cast<float4 *>(a.ttft + ri);
                for (int c = lane; c < I / 4; c += 32) dst[c] = src[c];
            } else {
                for (int c = lane; c < I; c += 32) a.ttft[ri + c] = a.ttft[rl + c];
            }
        }
        if (a.first_batch)
            for (int c = lane; c < I; c += 32) a.first_batch[ri + c] = a.first_batch[rl + c];
        if (a.features) {
            if (f2) {
                const int4 *src = reinterpret_cast<const int4 *>(a.features + rl * 5);
                int4 *dst = reinterpret_cast<int4 *>(a.features + ri * 5);
                for (int c = lane; c < I * 5 / 2; c += 32) dst[c] = src[c];
            } else {
                for (int c = lane; c < I * 5; c += 32) a.features[ri * 5 + c] = a.features[rl * 5 + c];
            }
        }
    }
}

// CTA: kEstGroup instances (strided over the pool), the walk's fields of their
// leading records staged in shared memory.  The CTAs of a group claim units of (32 queries, one instance),
// the longest prompts first, so the longest walks start first and no warp holds
// more than one instance's walks of one block.
template <int MODE>
__global__ void __launch_bounds__(kEstWarps * 32, 3) k_kv_estimate(const KvEst a, bool exact) {
    extern __shared__ __align__(16) unsigned char est_smem[];
    __shared__ KvView sv[kEstGroup];
    const DevConfig &c = a.cfg;
    const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
    // group y holds instances y, y + gy, y + 2 gy, ... (gy groups): every group mixes the
    // pool's models, whose walks differ in length, so the groups' work is alike
    const int gy = gridDim.y;
    const int ng = min(kEstGroup, (c.I - (int)blockIdx.y + gy - 1) / gy);
    const int active = load_acquire(&a.ctl->active);
    // the group's views, a thread each
    if ((int)threadIdx.x < ng) {
        const int gw = threadIdx.x;
        const int j = gw * gy + blockIdx.y;
        KvView v;
        v.nb = a.kv.nb[j];
        v.mctx = a.kv.mctx[j];
        v.bs = a.kv.bs[j];
        v.dv = make_div32(v.bs);
        v.B = c.B[j];
        const float *cf = c.coef + 5 * c.moi[j];
        for (int k = 0; k < 5; ++k) v.b[k] = cf[k];
        v.ns = 0;
        v.nrec = 0;
        if (active >= 0) {
            const StateBuf sb = active ? a.buf1 : a.buf0;
            const KvInst hd = sb.kvi[j];
            for (int k = 0; k < 5; ++k) v.fcum[k] = hd.fcum[k];
            v.la0 = hd.la0;
            v.nrec = hd.nrec;
            v.done = hd.done;
            v.rec = sb.kvr + (size_t)j * a.kv.horizon;
            v.pmx = sb.kvp + (size_t)j * a.kv.horizon;
            v.ns = min(v.nrec, kEstStage);
        }
        sv[gw] = v;
    }
    __syncthreads();
    // the walk's fields of the instances' leading records, staged by every thread of the
    // CTA in rounds whose loads are all issued before their stores
    if (active >= 0) {
        constexpr int kRound = 4;
        constexpr int kAll = kEstGroup * kEstStage;
        for (int r0 = 0; r0 < kAll; r0 += kRound * kEstWarps * 32) {
            long long f_sl[kRound], f_fa[kRound], f_th[kRound];
            int f_ba[kRound], f_bl[kRound], f_pm[kRound];
#pragma unroll
            for (int k = 0; k < kRound; ++k) {
                const int idx = r0 + (int)threadIdx.x + k * kEstWarps * 32;
                const int gw = idx / kEstStage, t = idx - gw * kEstStage;
                if (gw < ng && t < sv[gw].ns) {
                    const KvRec *r = sv[gw].rec + t;
                    f_sl[k] = __ldg(&r->slack);
                    f_fa[k] = __ldg(&r->far);
                    f_th[k] = __ldg(&r->thr);
                    f_ba[k] = __ldg(&r->bar);
                    f_bl[k] = __ldg(&r->bl);
                    f_pm[k] = __ldg(sv[gw].pmx + t);
                }
            }
#pragma unroll
            for (int k = 0; k < kRound; ++k) {
                const int idx = r0 + (int)threadIdx.x + k * kEstWarps * 32;
                const int gw = idx / kEstStage, t = idx - gw * kEstStage;
                if (gw < ng && t < sv[gw].ns) {
                    const KvStage st = kv_stage(est_smem, gw);
                    st.slack[t] = f_sl[k];
                    st.far[t] = f_fa[k];
                    st.thr[t] = f_th[k];
                    st.bar[t] = f_ba[k];
                    st.bl[t] = f_bl[k];
                    st.pmx[t] = f_pm[k];
                }
            }
        }
    }
    __syncthreads();
    // the work: one query per distinct prompt length, or every query, by length
    const int nwork = exact ? *a.nu : a.Q;
    const int32_t *work = exact ? a.leaders : a.order;
    const int nitems = (nwork + 31) / 32 * ng;
    // Software-pipelined: the claim of the next item and its query's prompt are in
    // flight while the current item is walked.
    auto claim = [&]() {
        int v = 0;
        if (lane == 0) v = atomicAdd(&a.claim[blockIdx.y], 1);
        return __shfl_sync(kFull, v, 0);
    };
    auto fetch = [&](int it_, int &i_, int &p_) {  // this lane's query of item it_ (i_ < 0: none)
        i_ = -1;
        p_ = 0;
        if (it_ < nitems) {
            const int pos_ = nwork - 1 - ((it_ / ng) * 32 + lane);
            if (pos_ >= 0) {
                i_ = work[pos_];
                p_ = a.prompt[i_];
            }
        }
    };
    int it = claim();
    int i_cur, p_cur;
    fetch(it, i_cur, p_cur);
    for (;;) {
        if (it >= nitems) break;
        const int it_next = claim();
        const int qb = it / ng, g = it - qb * ng;
        const int i = i_cur, p = p_cur;
        int i_nx, p_nx;
        fetch(it_next, i_nx, p_nx);
        // every lane of the warp takes part in the walks (their record tiles)
        const KvView &v = sv[g];
        long long F[5] = {-1, -1, -1, -1, -1};
        int lt = -1;
        int err = 0;
        // a query with one output token: its prompt below the context limit and
        // its first token within the instance's blocks
        if (i >= 0) {
            if (active < 0) err = kENoState;
            else if (!(p >= 1 && p <= c.pmax && (long long)p < v.mctx && kv_blocks32(p + 1, v.bs) <= v.nb))
                err = kEInval;
        }
        const int werr = kv_candidate<MODE>(v, kv_stage(est_smem, g), kv_tile(est_smem, w), lane,
                                            i >= 0 && err == 0, p, F, lt);
        if (err == 0) err = werr;
        if (i >= 0) {
            float tt = kNaN;
            if (err) {
                record_status(a.ctl, err);
                for (int k = 0; k < 5; ++k) F[k] = -1;
            } else {
                tt = __fmul_rn(v.b[0], __ll2float_rn(F[0]));
                tt = __fmaf_rn(v.b[2], __ll2float_rn(F[2]), tt);
                tt = __fmaf_rn(v.b[1], __ll2float_rn(F[1]), tt);
                tt = __fmaf_rn(v.b[3], __ll2float_rn(F[3]), tt);
                tt = __fmaf_rn(v.b[4], __ll2float_rn(F[4]), tt);
            }
            const size_t idx = (size_t)i * c.I + g * gy + blockIdx.y;
            if (a.ttft) a.ttft[idx] = tt;
            if (a.first_batch) a.first_batch[idx] = err ? -1 : v.la0 + lt;
            if (a.features)
                for (int k = 0; k < 5; ++k) a.features[idx * 5 + k] = F[k];
        }
        it = it_next;
        i_cur = i_nx;
        p_cur = p_nx;
    }
}

}  // namespace

cudaError_t launch_kv_load(const KvLoad &a, int grid, int warps, size_t smem, cudaStream_t st) {
    if (a.cfg.mode == 0) k_kv_load<0><<<grid, warps * 32, smem, st>>>(a);
    else k_kv_load<1><<<grid, warps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t set_kv_smem(size_t bytes) {
    cudaError_t e = cudaFuncSetAttribute(k_kv_load<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_kv_load<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_kv_estimate<0>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kEstSmem);
    if (e == cudaSuccess)
        e = cudaFuncSetAttribute(k_kv_estimate<1>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kEstSmem);
    return e;
}

cudaError_t launch_kv_estimate(const KvEst &a, int sms, cudaStream_t st) {
    const int gy = (a.cfg.I + kEstGroup - 1) / kEstGroup;
    const int blocks = (a.Q + 32 * kEstWarps - 1) / (32 * kEstWarps);
    const int gx = std::max(1, std::min(blocks, (sms * 3 + gy - 1) / gy));  // three CTAs fit an SM
    const dim3 grid(gx, gy);
    int shift = 0;
    while (2 + ((a.cfg.pmax - 1) >> shift) > kKvBuckets) ++shift;
    const int nbk = 2 + ((a.cfg.pmax - 1) >> shift);
    const bool exact = shift == 0;
    const int g1 = std::max(1, std::min((a.Q + 255) / 256, sms * 4));
    k_kv_count<<<g1, 256, 0, st>>>(a.prompt, a.Q, a.cfg.pmax, shift, a.cnt);
    const int tiles = (nbk + 4095) / 4096;
    k_kv_tile_sums<<<tiles, kScanThreads, 0, st>>>(a.cnt, a.tsum, a.claim, gy);
    k_kv_scan<<<tiles, kScanThreads, 0, st>>>(a.cnt, a.start, a.run, a.uid, a.nu, a.tsum);
    k_kv_scatter<<<g1, 256, 0, st>>>(a.prompt, a.Q, a.cfg.pmax, shift, a.run, a.start, a.uid, a.order, a.leaders);
    if (a.cfg.mode == 0) k_kv_estimate<0><<<grid, kEstWarps * 32, kEstSmem, st>>>(a, exact);
    else k_kv_estimate<1><<<grid, kEstWarps * 32, kEstSmem, st>>>(a, exact);
    if (exact) k_kv_expand<<<std::max(1, std::min((a.Q + 7) / 8, sms * 8)), 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace lr
