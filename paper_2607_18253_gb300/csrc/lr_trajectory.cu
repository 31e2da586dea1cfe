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
// keeps one slot (s, f, cb) per decoder in shared memory and jumps over runs
// of batches in which nothing but decoding happens.
#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;

struct WarpSmem {
    int32_t *s, *f, *cb, *freel, *wpre, *wdec, *rcum;
};

__device__ __forceinline__ WarpSmem carve(int32_t *base, const DevConfig &c) {
    WarpSmem w;
    w.s = base;
    w.f = w.s + c.slots;
    w.cb = w.f + c.slots;
    w.freel = w.cb + c.slots;
    w.wpre = w.freel + c.slots;
    w.wdec = w.wpre + c.capW;
    w.rcum = w.wdec + c.capW;
    return w;
}

// Decoder slots of one instance, manipulated by all 32 lanes in lockstep.
struct Slots {
    WarpSmem m;
    int n;          // slots in use
    int top;        // free-list size
    int fmin;       // smallest last-decode batch over used slots (kBig if none)
    long long f2d;  // this lane's share of decode tokens of finished decoders
    long long f3d;  // ... and of their decode context
    int lane;
    int nslots_cap;
    bool overflow;

    // Drop decoders whose last decode batch is before l; fold their features.
    __device__ void remove_before(int l) {
        int removed = 0;
        int mn = kBig;
        for (int base = 0; base < nslots_cap; base += 32) {
            const int idx = base + lane;
            const int f = m.f[idx];
            const bool rm = f < l;  // free slots hold kBig
            if (rm) {
                const int s = m.s[idx];
                const long long cnt = (long long)f - s + 1;
                f2d += cnt;
                f3d += cnt * (long long)m.cb[idx] + (((long long)s + f) * cnt) / 2;
                m.f[idx] = kBig;
                m.s[idx] = kBig;
            } else {
                mn = min(mn, f);
            }
            const unsigned b = __ballot_sync(kFull, rm);
            if (rm) m.freel[top + __popc(b & lanemask_lt())] = idx;
            top += __popc(b);
            removed += __popc(b);
        }
        __syncwarp();
        fmin = __reduce_min_sync(kFull, mn);
        n -= removed;
    }

    // New decoder: first decode batch s, last decode batch f, context at batch l is cb + l.
    __device__ void insert(int s, int f, int cb) {
        if (top <= 0) {  // more decoders than slots: excluded by the preconditions
            overflow = true;
            return;
        }
        const int idx = m.freel[top - 1];
        --top;
        if (lane == 0) {
            m.s[idx] = s;
            m.f[idx] = f;
            m.cb[idx] = cb;
        }
        fmin = min(fmin, f);
        ++n;
    }

    // Move to batch l: finished decoders leave.
    __device__ void advance_to(int l) {
        __syncwarp();
        if (l > fmin) remove_before(l);
    }
};

// A request finished its prompt in batch e with ce tokens of context and d
// output tokens to produce (Sec. 4.1: decode begins after the prefill).
__device__ __forceinline__ void prefill_done(Slots &sl, int mode, int e, int ce, int d) {
    if (mode == 0) {
        sl.insert(e + 1, e + d, ce - (e + 1));
    } else if (d >= 2) {  // first token sampled with the last chunk
        sl.insert(e + 1, e + d - 1, ce - (e + 1));
    }
}

__device__ void fail(DevCtl *ctl, int code, int lane) {
    if (lane == 0) {
        atomicCAS(&ctl->load_err, 0, code);
        record_status(ctl, code);
    }
}

__device__ void summarize_instance(const K1Launch &a, const StateBuf &out, int j, int lane, int32_t *wbase) {
    const DevConfig &c = a.cfg;
    const int B = c.B[j];
    const int S = c.S[j];
    const int nr = a.in.n_run[j];
    const int nw = a.in.n_wait[j];
    if (lane == 0) {
        out.n_run[j] = nr;
        out.n_wait[j] = nw;
    }
    if (!(nr >= 0 && nr <= c.capR && nr <= S && nw >= 0 && nw <= c.capW)) {
        fail(a.ctl, kEState, lane);
        return;
    }
    WarpSmem m = carve(wbase, c);
    const size_t rrow = (size_t)j * c.capR;
    const size_t wrow = (size_t)j * c.capW;

    // Copy the snapshot into library memory, validate it and total the prefill work.
    bool bad = false;
    long long f1 = 0, f4 = 0;
    for (int t = lane; t < c.capR; t += 32) {
        const int ctx = a.in.run_ctx[rrow + t];
        const int pre = a.in.run_pre[rrow + t];
        const int dec = a.in.run_dec[rrow + t];
        out.run_ctx[rrow + t] = ctx;
        out.run_pre[rrow + t] = pre;
        out.run_dec[rrow + t] = dec;
        if (t < nr) {
            bad |= ctx < 0 || ctx > (1 << 28) || pre < 0 || pre > (1 << 24) || dec < 1 || dec > (1 << 24);
            bad |= pre > 0 && t != nr - 1;
            f1 += pre;
            f4 += (long long)pre * ctx + ((long long)pre * (pre + 1)) / 2;
        }
    }
    for (int t = lane; t < c.capW; t += 32) {
        const int pre = a.in.wait_pre[wrow + t];
        const int dec = a.in.wait_dec[wrow + t];
        out.wait_pre[wrow + t] = pre;
        out.wait_dec[wrow + t] = dec;
        m.wpre[t] = pre;
        m.wdec[t] = dec;
        if (t < nw) {
            bad |= pre < 1 || pre > (1 << 24) || dec < 1 || dec > (1 << 24);
            f1 += pre;
            f4 += ((long long)pre * (pre + 1)) / 2;
        }
    }
    if (__any_sync(kFull, bad)) {
        fail(a.ctl, kEState, lane);
        return;
    }
    f1 = warp_sum64(f1);
    f4 = warp_sum64(f4);

    // Decoder slots: running request t (decoding from batch 1) takes slot t.
    for (int idx = lane; idx < c.slots; idx += 32) {
        int s = kBig, f = kBig, cb = 0;
        if (idx < nr) {
            const int pre = a.in.run_pre[rrow + idx];
            if (pre == 0) {
                s = 1;
                f = a.in.run_dec[rrow + idx];
                cb = a.in.run_ctx[rrow + idx] - 1;
            }
        }
        m.s[idx] = s;
        m.f[idx] = f;
        m.cb[idx] = cb;
    }
    __syncwarp();
    Slots sl;
    sl.m = m;
    sl.lane = lane;
    sl.nslots_cap = c.slots;
    sl.f2d = 0;
    sl.f3d = 0;
    sl.top = 0;
    sl.n = 0;
    sl.overflow = false;
    int mn = kBig;
    for (int base = 0; base < c.slots; base += 32) {
        const int idx = base + lane;
        const int f = m.f[idx];
        const bool fr = f == kBig;
        const unsigned b = __ballot_sync(kFull, fr);
        if (fr) m.freel[sl.top + __popc(b & lanemask_lt())] = idx;
        sl.top += __popc(b);
        sl.n += 32 - __popc(b);
        if (!fr) mn = min(mn, f);
    }
    __syncwarp();
    sl.fmin = __reduce_min_sync(kFull, mn);

    // The request still in prefill, if any (always the last running one).
    bool pf = false;
    int pfR = 0, pfC = 0, pfD = 0;
    if (nr > 0) {
        const int pre = a.in.run_pre[rrow + nr - 1];
        if (pre > 0) {
            pf = true;
            pfR = pre;
            pfC = a.in.run_ctx[rrow + nr - 1];
            pfD = a.in.run_dec[rrow + nr - 1];
        }
    }

    const int mode = c.mode;
    int l = 1, head = 0, iters = 0;
    bool found = false;
    int la = 0, r0 = 0;
    while (iters < c.max_iters && l < (1 << 30)) {
        ++iters;
        int cnt = sl.n + (pf ? 1 : 0);  // requests running in batch l
        if (!pf && cnt >= S) {
            // Every sequence slot is taken: nothing but decoding until one frees.
            l = sl.fmin + 1;
            sl.advance_to(l);
            continue;
        }
        int budget = B - sl.n;  // every decoder takes one token first
        if (pf) {
            if (budget <= 0) break;  // excluded by the preconditions
            if (pfR > budget) {
                // The prefill continues; skip the batches in which it cannot
                // finish and the number of decoders stays the same.
                const int m1 = (pfR - 1) / budget;
                const int m2 = (sl.fmin == kBig) ? kBig : (sl.fmin + 1 - l);
                const int step = min(m1, m2);
                pfR -= step * budget;
                pfC += step * budget;
                l += step;
                sl.advance_to(l);
                continue;
            }
            budget -= pfR;
            pfC += pfR;
            pfR = 0;
            pf = false;
            prefill_done(sl, mode, l, pfC, pfD);
        }
        // FCFS admission while budget and a sequence slot remain.
        while (budget > 0 && head < nw && cnt < S) {
            const int p = m.wpre[head];
            const int d = m.wdec[head];
            ++head;
            ++cnt;
            if (p <= budget) {
                budget -= p;
                prefill_done(sl, mode, l, p, d);
            } else {
                pf = true;
                pfR = p - budget;
                pfC = budget;
                pfD = d;
                budget = 0;
            }
        }
        if (!pf && head == nw && budget > 0 && cnt < S) {
            found = true;
            la = l;
            r0 = budget;
            break;
        }
        ++l;
        sl.advance_to(l);
    }
    __syncwarp();
    if (!found || sl.overflow) {
        fail(a.ctl, kETraj, lane);
        return;
    }

    // Budgets left to the query after its admission batch: cumulative sums until
    // they cover the longest prompt.
    int kp = 1;
    long long rc = r0;
    if (lane == 0) m.rcum[0] = r0;
    while (rc < c.pmax && kp < c.kph) {
        const int lk = la + kp;
        int nd = 0;
        for (int idx = lane; idx < c.slots; idx += 32) nd += (m.s[idx] <= lk && lk <= m.f[idx]) ? 1 : 0;
        nd = __reduce_add_sync(kFull, nd);
        rc += B - nd;
        if (lane == 0) m.rcum[kp] = (int)min(rc, (long long)kBig - 1);
        ++kp;
    }
    __syncwarp();
    if (rc < c.pmax) {
        fail(a.ctl, kETraj, lane);
        return;
    }

    // Residents' decode features up to each batch the query's first token can fall in.
    const int off = (mode == 0) ? 1 : 0;
    const long long f2done = warp_sum64(sl.f2d);
    const long long f3done = warp_sum64(sl.f3d);
    const int m_j = c.moi[j];
    const float b0 = c.coef[m_j * 5 + 0];
    const float b1d = c.coef[m_j * 5 + 2];
    const long long ppmax = ((long long)c.pmax * (c.pmax + 1)) / 2;
    bool fast = (f1 + c.pmax < kFastLimit) && (f4 + ppmax < kFastLimit);
    const long long lowmask = (1LL << kSplitBits) - 1;
    for (int k = 0; k < kp; ++k) {
        const int L = la + k + off;
        long long a2 = 0, a3 = 0;
        for (int idx = lane; idx < c.slots; idx += 32) {
            const int s = m.s[idx];
            if (s <= L) {
                const int e = min(m.f[idx], L);
                const long long cnt = (long long)e - s + 1;
                a2 += cnt;
                a3 += cnt * (long long)m.cb[idx] + (((long long)s + e) * cnt) / 2;
            }
        }
        const long long F2 = f2done + warp_sum64(a2) + off;  // + the query's own first decode token
        const long long F3 = f3done + warp_sum64(a3);
        fast = fast && (F3 + c.pmax < kFastLimit);
        if (lane == (k & 31)) {
            const float t = __fmaf_rn(b1d, __ll2float_rn(F2), __fmul_rn(b0, __int2float_rn(L)));
            const long long lo = F3 & lowmask;
            float4 e;
            e.x = t;
            e.y = __ll2float_rn(F3 - lo);
            e.z = __ll2float_rn(lo);
            e.w = __ll2float_rn(F3);
            const size_t o = (size_t)k * c.I + j;
            out.ent[o] = e;
            out.f2[o] = F2;
            out.f3[o] = F3;
            out.rcum[o] = m.rcum[k];
        }
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
    }
}

__global__ void __launch_bounds__(kK1Warps * 32) k_trajectory(const K1Launch a) {
    extern __shared__ int32_t k1_smem[];
    const int lane = threadIdx.x & 31;
    const int wid = threadIdx.x >> 5;
    const int j = blockIdx.x * kK1Warps + wid;
    const int active = *((volatile int32_t *)&a.ctl->active);
    const int dst = (active == 0) ? 1 : 0;
    const StateBuf out = dst ? a.buf1 : a.buf0;
    const size_t per_warp = trajectory_smem_per_warp(a.cfg) / sizeof(int32_t);
    if (j < a.cfg.I) summarize_instance(a, out, j, lane, k1_smem + wid * per_warp);

    // The last CTA to finish publishes the new snapshot if every instance succeeded.
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const unsigned prev = atomicAdd(&a.ctl->done_ctas, 1u);
        if (prev == gridDim.x - 1) {
            __threadfence();
            const int err = atomicExch(&a.ctl->load_err, 0);
            if (err == 0) atomicExch(&a.ctl->active, dst);
            atomicExch(&a.ctl->done_ctas, 0u);
            __threadfence();
        }
    }
}

}  // namespace

cudaError_t launch_trajectory(const K1Launch &a, int grid, int block, size_t smem, cudaStream_t st) {
    k_trajectory<<<grid, block, smem, st>>>(a);
    return cudaGetLastError();
}

cudaError_t set_k1_smem(size_t bytes) {
    return cudaFuncSetAttribute(k_trajectory, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

}  // namespace lr
