// KV-limited Serving Framework Simulation (Sec. 4.1 with App. F's "context limits,
// KV-cache allocation state, and preemption behavior").
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
// admitted what q's fate depends on: the budget, seats and free blocks left to it,
// the least block slack of the residents' scan (q, holding h blocks, is preempted in
// a batch whose slack is below h) and the residents' Eq. 9 features.  The estimate
// (k_kv_estimate) then follows each (query, instance) candidate through those
// records: waiting, admitted, prefilling chunk by chunk, preempted and readmitted,
// until its first token.
#include "lr_internal.cuh"

namespace lr {

namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr long long kHuge = 1LL << 62;

__device__ __forceinline__ long long kv_blocks(long long c, long long bs) { return (c + bs - 1) / bs; }

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

// One instance's residents alone, batch by batch, from the snapshot.  Every lane
// holds the same scalar state; lane r of a chunk handles running request base + r.
template <int MODE>
__device__ void kv_instance(const KvLoad &a, const StateBuf &out, int j, int lane, int32_t *wb) {
    const DevConfig &c = a.cfg;
    const int B = c.B[j];
    const int S = c.S[j];
    const long long bs = a.kv.bs[j], nbk = a.kv.nb[j], mctx = a.kv.mctx[j];
    const int C = c.capR + c.capW;  // at most this many residents
    int32_t *rctx = wb, *rpre = rctx + C, *rdec = rpre + C, *rx = rdec + C;  // running list, chunk of the batch
    int32_t *wpre = rx + C, *wdec = wpre + C;                                  // waiting ring
    long long *scr = reinterpret_cast<long long *>(wdec + C);                  // [8] lane 0 -> warp
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
    // Copy and validate the snapshot: only the last running request may still be in
    // prefill, no context reaches the limit, every request's whole context fits the
    // instance's blocks, and the running requests' blocks fit together.
    const size_t rrow = (size_t)j * c.capR, wrow = (size_t)j * c.capW;
    bool bad = false;
    long long held = 0;
    for (int t = lane; t < c.capR; t += 32) {
        const int ctx = a.in.run_ctx[rrow + t], pre = a.in.run_pre[rrow + t], dec = a.in.run_dec[rrow + t];
        out.run_ctx[rrow + t] = ctx;
        out.run_pre[rrow + t] = pre;
        out.run_dec[rrow + t] = dec;
        if (t < nr0) {
            bad |= ctx < 0 || ctx > (1 << 28) || pre < 0 || pre > (1 << 24) || dec < 1 || dec > (1 << 24);
            bad |= pre > 0 && t != nr0 - 1;
            bad |= (long long)ctx + pre >= mctx;
            bad |= kv_blocks(min((long long)ctx + pre + dec, mctx), bs) > nbk;
            held += kv_blocks(max(ctx, 0), bs);
            rctx[t] = ctx;
            rpre[t] = pre;
            rdec[t] = dec;
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
            wpre[t] = pre;
            wdec[t] = dec;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) held += __shfl_xor_sync(kFull, held, o);
    if (__any_sync(kFull, bad) || held > nbk) {
        kv_fail(a.ctl, kEState, lane);
        return;
    }
    __syncwarp();

    long long freeb = nbk - held;
    int nr = nr0, wh = 0, wc = nw0;  // running count; waiting ring head and count
    long long fcum[5] = {0, 0, 0, 0, 0};
    int la0 = 0, nrec = 0, done = 0;
    KvRec *rec = out.kvr + (size_t)j * a.kv.horizon;
    for (int l = 1;; ++l) {
        if (l > c.max_iters) {
            kv_fail(a.ctl, kETraj, lane);
            return;
        }
        // 1. The running scan.  n_run <= S <= B and only the last request may be in
        //    prefill, so every request gets its tokens: one per decoder, and the last
        //    one's chunk from what the decoders leave.
        long long need_all = 0;
        for (int base = 0; base < nr; base += 32) {
            const int r = base + lane;
            long long need = 0;
            if (r < nr) {
                const int x = rpre[r] > 0 ? min(rpre[r], B - (nr - 1)) : 1;
                rx[r] = x;
                need = kv_blocks((long long)rctx[r] + x, bs) - kv_blocks(rctx[r], bs);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) need += __shfl_xor_sync(kFull, need, o);
            need_all += need;
        }
        __syncwarp();
        long long slack;
        int budget;
        if (need_all <= freeb) {
            // nobody runs out: the least slack is at the last request
            slack = nr > 0 ? freeb - need_all : kHuge;
            freeb -= need_all;
            budget = nr > 0 ? B - (nr - 1) - rx[nr - 1] : B;
        } else {
            // a request runs out of blocks: the scan as the rule states it, with tail
            // preemptions, on one lane (rare)
            if (lane == 0) {
                long long fb = freeb, sl = kHuge;
                int n = nr, bud = B, r = 0, h = wh, cnt = wc;
                while (r < n && bud > 0) {
                    const int x = rpre[r] > 0 ? min(rpre[r], bud) : 1;
                    const long long need = kv_blocks((long long)rctx[r] + x, bs) - kv_blocks(rctx[r], bs);
                    sl = min(sl, fb - need);
                    while (fb < need && n - 1 >= r) {
                        const int v = n - 1;  // recompute: the whole context becomes prefill
                        fb += kv_blocks(rctx[v], bs);
                        h = (h - 1 + C) % C;
                        wpre[h] = rpre[v] + rctx[v];
                        wdec[h] = rdec[v];
                        ++cnt;
                        --n;
                    }
                    if (r >= n) break;
                    fb -= need;
                    rx[r] = x;
                    bud -= x;
                    ++r;
                }
                scr[0] = n;
                scr[1] = bud;
                scr[2] = fb;
                scr[3] = sl;
                scr[4] = h;
                scr[5] = cnt;
            }
            __syncwarp();
            nr = (int)scr[0];
            budget = (int)scr[1];
            freeb = scr[2];
            slack = scr[3];
            wh = (int)scr[4];
            wc = (int)scr[5];
            __syncwarp();
        }
        const int bar = budget;
        const long long far = freeb;
        // 2. Admission from the waiting front while budget, a seat and the first chunk's
        //    blocks allow: the prompts that fit whole are a prefix (lane i tests the
        //    i-th waiting request), then possibly one partial chunk.
        while (budget > 0 && wc > 0 && nr < S) {
            const bool in = lane < wc && lane < S - nr;
            const int slot = (wh + lane) % C;
            const int pre_i = in ? wpre[slot] : 0;
            const long long cp = warp_incl_sum64(pre_i, lane);
            const long long cb = warp_incl_sum64(in ? kv_blocks(pre_i, bs) : 0, lane);
            const bool whole = in && cp <= budget && cb <= freeb;
            const int k = __popc(__ballot_sync(kFull, whole));
            if (whole) {
                rctx[nr + lane] = 0;
                rpre[nr + lane] = pre_i;
                rdec[nr + lane] = wdec[slot];
                rx[nr + lane] = pre_i;
            }
            if (k > 0) {
                budget -= (int)__shfl_sync(kFull, cp, k - 1);
                freeb -= __shfl_sync(kFull, cb, k - 1);
                nr += k;
                wh = (wh + k) % C;
                wc -= k;
            }
            __syncwarp();
            if (k < 32) {
                if (budget > 0 && wc > 0 && nr < S) {
                    const int pre_h = wpre[wh];
                    const int x = min(pre_h, budget);
                    const long long need = kv_blocks(x, bs);
                    if (x < pre_h && need <= freeb) {
                        if (lane == 0) {
                            rctx[nr] = 0;
                            rpre[nr] = pre_h;
                            rdec[nr] = wdec[wh];
                            rx[nr] = x;
                        }
                        ++nr;
                        wh = (wh + 1) % C;
                        --wc;
                        budget -= x;
                        freeb -= need;
                    }
                }
                break;
            }
        }
        __syncwarp();
        const bool qcan = wc == 0;
        if (la0 == 0 && qcan && budget > 0 && nr < S) la0 = l;
        // 3. The batch's features, and each request's progress.
        long long f1 = 0, f2 = 0, f3 = 0, f4 = 0;
        for (int base = 0; base < nr; base += 32) {
            const int r = base + lane;
            if (r < nr) {
                long long ctx = rctx[r];
                int pre = rpre[r], dec = rdec[r];
                if (pre > 0) {
                    const long long x = rx[r];
                    f1 += x;
                    f4 += x * ctx + x * (x + 1) / 2;
                    ctx += x;
                    pre -= (int)x;
                    if (pre == 0 && MODE == 1) dec -= 1;
                } else {
                    f2 += 1;
                    f3 += ctx;
                    ctx += 1;
                    dec -= 1;
                }
                if (pre == 0 && ctx >= mctx) dec = 0;  // the context limit ends the response
                rctx[r] = (int)ctx;
                rpre[r] = pre;
                rdec[r] = dec;
            }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            f1 += __shfl_xor_sync(kFull, f1, o);
            f2 += __shfl_xor_sync(kFull, f2, o);
            f3 += __shfl_xor_sync(kFull, f3, o);
            f4 += __shfl_xor_sync(kFull, f4, o);
        }
        if (la0 != 0) {
            if (lane == 0) {
                KvRec R;
                R.f3 = f3;
                R.f4 = f4;
                R.f1 = (int)f1;
                R.f2 = (int)f2;
                R.bar = bar;
                R.bl = budget;
                R.seats = S - nr;
                R.flags = qcan ? 1 : 0;
                R.slack = slack;
                R.far = far;
                R.fa = freeb;
                rec[nrec] = R;
            }
            ++nrec;
        } else {
            fcum[0] += 1;
            fcum[1] += f1;
            fcum[2] += f2;
            fcum[3] += f3;
            fcum[4] += f4;
        }
        __syncwarp();
        // 4. Finished requests leave in order and return their blocks.
        int kept = 0;
        long long back = 0;
        for (int base = 0; base < nr; base += 32) {
            const int r = base + lane;
            const bool live = r < nr && rdec[r] > 0;
            const int v0 = r < nr ? rctx[r] : 0, v1 = r < nr ? rpre[r] : 0, v2 = r < nr ? rdec[r] : 0;
            if (r < nr && !live) back += kv_blocks(v0, bs);
            const unsigned m = __ballot_sync(kFull, live);
            __syncwarp();
            if (live) {
                const int dst = kept + __popc(m & ((1u << lane) - 1u));
                rctx[dst] = v0;
                rpre[dst] = v1;
                rdec[dst] = v2;
            }
            kept += __popc(m);
            __syncwarp();
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) back += __shfl_xor_sync(kFull, back, o);
        nr = kept;
        freeb += back;
        if (nr == 0 && wc == 0) {  // no resident left: every later batch is empty
            if (la0 == 0) la0 = l + 1;
            done = 1;
            break;
        }
        if (nrec == a.kv.horizon) break;
    }
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
    const size_t per_warp = kv_smem_per_warp(a.cfg) / sizeof(int32_t);
    if (j < a.cfg.I) kv_instance<MODE>(a, out, j, lane, kv_smem + wid * per_warp);
    // the last CTA to finish publishes the new snapshot if every instance succeeded
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

constexpr float kNaN = __builtin_nanf("");

// One (query, instance) candidate through the instance's records (one thread each).
// The query's state: waiting, or running with ctx tokens in the cache (h blocks) and
// pre still to prefill.  In a batch it is preempted if the residents' scan leaves a
// slack below h, or if its own tokens need more blocks than are free to it (it is
// the last running request: it preempts itself); a preempted query recomputes its
// whole context and may be readmitted in the same batch.  Admission needs the
// residents' queue empty, budget, a seat and the first chunk's blocks.
template <int MODE>
__global__ void __launch_bounds__(256) k_kv_estimate(const KvEst a) {
    const DevConfig &c = a.cfg;
    const int active = load_acquire(&a.ctl->active);
    const long long total = (long long)a.Q * c.I;
    for (long long idx = blockIdx.x * (long long)blockDim.x + threadIdx.x; idx < total;
         idx += (long long)gridDim.x * blockDim.x) {
        const int i = (int)(idx / c.I);
        const int j = (int)(idx - (long long)i * c.I);
        const int p = a.prompt[i];
        const long long bs = a.kv.bs[j], nbk = a.kv.nb[j], mctx = a.kv.mctx[j];
        // a query with one output token: its prompt below the context limit and its
        // whole context within the instance's blocks
        const bool valid = p >= 1 && p <= c.pmax && (long long)p < mctx && kv_blocks(min((long long)p + 1, mctx), bs) <= nbk;
        long long F[5] = {-1, -1, -1, -1, -1};
        int lt = -1;
        int err = 0;
        if (active < 0) {
            err = kENoState;
        } else if (!valid) {
            err = kEInval;
        } else {
            const StateBuf sb = active ? a.buf1 : a.buf0;
            const KvInst hd = sb.kvi[j];
            const KvRec *rec = sb.kvr + (size_t)j * a.kv.horizon;
            for (int k = 0; k < 5; ++k) F[k] = hd.fcum[k];
            const int B = c.B[j], S = c.S[j];
            bool run = false;
            long long pre = p, ctx = 0, held = 0;
            // after the records the instance is empty; the query then needs at most
            // ceil(p / B) + 2 batches
            const int limit = hd.nrec + (hd.done ? (p / B + 3) : 0);
            for (int t = 0;; ++t) {
                if (t >= limit) {
                    err = kETraj;
                    break;
                }
                KvRec R;
                if (t < hd.nrec) {
                    R = rec[t];
                } else {
                    R.f3 = 0;
                    R.f4 = 0;
                    R.f1 = 0;
                    R.f2 = 0;
                    R.bar = B;
                    R.bl = B;
                    R.seats = S;
                    R.flags = 1;
                    R.slack = kHuge;
                    R.far = nbk;
                    R.fa = nbk;
                }
                const int l = hd.la0 + t;
                F[0] += 1;
                F[1] += R.f1;
                F[2] += R.f2;
                F[3] += R.f3;
                F[4] += R.f4;
                bool first = false;
                if (run) {
                    if (R.slack < held) {  // a resident needs the query's blocks
                        pre += ctx;
                        ctx = 0;
                        held = 0;
                        run = false;
                    } else if (R.bar > 0) {
                        const long long x = pre > 0 ? min(pre, (long long)R.bar) : 1;
                        const long long need = kv_blocks(ctx + x, bs) - held;
                        if (need > R.far - held) {  // its own tokens do not fit: it preempts itself
                            pre += ctx;
                            ctx = 0;
                            held = 0;
                            run = false;
                        } else {
                            held += need;
                            if (pre > 0) {
                                F[1] += x;
                                F[4] += x * ctx + x * (x + 1) / 2;
                                ctx += x;
                                pre -= x;
                                first = (pre == 0 && MODE == 1);
                            } else {
                                F[2] += 1;
                                F[3] += ctx;
                                first = true;
                            }
                            if (first) {
                                lt = l;
                                break;
                            }
                            continue;
                        }
                    } else {
                        continue;  // no budget reached the query this batch
                    }
                }
                if ((R.flags & 1) && R.bl > 0 && R.seats > 0) {
                    const long long x = min(pre, (long long)R.bl);
                    const long long need = kv_blocks(x, bs);
                    if (R.fa >= need) {
                        held = need;
                        F[1] += x;
                        F[4] += x * (x + 1) / 2;
                        ctx = x;
                        pre -= x;
                        run = true;
                        if (pre == 0 && MODE == 1) {
                            lt = l;
                            break;
                        }
                    }
                }
            }
        }
        if (err) record_status(a.ctl, err);
        if (a.ttft) {
            float t = kNaN;
            if (!err) {
                const int m = c.moi[j];
                const float *b = c.coef + 5 * m;
                t = __fmul_rn(b[0], __ll2float_rn(F[0]));
                t = __fmaf_rn(b[2], __ll2float_rn(F[2]), t);
                t = __fmaf_rn(b[1], __ll2float_rn(F[1]), t);
                t = __fmaf_rn(b[3], __ll2float_rn(F[3]), t);
                t = __fmaf_rn(b[4], __ll2float_rn(F[4]), t);
            }
            a.ttft[idx] = t;
        }
        if (a.first_batch) a.first_batch[idx] = err ? -1 : lt;
        if (a.features)
            for (int k = 0; k < 5; ++k) a.features[idx * 5 + k] = err ? -1 : F[k];
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
    return e;
}

cudaError_t launch_kv_estimate(const KvEst &a, int sms, cudaStream_t st) {
    const long long total = (long long)a.Q * a.cfg.I;
    const int grid = (int)std::max<long long>(1, std::min<long long>((total + 255) / 256, (long long)sms * 8));
    if (a.cfg.mode == 0) k_kv_estimate<0><<<grid, 256, 0, st>>>(a);
    else k_kv_estimate<1><<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace lr
