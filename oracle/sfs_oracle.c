/*
 * CPU oracle for the latency-aware router -- test infrastructure only.
 *
 * Literal restatement of the paper's Serving Framework Simulation (Sec. 4.1)
 * and routing objectives (Sec. 3).  Nothing here is blocked, fused or
 * reordered: each candidate is simulated on its own, one token batch after
 * another, with the whole resident set in a plain array.  Built with
 * -ffp-contract=off so that the only fused multiply-adds are the explicit
 * fmaf() calls of the canonical expressions below.
 *
 * Readings of points the paper leaves open (each is a stated convention):
 *  - Scheduler step (Sec. 2 on chunked prefill; App. F on queue order, admission
 *    limits and the token budget): a batch starts with budget B; the
 *    running list is served in order, a request with remaining prefill taking
 *    min(remaining, budget) tokens and a decoding request one token, until the
 *    budget is spent; then, while budget remains, the waiting list is non-empty
 *    and fewer than S requests run, the waiting head is admitted FCFS with a
 *    prefill chunk of min(prompt, budget).  Requests whose decode count reaches
 *    zero leave after the batch.
 *  - First output token: by default a separate decode batch after the last
 *    prefill chunk (Sec. 4.1: decoding starts once every prompt token has been
 *    processed); optionally sampled in the batch of the last chunk.
 *  - Context of a decode token = tokens in the KV cache before the batch.
 *  - orc_sfs_candidate: KV capacity is unbounded and nothing is preempted;
 *    orc_sfs_candidate_kv adds block and context limits with preemption (the
 *    reading stated before kv_sim below).
 *  - Canonical fp32 order for Eq. 9 summed over batches: intercept, decode
 *    tokens, prefill tokens, decode context, prefill attention.
 *
 * parity pins: tests/test_oracle_pins.py (closed forms, hand traces, invariants).
 */
#include "sfs_oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int64_t ctx;  /* tokens already in the KV cache */
    int64_t pre;  /* remaining prefill tokens */
    int64_t dec;  /* remaining decode tokens */
    int is_query; /* the new query q_i */
    int64_t id;   /* stream step: tracked query id until its first output token, else -1 */
} orc_req;

enum { SCHED_NONE = 0, SCHED_PREFILL = 1, SCHED_DECODE = 2 };

static int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

/*
 * The augmented workload X_{i,j} (Sec. 4.1): the resident set R_j = Q_j u A_j
 * plus q_i at the tail of the waiting queue.  Simulate token batches
 * l = 1, 2, ... until q_i produces its first output token (Eq. 7) and return
 * the batch features whose Eq. 9 weighted sum, added over those batches,
 * is the SFS TTFT of Eq. 8.
 */
int orc_sfs_candidate(const orc_instance *inst, int32_t B, int32_t S, int32_t mode,
                      int32_t p, int32_t d, int64_t max_batches,
                      int64_t F[5], int64_t *l_admit, int64_t *l_ttft)
{
    if (!inst || !F || B < 1 || S < 1 || p < 1 || d < 1 || inst->n_run < 0 || inst->n_wait < 0)
        return ORC_EINVAL;
    if (mode != ORC_FIRST_TOKEN_SEPARATE_DECODE && mode != ORC_FIRST_TOKEN_WITH_LAST_CHUNK)
        return ORC_EINVAL;
    const int64_t total = (int64_t)inst->n_run + inst->n_wait + 1;
    orc_req *run = (orc_req *)calloc((size_t)total, sizeof(orc_req));
    orc_req *wait = (orc_req *)calloc((size_t)total, sizeof(orc_req));
    int64_t *alloc = (int64_t *)calloc((size_t)total, sizeof(int64_t));
    int *kind = (int *)calloc((size_t)total, sizeof(int));
    if (!run || !wait || !alloc || !kind) {
        free(run); free(wait); free(alloc); free(kind);
        return ORC_ENOMEM;
    }
    int64_t nr = 0, nw = 0, wh = 0;
    for (int32_t r = 0; r < inst->n_run; ++r) {
        run[nr].ctx = inst->run_ctx[r];
        run[nr].pre = inst->run_pre[r];
        run[nr].dec = inst->run_dec[r];
        run[nr].is_query = 0;
        if (run[nr].ctx < 0 || run[nr].pre < 0 || run[nr].dec < 1) goto bad;
        ++nr;
    }
    for (int32_t w = 0; w < inst->n_wait; ++w) {
        wait[nw].ctx = 0;
        wait[nw].pre = inst->wait_pre[w];
        wait[nw].dec = inst->wait_dec[w];
        wait[nw].is_query = 0;
        if (wait[nw].pre < 1 || wait[nw].dec < 1) goto bad;
        ++nw;
    }
    wait[nw].ctx = 0; wait[nw].pre = p; wait[nw].dec = d; wait[nw].is_query = 1;
    ++nw;

    for (int k = 0; k < 5; ++k) F[k] = 0;
    int64_t admitted_at = 0;
    for (int64_t l = 1; l <= max_batches; ++l) {
        /* 1. serve the running list in order until the token budget is spent */
        int64_t budget = B;
        for (int64_t r = 0; r < nr; ++r) { kind[r] = SCHED_NONE; alloc[r] = 0; }
        for (int64_t r = 0; r < nr && budget > 0; ++r) {
            if (run[r].pre > 0) {
                alloc[r] = min64(run[r].pre, budget);
                kind[r] = SCHED_PREFILL;
            } else {
                alloc[r] = 1;
                kind[r] = SCHED_DECODE;
            }
            budget -= alloc[r];
        }
        /* 2. admit from the waiting head while budget and a sequence slot remain */
        while (budget > 0 && wh < nw && nr < S) {
            run[nr] = wait[wh++];
            alloc[nr] = min64(run[nr].pre, budget);
            kind[nr] = SCHED_PREFILL;
            budget -= alloc[nr];
            if (run[nr].is_query) admitted_at = l;
            ++nr;
        }
        /* 3. account the batch: the feature vector of Eq. 9 */
        int done = 0;
        F[0] += 1;
        for (int64_t r = 0; r < nr; ++r) {
            if (kind[r] == SCHED_PREFILL) {
                const int64_t x = alloc[r];
                F[1] += x;
                F[4] += x * run[r].ctx + x * (x + 1) / 2;
                run[r].ctx += x;
                run[r].pre -= x;
                if (run[r].pre == 0 && mode == ORC_FIRST_TOKEN_WITH_LAST_CHUNK) {
                    run[r].dec -= 1;              /* first token sampled with the last chunk */
                    if (run[r].is_query) done = 1;
                }
            } else if (kind[r] == SCHED_DECODE) {
                F[2] += 1;
                F[3] += run[r].ctx;
                run[r].ctx += 1;
                run[r].dec -= 1;
                if (run[r].is_query) done = 1;    /* Eq. 7: first batch with a decode token of q_i */
            }
        }
        if (done) {
            if (l_admit) *l_admit = admitted_at;
            if (l_ttft) *l_ttft = l;
            free(run); free(wait); free(alloc); free(kind);
            return ORC_OK;
        }
        /* 4. finished requests leave the running list (order kept) */
        int64_t keep = 0;
        for (int64_t r = 0; r < nr; ++r)
            if (run[r].dec > 0) run[keep++] = run[r];
        nr = keep;
    }
    free(run); free(wait); free(alloc); free(kind);
    return ORC_ELIMIT;
bad:
    free(run); free(wait); free(alloc); free(kind);
    return ORC_EINVAL;
}

/* Eq. 9 summed over the batches up to the first-token batch (Eq. 8):
 * T = b0*F0 + b1p*F1 + b1d*F2 + b2*F3 + b3*F4, evaluated in this fixed fp32 order. */
float orc_ttft_f32(const float coef[5], const int64_t F[5])
{
    const float f0 = (float)F[0], f1 = (float)F[1], f2 = (float)F[2];
    const float f3 = (float)F[3], f4 = (float)F[4];
    float t = coef[0] * f0;
    t = fmaf(coef[2], f2, t);
    t = fmaf(coef[1], f1, t);
    t = fmaf(coef[3], f3, t);
    t = fmaf(coef[4], f4, t);
    return t;
}

int orc_estimate_candidates_kv(int32_t num_instances, const int32_t *model_of_instance,
                               const float *coef, const int32_t *B, const int32_t *S,
                               int32_t cap_running, int32_t cap_waiting,
                               const int32_t *n_run, const int32_t *run_ctx, const int32_t *run_pre,
                               const int32_t *run_dec, const int32_t *n_wait, const int32_t *wait_pre,
                               const int32_t *wait_dec, const int32_t *prompt_len,
                               const int32_t *block_size, const int64_t *num_blocks, const int64_t *max_ctx,
                               int32_t mode, int64_t max_batches,
                               int64_t num_cand, const int32_t *cand_q, const int32_t *cand_j,
                               int32_t *status, int64_t *F, int64_t *l_ttft, float *ttft32, double *ttft64)
{
    for (int64_t c = 0; c < num_cand; ++c) {
        const int32_t i = cand_q[c], j = cand_j[c];
        if (j < 0 || j >= num_instances) return ORC_EINVAL;
        orc_instance inst;
        inst.n_run = n_run[j];
        inst.run_ctx = run_ctx + (int64_t)j * cap_running;
        inst.run_pre = run_pre + (int64_t)j * cap_running;
        inst.run_dec = run_dec + (int64_t)j * cap_running;
        inst.n_wait = n_wait[j];
        inst.wait_pre = wait_pre + (int64_t)j * cap_waiting;
        inst.wait_dec = wait_dec + (int64_t)j * cap_waiting;
        if (inst.n_run > cap_running || inst.n_wait > cap_waiting) return ORC_EINVAL;
        const orc_kv kv = {block_size[j], num_blocks[j], max_ctx[j]};
        int64_t Fc[5] = {-1, -1, -1, -1, -1}, la = 0, lt = -1;
        /* the query up to its first token: one output token */
        const int rc = orc_sfs_candidate_kv(&inst, B[j], S[j], mode, &kv, prompt_len[i], 1, max_batches, Fc, &la,
                                            &lt, NULL, NULL);
        status[c] = rc;
        if (rc != ORC_OK) {
            for (int k = 0; k < 5; ++k) Fc[k] = -1;
            lt = -1;
        }
        for (int k = 0; k < 5; ++k) F[c * 5 + k] = Fc[k];
        if (l_ttft) l_ttft[c] = lt;
        const float *cf = coef + 5 * model_of_instance[j];
        if (ttft32) ttft32[c] = rc == ORC_OK ? orc_ttft_f32(cf, Fc) : NAN;
        if (ttft64) ttft64[c] = rc == ORC_OK ? orc_ttft_f64(cf, Fc) : NAN;
    }
    return ORC_OK;
}

double orc_ttft_f64(const float coef[5], const int64_t F[5])
{
    return (double)coef[0] * (double)F[0] + (double)coef[1] * (double)F[1] +
           (double)coef[2] * (double)F[2] + (double)coef[3] * (double)F[3] +
           (double)coef[4] * (double)F[4];
}

int orc_estimate_candidates(int32_t num_instances, const int32_t *model_of_instance,
                            const float *coef, const int32_t *B, const int32_t *S,
                            int32_t cap_running, int32_t cap_waiting,
                            const int32_t *n_run, const int32_t *run_ctx, const int32_t *run_pre,
                            const int32_t *run_dec, const int32_t *n_wait, const int32_t *wait_pre,
                            const int32_t *wait_dec, int32_t num_models, const int32_t *prompt_len,
                            const int32_t *dec_hat, int32_t mode, int64_t max_batches,
                            int64_t num_cand, const int32_t *cand_q, const int32_t *cand_j,
                            int64_t *F, int64_t *l_ttft, float *ttft32, double *ttft64)
{
    for (int64_t c = 0; c < num_cand; ++c) {
        const int32_t i = cand_q[c], j = cand_j[c];
        if (j < 0 || j >= num_instances) return ORC_EINVAL;
        const int32_t m = model_of_instance[j];
        if (m < 0 || m >= num_models) return ORC_EINVAL;
        orc_instance inst;
        inst.n_run = n_run[j];
        inst.run_ctx = run_ctx + (int64_t)j * cap_running;
        inst.run_pre = run_pre + (int64_t)j * cap_running;
        inst.run_dec = run_dec + (int64_t)j * cap_running;
        inst.n_wait = n_wait[j];
        inst.wait_pre = wait_pre + (int64_t)j * cap_waiting;
        inst.wait_dec = wait_dec + (int64_t)j * cap_waiting;
        if (inst.n_run > cap_running || inst.n_wait > cap_waiting) return ORC_EINVAL;
        int64_t Fc[5], la = 0, lt = 0;
        const int rc = orc_sfs_candidate(&inst, B[j], S[j], mode, prompt_len[i],
                                         dec_hat[(int64_t)i * num_models + m], max_batches, Fc, &la, &lt);
        if (rc != ORC_OK) return rc;
        for (int k = 0; k < 5; ++k) F[c * 5 + k] = Fc[k];
        if (l_ttft) l_ttft[c] = lt;
        if (ttft32) ttft32[c] = orc_ttft_f32(coef + 5 * m, Fc);
        if (ttft64) ttft64[c] = orc_ttft_f64(coef + 5 * m, Fc);
    }
    return ORC_OK;
}

/* Eq. 2 with the predicted cost of App. B.4:
 * cost = p * price_in + dec_hat * price_out, U = acc - lambda * cost (fp32, explicit fma). */
float orc_utility(float acc, float lambda, int32_t p, int32_t dec_hat, float price_in, float price_out)
{
    const float cost = fmaf((float)dec_hat, price_out, (float)p * price_in);
    return fmaf(-lambda, cost, acc);
}

int orc_route(int32_t Q, int32_t I, int32_t M, const int32_t *model_of_instance,
              const float *price_in, const float *price_out, const int32_t *prompt_len,
              const int32_t *dec_hat, const float *acc, const float *ttft, const float *tau,
              int32_t P, const float *lambda, const float *mu,
              int32_t *assign, float *util, float *ttft_chosen)
{
    if (Q < 0 || I < 1 || M < 1 || P < 1) return ORC_EINVAL;
    for (int32_t pp = 0; pp < P; ++pp) {
        for (int32_t i = 0; i < Q; ++i) {
            const float *row = ttft + (int64_t)i * I;
            int32_t best_j = -1, fast_j = -1;
            float best = 0.0f, best_u = 0.0f, fast_t = 0.0f;
            for (int32_t j = 0; j < I; ++j) {
                const int32_t m = model_of_instance[j];
                const float u = orc_utility(acc[(int64_t)i * M + m], lambda[pp], prompt_len[i],
                                            dec_hat[(int64_t)i * M + m], price_in[m], price_out[m]);
                const float t = row[j];
                if (t != t) continue;  /* no estimate (an invalid candidate): not eligible */
                if (tau == NULL) {
                    /* Eq. 5: argmax_j U - mu * L, ties to the lowest index */
                    const float J = fmaf(-mu[pp], t, u);
                    if (best_j < 0 || J > best) { best = J; best_j = j; best_u = u; }
                } else {
                    /* Eq. 3: argmax U over {j : L <= tau}; empty set -> least latency */
                    if (t <= tau[i] && (best_j < 0 || u > best_u)) { best_u = u; best_j = j; }
                    if (fast_j < 0 || t < fast_t) { fast_t = t; fast_j = j; }
                }
            }
            int32_t pick = best_j;
            if (tau != NULL && best_j < 0) pick = fast_j;
            if (pick < 0) {  /* no eligible instance */
                assign[(int64_t)pp * Q + i] = -1;
                util[(int64_t)pp * Q + i] = NAN;
                if (ttft_chosen) ttft_chosen[(int64_t)pp * Q + i] = NAN;
                continue;
            }
            const int32_t m = model_of_instance[pick];
            assign[(int64_t)pp * Q + i] = pick;
            util[(int64_t)pp * Q + i] = orc_utility(acc[(int64_t)i * M + m], lambda[pp], prompt_len[i],
                                                    dec_hat[(int64_t)i * M + m], price_in[m], price_out[m]);
            if (ttft_chosen) ttft_chosen[(int64_t)pp * Q + i] = row[pick];
        }
    }
    return ORC_OK;
}

int orc_frontier(int32_t Q, int32_t I, int32_t M, const int32_t *model_of_instance,
                 const float *price_in, const float *price_out, const int32_t *prompt_len,
                 const int32_t *dec_hat, const float *acc, int32_t P, const int32_t *assign,
                 const float *ttft_chosen, double *out)
{
    if (Q < 1 || P < 1) return ORC_EINVAL;
    for (int32_t pp = 0; pp < P; ++pp) {
        double sa = 0.0, sc = 0.0, st = 0.0;
        for (int32_t i = 0; i < Q; ++i) {
            const int32_t j = assign[(int64_t)pp * Q + i];
            if (j < 0 || j >= I) return ORC_EINVAL;
            const int32_t m = model_of_instance[j];
            const float cost = fmaf((float)dec_hat[(int64_t)i * M + m], price_out[m],
                                    (float)prompt_len[i] * price_in[m]);
            sa += (double)acc[(int64_t)i * M + m];
            sc += (double)cost;
            st += (double)ttft_chosen[(int64_t)pp * Q + i];
        }
        out[pp * 3 + 0] = sa / Q;
        out[pp * 3 + 1] = sc / Q;
        out[pp * 3 + 2] = st / Q;
    }
    return ORC_OK;
}

/*
 * Online stream step.  The engine behind each instance keeps executing token
 * batches (Sec. 2, continuous batching) and publishes its state after each one
 * (App. F); the router sees the state after the last batch completed by the
 * current time.  Batch times follow Eq. 9 for the batch actually executed.
 */
int orc_advance(int32_t I, const int32_t *model_of_instance, const float *coef, const int32_t *B,
                const int32_t *S, int32_t cap_running, int32_t cap_waiting, int32_t *n_run,
                int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre,
                int32_t *wait_dec, double *clock, int32_t Q, const int32_t *assign,
                const int32_t *prompt_len, const int32_t *dec, int32_t mode, double t_now,
                int64_t max_batches)
{
    return orc_advance_ids(I, model_of_instance, coef, B, S, cap_running, cap_waiting, n_run, run_ctx, run_pre,
                           run_dec, n_wait, wait_pre, wait_dec, clock, Q, assign, prompt_len, dec, mode, t_now,
                           max_batches, NULL, NULL, -1, NULL);
}

/* The realized first output token (Sec. 4.1: the TTFT ends with the first output
 * token; Eq. 4 scores each query by its realized TTFT).  A tracked request emits it
 * in the first executed batch that gives it a decode token, or, when the first token
 * comes with the last prompt chunk, in the batch that completes its prompt; the time
 * is that batch's end on the instance's clock. */
static void first_token(orc_req *q, int emitted, double t_end, double *first_token_time)
{
    if (emitted && q->id >= 0) {
        first_token_time[q->id] = t_end;
        q->id = -1;
    }
}

int orc_advance_ids(int32_t I, const int32_t *model_of_instance, const float *coef, const int32_t *B,
                    const int32_t *S, int32_t cap_running, int32_t cap_waiting, int32_t *n_run,
                    int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre,
                    int32_t *wait_dec, double *clock, int32_t Q, const int32_t *assign,
                    const int32_t *prompt_len, const int32_t *dec, int32_t mode, double t_now,
                    int64_t max_batches, int64_t *run_id, int64_t *wait_id, int64_t id_base,
                    double *first_token_time)
{
    const int track = run_id != NULL && wait_id != NULL && first_token_time != NULL;
    int rc_all = ORC_OK;
    for (int32_t j = 0; j < I; ++j) {
        const int64_t total = (int64_t)cap_running + cap_waiting + Q + 1;
        orc_req *run = (orc_req *)calloc((size_t)total, sizeof(orc_req));
        orc_req *wait = (orc_req *)calloc((size_t)total, sizeof(orc_req));
        int64_t *alloc = (int64_t *)calloc((size_t)total, sizeof(int64_t));
        int *kind = (int *)calloc((size_t)total, sizeof(int));
        if (!run || !wait || !alloc || !kind) {
            free(run); free(wait); free(alloc); free(kind);
            return ORC_ENOMEM;
        }
        int64_t nr = 0, nw = 0, wh = 0;
        for (int32_t r = 0; r < n_run[j]; ++r) {
            const int64_t o = (int64_t)j * cap_running + r;
            run[nr].ctx = run_ctx[o]; run[nr].pre = run_pre[o]; run[nr].dec = run_dec[o]; run[nr].is_query = 0;
            run[nr].id = track ? run_id[o] : -1;
            ++nr;
        }
        for (int32_t w = 0; w < n_wait[j]; ++w) {
            const int64_t o = (int64_t)j * cap_waiting + w;
            wait[nw].ctx = 0; wait[nw].pre = wait_pre[o]; wait[nw].dec = wait_dec[o]; wait[nw].is_query = 0;
            wait[nw].id = track ? wait_id[o] : -1;
            ++nw;
        }
        /* 1. the routed queries join the waiting tail in query order (query i tracked
         *    as id_base + i when id_base >= 0) */
        for (int32_t i = 0; i < Q; ++i) {
            if (assign[i] != j) continue;
            wait[nw].ctx = 0; wait[nw].pre = prompt_len[i]; wait[nw].dec = dec[i]; wait[nw].is_query = 0;
            wait[nw].id = (track && id_base >= 0) ? id_base + i : -1;
            ++nw;
        }
        int rc = (nw > cap_waiting) ? ORC_ELIMIT : ORC_OK;
        const float *cf = coef + 5 * model_of_instance[j];
        double t = clock[j];
        /* 2. execute whole batches that end by t_now */
        for (int64_t step = 0; rc == ORC_OK; ++step) {
            if (nr == 0 && wh == nw) {                        /* idle: nothing to run */
                if (t < t_now) t = t_now;                     /* a clock never runs backwards */
                break;
            }
            if (step >= max_batches) { rc = ORC_ELIMIT; break; }
            /* plan the batch with the scheduler step (running list, then FCFS admission) */
            int64_t budget = B[j];
            for (int64_t r = 0; r < nr; ++r) { kind[r] = SCHED_NONE; alloc[r] = 0; }
            for (int64_t r = 0; r < nr && budget > 0; ++r) {
                if (run[r].pre > 0) { alloc[r] = min64(run[r].pre, budget); kind[r] = SCHED_PREFILL; }
                else { alloc[r] = 1; kind[r] = SCHED_DECODE; }
                budget -= alloc[r];
            }
            int64_t na = 0;
            int64_t wbud = budget;
            while (wbud > 0 && wh + na < nw && nr + na < S[j]) {
                alloc[nr + na] = min64(wait[wh + na].pre, wbud);
                kind[nr + na] = SCHED_PREFILL;
                wbud -= alloc[nr + na];
                ++na;
            }
            int64_t F[5] = {1, 0, 0, 0, 0};
            for (int64_t r = 0; r < nr + na; ++r) {
                const orc_req *q = (r < nr) ? &run[r] : &wait[wh + r - nr];
                if (kind[r] == SCHED_PREFILL) {
                    const int64_t x = alloc[r];
                    F[1] += x;
                    F[4] += x * q->ctx + x * (x + 1) / 2;
                } else if (kind[r] == SCHED_DECODE) {
                    F[2] += 1;
                    F[3] += q->ctx;
                }
            }
            const float T = orc_ttft_f32(cf, F);   /* Eq. 9 for this one batch */
            if (t + (double)T > t_now) break;       /* still running at t_now */
            /* apply the batch */
            for (int64_t k = 0; k < na; ++k) run[nr + k] = wait[wh + k];
            nr += na;
            wh += na;
            if (nr > cap_running) { rc = ORC_ELIMIT; break; }
            for (int64_t r = 0; r < nr; ++r) {
                if (kind[r] == SCHED_PREFILL) {
                    run[r].ctx += alloc[r];
                    run[r].pre -= alloc[r];
                    if (run[r].pre == 0 && mode == ORC_FIRST_TOKEN_WITH_LAST_CHUNK) {
                        run[r].dec -= 1;
                        if (track) first_token(&run[r], 1, t + (double)T, first_token_time);
                    }
                } else if (kind[r] == SCHED_DECODE) {
                    run[r].ctx += 1;
                    run[r].dec -= 1;
                    if (track) first_token(&run[r], mode == ORC_FIRST_TOKEN_SEPARATE_DECODE, t + (double)T,
                                           first_token_time);
                }
            }
            int64_t keep = 0;
            for (int64_t r = 0; r < nr; ++r)
                if (run[r].dec > 0) run[keep++] = run[r];
            nr = keep;
            t += (double)T;
        }
        if (rc == ORC_OK) {
            n_run[j] = (int32_t)nr;
            for (int64_t r = 0; r < cap_running; ++r) {
                const int64_t o = (int64_t)j * cap_running + r;
                run_ctx[o] = r < nr ? (int32_t)run[r].ctx : 0;
                run_pre[o] = r < nr ? (int32_t)run[r].pre : 0;
                run_dec[o] = r < nr ? (int32_t)run[r].dec : 0;
                if (track) run_id[o] = r < nr ? run[r].id : -1;
            }
            n_wait[j] = (int32_t)(nw - wh);
            for (int64_t w = 0; w < cap_waiting; ++w) {
                const int64_t o = (int64_t)j * cap_waiting + w;
                wait_pre[o] = w < nw - wh ? (int32_t)wait[wh + w].pre : 0;
                wait_dec[o] = w < nw - wh ? (int32_t)wait[wh + w].dec : 0;
                if (track) wait_id[o] = w < nw - wh ? wait[wh + w].id : -1;
            }
            clock[j] = t;
        } else {
            rc_all = rc;
        }
        free(run); free(wait); free(alloc); free(kind);
    }
    return rc_all;
}

/* ------------------------------------------------------------------------- */
/* Average-case estimators (Sec. 4, average-case TTFT estimation; App. E).   */

double orc_pow_int(double x, int32_t k)
{
    double r = 1.0, b = x;
    int32_t e = k;
    while (e > 0) {
        if (e & 1) r = r * b;
        e >>= 1;
        if (e > 0) b = b * b;
    }
    return r;
}

/* Limited processor sharing: Poisson arrivals at alpha, aggregate service rate mu
 * shared by at most k active requests, FIFO beyond them.  An arrival that sees n >= k
 * residents waits for n - k + 1 completions at rate mu; averaging over the M/M/1
 * stationary law gives rho^k / (mu - alpha).  The G/G/k form scales it by
 * (ca2 + cs2) / 2, with E[Q] = 1 / mu. */
double orc_lps_wait(double alpha, double mu, int32_t k, double ca2, double cs2)
{
    if (!(mu > 0.0) || !(alpha >= 0.0) || !(alpha < mu) || k < 1) return NAN;
    const double rho = alpha / mu;
    const double c = (ca2 + cs2) * 0.5;
    return (c * orc_pow_int(rho, k)) / (mu - alpha);
}

double orc_throughput_wait(const orc_instance *inst, double theta)
{
    int64_t tokens = 0;
    for (int32_t r = 0; r < inst->n_run; ++r) tokens += inst->run_pre[r];
    for (int32_t w = 0; w < inst->n_wait; ++w) tokens += inst->wait_pre[w];
    return (double)tokens / theta;
}

int orc_avgcase_ttft(int32_t I, int32_t Q, const double *W, const double *theta, const double *tdec,
                     const int32_t *prompt_len, float *t32, double *t64)
{
    for (int32_t j = 0; j < I; ++j)
        if (!(theta[j] > 0.0) || !(tdec[j] >= 0.0) || !(W[j] >= 0.0)) return ORC_EINVAL;
    for (int32_t i = 0; i < Q; ++i) {
        const int32_t p = prompt_len[i];
        for (int32_t j = 0; j < I; ++j) {
            const float g = (float)(1.0 / theta[j]);
            const float c = (float)(W[j] + tdec[j]);
            t32[(int64_t)i * I + j] = fmaf((float)p, g, c);
            t64[(int64_t)i * I + j] = W[j] + (double)p / theta[j] + tdec[j];
        }
    }
    return ORC_OK;
}

/* ---- Baseline routing policies and stream metrics (Sec. 6 baselines; Eq. 4) ---- */

int orc_round_robin(int32_t Q, int32_t I, int64_t start, int32_t *assign)
{
    if (Q < 0 || I < 1 || start < 0) return ORC_EINVAL;
    for (int32_t q = 0; q < Q; ++q) assign[q] = (int32_t)((start + q) % I);
    return ORC_OK;
}

int orc_shortest_queue(int32_t Q, int32_t I, const int32_t *counts, int32_t *assign)
{
    if (Q < 0 || I < 1) return ORC_EINVAL;
    int64_t *n = (int64_t *)malloc(sizeof(int64_t) * (size_t)I);
    if (!n) return ORC_EINVAL;
    for (int32_t j = 0; j < I; ++j) n[j] = counts[j];
    for (int32_t q = 0; q < Q; ++q) {
        int32_t best = 0;
        for (int32_t j = 1; j < I; ++j)
            if (n[j] < n[best]) best = j;
        assign[q] = best;
        n[best] += 1;  /* the routed query joins that queue */
    }
    free(n);
    return ORC_OK;
}

int orc_latency_agnostic(int32_t Q, int32_t I, int32_t M, const int32_t *model_of_instance,
                         const float *price_in, const float *price_out, const int32_t *prompt_len,
                         const int32_t *dec_hat, const float *acc, float lambda, int32_t *assign)
{
    if (Q < 0 || I < 1 || M < 1) return ORC_EINVAL;
    for (int32_t i = 0; i < Q; ++i) {
        int32_t best_j = 0;
        float best = 0.0f;
        for (int32_t j = 0; j < I; ++j) {
            const int32_t m = model_of_instance[j];
            const float u = orc_utility(acc[(int64_t)i * M + m], lambda, prompt_len[i],
                                        dec_hat[(int64_t)i * M + m], price_in[m], price_out[m]);
            if (j == 0 || u > best) { best = u; best_j = j; }
        }
        assign[i] = best_j;
    }
    return ORC_OK;
}

int orc_on_time_utility(int32_t Q, const float *util, const float *ttft, const float *tau,
                        const float *delay, double *out)
{
    if (Q < 1) return ORC_EINVAL;
    double su = 0.0, sn = 0.0;
    for (int32_t i = 0; i < Q; ++i) {
        const float realized = delay ? delay[i] + ttft[i] : ttft[i];
        if (realized <= tau[i]) {  /* false for NaN */
            su += (double)util[i];
            sn += 1.0;
        }
    }
    out[0] = su / Q;
    out[1] = sn / Q;
    return ORC_OK;
}

/* ---- KV-cache limits, context limit and preemption (App. F) ----
 *
 * App. F names context limits, the KV-cache allocation state and preemption
 * among what the simulation models, without a rule.  Reading
 * (a paged KV cache as in vLLM, whose engine the paper uses):
 *  - an instance has num_blocks blocks of block_size tokens; a request with ctx
 *    tokens in the cache holds ceil(ctx / block_size) blocks;
 *  - the running list is served in order as before; a request whose tokens of
 *    this batch need blocks that are not free makes room by preempting the last
 *    running request (recompute: its blocks are freed, its whole context becomes
 *    prefill again, and it goes to the front of the waiting queue), repeatedly,
 *    and preempts itself if it is the last;
 *  - the waiting head is admitted only if the blocks of its first chunk are free
 *    (FCFS, no skipping, no preemption for admission);
 *  - a request whose context reaches max_ctx stops (its response ends there);
 *  - a request whose whole context (capped at max_ctx) needs more blocks than the
 *    instance has can never finish and is rejected with the input (an engine
 *    refuses it).  Then the oldest running request can always proceed by
 *    preempting later ones, so every simulation ends.
 */
static int64_t kv_blocks(int64_t ctx, int64_t bs) { return (ctx + bs - 1) / bs; }

static int kv_sim(const orc_instance *inst, int32_t B, int32_t S, int32_t mode, const orc_kv *kv,
                  int with_query, int32_t p, int32_t d, int64_t max_batches,
                  int64_t F[5], int64_t *l_admit, int64_t *l_ttft, int64_t *res_F, int64_t *max_used)
{
    if (!inst || !kv || B < 1 || S < 1 || inst->n_run < 0 || inst->n_wait < 0) return ORC_EINVAL;
    if (kv->block_size < 1 || kv->num_blocks < 0 || kv->max_ctx < 2) return ORC_EINVAL;
    if (mode != ORC_FIRST_TOKEN_SEPARATE_DECODE && mode != ORC_FIRST_TOKEN_WITH_LAST_CHUNK) return ORC_EINVAL;
    if (with_query && (p < 1 || d < 1 || p >= kv->max_ctx)) return ORC_EINVAL;
    const int64_t bs = kv->block_size;
    const int64_t total = (int64_t)inst->n_run + inst->n_wait + 1;
    orc_req *run = (orc_req *)calloc((size_t)total, sizeof(orc_req));
    orc_req *wait = (orc_req *)calloc((size_t)(2 * total + 1), sizeof(orc_req)); /* room at the front */
    int64_t *alloc = (int64_t *)calloc((size_t)total, sizeof(int64_t));
    int *kind = (int *)calloc((size_t)total, sizeof(int));
    if (!run || !wait || !alloc || !kind) {
        free(run); free(wait); free(alloc); free(kind);
        return ORC_ENOMEM;
    }
    int rc = ORC_EINVAL;
    int64_t nr = 0, wh = total, we = total;  /* waiting queue: wait[wh .. we) */
    int64_t free_blocks = kv->num_blocks;
    for (int32_t r = 0; r < inst->n_run; ++r) {
        orc_req q = {inst->run_ctx[r], inst->run_pre[r], inst->run_dec[r], 0};
        if (q.ctx < 0 || q.pre < 0 || q.dec < 1 || q.ctx + q.pre >= kv->max_ctx) goto done;
        if (kv_blocks(min64(q.ctx + q.pre + q.dec, kv->max_ctx), bs) > kv->num_blocks) goto done;
        free_blocks -= kv_blocks(q.ctx, bs);
        run[nr++] = q;
    }
    if (free_blocks < 0) goto done;
    for (int32_t w = 0; w < inst->n_wait; ++w) {
        orc_req q = {0, inst->wait_pre[w], inst->wait_dec[w], 0};
        if (q.pre < 1 || q.dec < 1 || q.pre >= kv->max_ctx) goto done;
        if (kv_blocks(min64(q.pre + q.dec, kv->max_ctx), bs) > kv->num_blocks) goto done;
        wait[we++] = q;
    }
    if (with_query) {
        orc_req q = {0, p, d, 1};
        if (kv_blocks(min64((int64_t)p + d, kv->max_ctx), bs) > kv->num_blocks) goto done;
        wait[we++] = q;
    }
    if (F) for (int k = 0; k < 5; ++k) F[k] = 0;
    if (max_used) *max_used = kv->num_blocks - free_blocks;
    int64_t admitted_at = 0;
    rc = ORC_ELIMIT;
    for (int64_t l = 1; l <= max_batches; ++l) {
        int64_t *rf = res_F ? res_F + (l - 1) * 5 : NULL;
        if (rf) for (int k = 0; k < 5; ++k) rf[k] = 0;
        /* 1. the running list in order, each request's blocks found or made */
        int64_t budget = B;
        for (int64_t r = 0; r < nr; ++r) { kind[r] = SCHED_NONE; alloc[r] = 0; }
        int64_t r = 0;
        while (r < nr && budget > 0) {
            const int64_t x = run[r].pre > 0 ? min64(run[r].pre, budget) : 1;
            const int64_t need = kv_blocks(run[r].ctx + x, bs) - kv_blocks(run[r].ctx, bs);
            while (free_blocks < need && nr - 1 >= r) {
                /* preempt the last running request (possibly r itself) */
                orc_req v = run[nr - 1];
                free_blocks += kv_blocks(v.ctx, bs);
                v.pre += v.ctx;
                v.ctx = 0;
                wait[--wh] = v;
                --nr;
            }
            if (r >= nr) break;  /* r preempted itself */
            free_blocks -= need;
            alloc[r] = x;
            kind[r] = run[r].pre > 0 ? SCHED_PREFILL : SCHED_DECODE;
            budget -= x;
            ++r;
        }
        /* 2. admission from the waiting head while budget, a slot and its blocks allow */
        while (budget > 0 && wh < we && nr < S) {
            const int64_t x = min64(wait[wh].pre, budget);
            const int64_t need = kv_blocks(x, bs);
            if (free_blocks < need) break;
            free_blocks -= need;
            run[nr] = wait[wh++];
            alloc[nr] = x;
            kind[nr] = SCHED_PREFILL;
            budget -= x;
            if (run[nr].is_query) admitted_at = l;
            ++nr;
        }
        if (max_used && kv->num_blocks - free_blocks > *max_used) *max_used = kv->num_blocks - free_blocks;
        /* 3. account the batch */
        int done_q = 0;
        if (F) F[0] += 1;
        if (rf) rf[0] = 1;
        for (int64_t t = 0; t < nr; ++t) {
            int64_t f[5] = {0, 0, 0, 0, 0};
            if (kind[t] == SCHED_PREFILL) {
                const int64_t x = alloc[t];
                f[1] = x;
                f[4] = x * run[t].ctx + x * (x + 1) / 2;
                run[t].ctx += x;
                run[t].pre -= x;
                if (run[t].pre == 0 && mode == ORC_FIRST_TOKEN_WITH_LAST_CHUNK) {
                    run[t].dec -= 1;
                    if (run[t].is_query) done_q = 1;
                }
            } else if (kind[t] == SCHED_DECODE) {
                f[2] = 1;
                f[3] = run[t].ctx;
                run[t].ctx += 1;
                run[t].dec -= 1;
                if (run[t].is_query) done_q = 1;
            }
            if (run[t].pre == 0 && run[t].ctx >= kv->max_ctx) run[t].dec = 0;  /* context limit */
            for (int k = 1; k < 5; ++k) {
                if (F) F[k] += f[k];
                if (rf && !run[t].is_query) rf[k] += f[k];
            }
        }
        if (with_query && done_q) {
            if (l_admit) *l_admit = admitted_at;
            if (l_ttft) *l_ttft = l;
            rc = ORC_OK;
            break;
        }
        if (!with_query && l == max_batches) {
            rc = ORC_OK;
            break;
        }
        /* 4. finished requests leave and free their blocks */
        int64_t keep = 0;
        for (int64_t t = 0; t < nr; ++t) {
            if (run[t].dec > 0) run[keep++] = run[t];
            else free_blocks += kv_blocks(run[t].ctx, bs);
        }
        nr = keep;
    }
done:
    free(run); free(wait); free(alloc); free(kind);
    return rc;
}

int orc_sfs_candidate_kv(const orc_instance *inst, int32_t B, int32_t S, int32_t mode, const orc_kv *kv,
                         int32_t p, int32_t d, int64_t max_batches,
                         int64_t F[5], int64_t *l_admit, int64_t *l_ttft, int64_t *res_F, int64_t *max_used)
{
    if (!F) return ORC_EINVAL;
    return kv_sim(inst, B, S, mode, kv, 1, p, d, max_batches, F, l_admit, l_ttft, res_F, max_used);
}

int orc_kv_residents(const orc_instance *inst, int32_t B, int32_t S, int32_t mode, const orc_kv *kv,
                     int64_t L, int64_t *res_F)
{
    if (L < 1 || !res_F) return ORC_EINVAL;
    return kv_sim(inst, B, S, mode, kv, 0, 1, 1, L, NULL, NULL, NULL, res_F, NULL);
}


/* Online stream step under KV-cache limits: orc_advance with the KV step rule of kv_sim
 * above (App. F names KV-cache allocation, context limits and preemption among what
 * the serving simulation models; the same reading).  Each executed batch: the running
 * list in order, each request's new blocks found, preempting the last running request
 * (possibly itself) while they are not free; then FCFS admission while budget, a slot
 * and the first chunk's blocks allow; a request whose context reaches max_ctx ends and
 * frees its blocks.  The batch takes the Eq. 9 time of its own composition (canonical
 * fp32, accumulated into the fp64 clock) and runs only if it ends by t_now.  Limits per
 * instance: block_size[I], num_blocks[I], max_ctx[I].  First-token tracking as in
 * orc_advance_ids (run_id, wait_id, first_token_time may be NULL).  Returns ORC_EINVAL
 * when a routed query could never run (its prompt reaches max_ctx, or its whole
 * context capped at max_ctx needs more blocks than the instance has), ORC_ELIMIT when
 * a queue outgrows its capacity or an instance needs more than max_batches batches;
 * an instance that fails keeps its state. */
int orc_advance_kv(int32_t I, const int32_t *model_of_instance, const float *coef, const int32_t *B,
                   const int32_t *S, int32_t cap_running, int32_t cap_waiting, int32_t *n_run,
                   int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre,
                   int32_t *wait_dec, double *clock, int32_t Q, const int32_t *assign,
                   const int32_t *prompt_len, const int32_t *dec, int32_t mode, double t_now,
                   int64_t max_batches, const int32_t *block_size, const int64_t *num_blocks,
                   const int64_t *max_ctx, int64_t *run_id, int64_t *wait_id, int64_t id_base,
                   double *first_token_time)
{
    const int track = run_id != NULL && wait_id != NULL && first_token_time != NULL;
    int rc_all = ORC_OK;
    for (int32_t j = 0; j < I; ++j) {
        const int64_t bs = block_size[j], nb = num_blocks[j], mc = max_ctx[j];
        const int64_t total = (int64_t)cap_running + cap_waiting + Q + 1;
        orc_req *run = (orc_req *)calloc((size_t)total, sizeof(orc_req));
        orc_req *next = (orc_req *)calloc((size_t)total, sizeof(orc_req));  /* the planned running list */
        orc_req *wait = (orc_req *)calloc((size_t)(2 * total + 1), sizeof(orc_req)); /* room at the front */
        int64_t *alloc = (int64_t *)calloc((size_t)total, sizeof(int64_t));
        int *kind = (int *)calloc((size_t)total, sizeof(int));
        if (!run || !next || !wait || !alloc || !kind) {
            free(run); free(next); free(wait); free(alloc); free(kind);
            return ORC_ENOMEM;
        }
        int64_t nr = 0, wh = total, we = total;  /* waiting queue: wait[wh .. we) */
        int64_t free_blocks = nb;
        for (int32_t r = 0; r < n_run[j]; ++r) {
            const int64_t o = (int64_t)j * cap_running + r;
            run[nr].ctx = run_ctx[o]; run[nr].pre = run_pre[o]; run[nr].dec = run_dec[o]; run[nr].is_query = 0;
            run[nr].id = track ? run_id[o] : -1;
            free_blocks -= kv_blocks(run[nr].ctx, bs);
            ++nr;
        }
        for (int32_t w = 0; w < n_wait[j]; ++w) {
            const int64_t o = (int64_t)j * cap_waiting + w;
            wait[we].ctx = 0; wait[we].pre = wait_pre[o]; wait[we].dec = wait_dec[o]; wait[we].is_query = 0;
            wait[we].id = track ? wait_id[o] : -1;
            ++we;
        }
        int rc = ORC_OK;
        /* 1. the routed queries join the waiting tail in query order */
        for (int32_t i = 0; i < Q; ++i) {
            if (assign[i] != j) continue;
            if ((int64_t)prompt_len[i] >= mc || kv_blocks(min64((int64_t)prompt_len[i] + dec[i], mc), bs) > nb)
                rc = ORC_EINVAL;
            wait[we].ctx = 0; wait[we].pre = prompt_len[i]; wait[we].dec = dec[i]; wait[we].is_query = 0;
            wait[we].id = (track && id_base >= 0) ? id_base + i : -1;
            ++we;
        }
        if (rc == ORC_OK && we - wh > cap_waiting) rc = ORC_ELIMIT;
        const float *cf = coef + 5 * model_of_instance[j];
        double t = clock[j];
        /* 2. execute whole batches that end by t_now */
        for (int64_t step = 0; rc == ORC_OK; ++step) {
            if (nr == 0 && wh == we) {                        /* idle: nothing to run */
                if (t < t_now) t = t_now;
                break;
            }
            if (step >= max_batches) { rc = ORC_ELIMIT; break; }
            /* plan the batch on a copy of the running list; a preempted request is written
             * below the waiting head, which moves only if the batch runs */
            memcpy(next, run, sizeof(orc_req) * (size_t)nr);
            int64_t pnr = nr, pwh = wh, pfree = free_blocks;
            int64_t budget = B[j];
            for (int64_t r = 0; r < nr; ++r) { kind[r] = SCHED_NONE; alloc[r] = 0; }
            int64_t r = 0;
            while (r < pnr && budget > 0) {
                const int64_t x = next[r].pre > 0 ? min64(next[r].pre, budget) : 1;
                const int64_t need = kv_blocks(next[r].ctx + x, bs) - kv_blocks(next[r].ctx, bs);
                while (pfree < need && pnr - 1 >= r) {          /* preempt the last running request */
                    orc_req v = next[pnr - 1];
                    pfree += kv_blocks(v.ctx, bs);
                    v.pre += v.ctx;
                    v.ctx = 0;
                    wait[--pwh] = v;
                    --pnr;
                }
                if (r >= pnr) break;                             /* r preempted itself */
                pfree -= need;
                alloc[r] = x;
                kind[r] = next[r].pre > 0 ? SCHED_PREFILL : SCHED_DECODE;
                budget -= x;
                ++r;
            }
            while (budget > 0 && pwh < we && pnr < S[j]) {      /* admission */
                const int64_t x = min64(wait[pwh].pre, budget);
                const int64_t need = kv_blocks(x, bs);
                if (pfree < need) break;
                pfree -= need;
                next[pnr] = wait[pwh++];
                alloc[pnr] = x;
                kind[pnr] = SCHED_PREFILL;
                budget -= x;
                ++pnr;
            }
            int64_t F[5] = {1, 0, 0, 0, 0};
            for (int64_t q = 0; q < pnr; ++q) {
                if (kind[q] == SCHED_PREFILL) {
                    const int64_t x = alloc[q];
                    F[1] += x;
                    F[4] += x * next[q].ctx + x * (x + 1) / 2;
                } else if (kind[q] == SCHED_DECODE) {
                    F[2] += 1;
                    F[3] += next[q].ctx;
                }
            }
            const float T = orc_ttft_f32(cf, F);   /* Eq. 9 for this one batch */
            if (t + (double)T > t_now) break;       /* still running at t_now */
            if (pnr > cap_running) { rc = ORC_ELIMIT; break; }
            /* apply the batch */
            for (int64_t q = 0; q < pnr; ++q) {
                if (kind[q] == SCHED_PREFILL) {
                    next[q].ctx += alloc[q];
                    next[q].pre -= alloc[q];
                    if (next[q].pre == 0 && mode == ORC_FIRST_TOKEN_WITH_LAST_CHUNK) {
                        next[q].dec -= 1;
                        if (track) first_token(&next[q], 1, t + (double)T, first_token_time);
                    }
                } else if (kind[q] == SCHED_DECODE) {
                    next[q].ctx += 1;
                    next[q].dec -= 1;
                    if (track) first_token(&next[q], mode == ORC_FIRST_TOKEN_SEPARATE_DECODE, t + (double)T,
                                           first_token_time);
                }
                if (next[q].pre == 0 && next[q].ctx >= mc) next[q].dec = 0;  /* context limit */
            }
            int64_t keep = 0;
            for (int64_t q = 0; q < pnr; ++q) {
                if (next[q].dec > 0) run[keep++] = next[q];
                else pfree += kv_blocks(next[q].ctx, bs);      /* finished: its blocks return */
            }
            nr = keep;
            wh = pwh;
            free_blocks = pfree;
            t += (double)T;
            if (we - wh > cap_waiting) { rc = ORC_ELIMIT; break; }
        }
        if (rc == ORC_OK) {
            n_run[j] = (int32_t)nr;
            for (int64_t q = 0; q < cap_running; ++q) {
                const int64_t o = (int64_t)j * cap_running + q;
                run_ctx[o] = q < nr ? (int32_t)run[q].ctx : 0;
                run_pre[o] = q < nr ? (int32_t)run[q].pre : 0;
                run_dec[o] = q < nr ? (int32_t)run[q].dec : 0;
                if (track) run_id[o] = q < nr ? run[q].id : -1;
            }
            n_wait[j] = (int32_t)(we - wh);
            for (int64_t w = 0; w < cap_waiting; ++w) {
                const int64_t o = (int64_t)j * cap_waiting + w;
                wait_pre[o] = w < we - wh ? (int32_t)wait[wh + w].pre : 0;
                wait_dec[o] = w < we - wh ? (int32_t)wait[wh + w].dec : 0;
                if (track) wait_id[o] = w < we - wh ? wait[wh + w].id : -1;
            }
            clock[j] = t;
        } else {
            rc_all = rc;
        }
        free(run); free(next); free(wait); free(alloc); free(kind);
    }
    return rc_all;
}
