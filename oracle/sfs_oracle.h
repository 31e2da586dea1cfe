/*
 * CPU oracle for the latency-aware router (test infrastructure only).
 *
 * Plain, slow, literal C: for every (query, instance) candidate it copies the
 * instance's resident set, appends the query at the FCFS waiting tail and
 * steps the serving scheduler one token batch at a time until the query's
 * first output token (Sec. 4.1, Eq. 7 and Eq. 8), accumulating the five batch
 * features that Eq. 9 is linear in.  Routing is brute-force enumeration over
 * instances (Eq. 2, Eq. 3, Eq. 5).
 *
 * Only the test suite, the package smoke check and the benchmark's CPU
 * baseline use this library.  It shares no code, header or constant with the
 * CUDA library and is never on the product path.
 */
#ifndef SFS_ORACLE_H
#define SFS_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum { ORC_OK = 0, ORC_EINVAL = 1, ORC_ELIMIT = 2, ORC_ENOMEM = 3 };
enum { ORC_FIRST_TOKEN_SEPARATE_DECODE = 0, ORC_FIRST_TOKEN_WITH_LAST_CHUNK = 1 };

/* One instance's snapshot: running list (admission order) and waiting list (FCFS order). */
typedef struct {
    int32_t n_run;
    const int32_t *run_ctx, *run_pre, *run_dec;
    int32_t n_wait;
    const int32_t *wait_pre, *wait_dec;
} orc_instance;

/* Simulate one candidate: instance `inst` with budget B and sequence cap S plus a new
 * query of prompt p and predicted decode d appended at the waiting tail.
 * Writes F[5] = (batches, prefill tokens, decode tokens, sum ctx*dec, sum prefill
 * attention pairs) over batches 1..l_ttft, the batch index that admitted the query
 * and the query's first-token batch.  Returns ORC_ELIMIT after max_batches. */
int orc_sfs_candidate(const orc_instance *inst, int32_t B, int32_t S, int32_t mode,
                      int32_t p, int32_t d, int64_t max_batches,
                      int64_t F[5], int64_t *l_admit, int64_t *l_ttft);

/* KV-cache limits of one instance (App. F names context limits, KV-cache
 * allocation and preemption among what the simulation models): block_size tokens
 * per block, num_blocks blocks, and max_ctx, the longest context a request may
 * reach. */
typedef struct {
    int32_t block_size;
    int64_t num_blocks;
    int64_t max_ctx;
} orc_kv;

/* orc_sfs_candidate with the KV-cache limits of `kv` (the step rule in sfs_oracle.c).
 * If res_F is not NULL it receives, for each batch 1..l_ttft, the features of the
 * batch without the query's own tokens ([l_ttft][5], room for max_batches rows);
 * *max_used (may be NULL) receives the most blocks in use at the end of any batch's
 * scheduling.  Returns ORC_EINVAL if the residents hold more blocks than the
 * instance has, a context reaches max_ctx in the input, p >= max_ctx, or a request's
 * whole context (capped at max_ctx) needs more blocks than the instance has. */
int orc_sfs_candidate_kv(const orc_instance *inst, int32_t B, int32_t S, int32_t mode, const orc_kv *kv,
                         int32_t p, int32_t d, int64_t max_batches,
                         int64_t F[5], int64_t *l_admit, int64_t *l_ttft, int64_t *res_F, int64_t *max_used);

/* The residents alone (no query) for exactly L batches under the same rule:
 * res_F[L][5] per-batch features. */
int orc_kv_residents(const orc_instance *inst, int32_t B, int32_t S, int32_t mode, const orc_kv *kv,
                     int64_t L, int64_t *res_F);

/* Every candidate of a list under per-instance KV limits, the query taken up to its
 * first token (one output token).  status[c] receives the candidate's return code
 * (ORC_OK, ORC_EINVAL for an invalid snapshot or query, ORC_ELIMIT past max_batches);
 * a failed candidate gets F = -1, l_ttft = -1 and NaN times.  Returns ORC_EINVAL only
 * for a bad candidate index or row count. */
int orc_estimate_candidates_kv(int32_t num_instances, const int32_t *model_of_instance,
                               const float *coef, const int32_t *B, const int32_t *S,
                               int32_t cap_running, int32_t cap_waiting,
                               const int32_t *n_run, const int32_t *run_ctx, const int32_t *run_pre,
                               const int32_t *run_dec, const int32_t *n_wait, const int32_t *wait_pre,
                               const int32_t *wait_dec, const int32_t *prompt_len,
                               const int32_t *block_size, const int64_t *num_blocks, const int64_t *max_ctx,
                               int32_t mode, int64_t max_batches,
                               int64_t num_cand, const int32_t *cand_q, const int32_t *cand_j,
                               int32_t *status, int64_t *F, int64_t *l_ttft, float *ttft32, double *ttft64);

/* Canonical single-precision batch-time sum (Eq. 9 summed per Eq. 8) and its fp64 value. */
float orc_ttft_f32(const float coef[5], const int64_t F[5]);
double orc_ttft_f64(const float coef[5], const int64_t F[5]);

/* Every candidate of a list: cand_q[c], cand_j[c] index the queries / instances.
 * State arrays are [I][cap] row-major.  Outputs per candidate: F[c][5],
 * l_ttft[c], ttft32[c], ttft64[c]. */
int orc_estimate_candidates(int32_t num_instances, const int32_t *model_of_instance,
                            const float *coef, const int32_t *B, const int32_t *S,
                            int32_t cap_running, int32_t cap_waiting,
                            const int32_t *n_run, const int32_t *run_ctx, const int32_t *run_pre,
                            const int32_t *run_dec, const int32_t *n_wait, const int32_t *wait_pre,
                            const int32_t *wait_dec, int32_t num_models, const int32_t *prompt_len,
                            const int32_t *dec_hat, int32_t mode, int64_t max_batches,
                            int64_t num_cand, const int32_t *cand_q, const int32_t *cand_j,
                            int64_t *F, int64_t *l_ttft, float *ttft32, double *ttft64);

/* Brute-force routing of Q queries given their full TTFT rows ttft[Q][I] (canonical fp32).
 * tau == NULL: Lagrangian objective (Eq. 5) for each of the P (lambda, mu) pairs.
 * tau != NULL: constrained objective (Eq. 3) for each lambda; mu is ignored.
 * A candidate whose TTFT is NaN (no estimate: an invalid prompt, or an instance that
 * cannot take the query under KV limits) is not eligible; a query with no eligible
 * instance gets assign -1 and NaN utility and TTFT.
 * Outputs [P][Q]: assign, util (U of the chosen instance), ttft_chosen. */
int orc_route(int32_t Q, int32_t I, int32_t M, const int32_t *model_of_instance,
              const float *price_in, const float *price_out, const int32_t *prompt_len,
              const int32_t *dec_hat, const float *acc, const float *ttft, const float *tau,
              int32_t P, const float *lambda, const float *mu,
              int32_t *assign, float *util, float *ttft_chosen);

/* Per-pair means of accuracy, cost and TTFT of the chosen instances: out[P][3]. */
int orc_frontier(int32_t Q, int32_t I, int32_t M, const int32_t *model_of_instance,
                 const float *price_in, const float *price_out, const int32_t *prompt_len,
                 const int32_t *dec_hat, const float *acc, int32_t P, const int32_t *assign,
                 const float *ttft_chosen, double *out);

/* Online stream step: append the routed queries (assign[i] >= 0) to their instances'
 * waiting queues in query order, then advance every instance by the whole token batches
 * that end by t_now, each taking the Eq. 9 time of its own composition (canonical fp32,
 * accumulated in fp64 clocks).  An instance with nothing to run jumps to t_now.  State
 * arrays ([I][cap] row-major) and clocks are updated in place.  Returns ORC_ELIMIT if a
 * queue would exceed its capacity or an instance needs more than max_batches batches. */
int orc_advance(int32_t I, const int32_t *model_of_instance, const float *coef, const int32_t *B,
                const int32_t *S, int32_t cap_running, int32_t cap_waiting, int32_t *n_run,
                int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre,
                int32_t *wait_dec, double *clock, int32_t Q, const int32_t *assign,
                const int32_t *prompt_len, const int32_t *dec, int32_t mode, double t_now,
                int64_t max_batches);

/* orc_advance that also follows tracked queries to their first output token (Sec. 4.1;
 * Eq. 4 scores the realized TTFT).  run_id / wait_id ([I][cap], in/out) hold each
 * request's tracking id or -1; routed query i joins as id_base + i (id_base < 0: -1).
 * When a tracked request emits its first output token in an executed batch -- its first
 * decode token, or the last prompt chunk's token when the first token comes with it --
 * first_token_time[id] receives that batch's end time and the request's id becomes -1.
 * NULL id arrays: nothing is tracked (exactly orc_advance). */
int orc_advance_ids(int32_t I, const int32_t *model_of_instance, const float *coef, const int32_t *B,
                    const int32_t *S, int32_t cap_running, int32_t cap_waiting, int32_t *n_run,
                    int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre,
                    int32_t *wait_dec, double *clock, int32_t Q, const int32_t *assign,
                    const int32_t *prompt_len, const int32_t *dec, int32_t mode, double t_now,
                    int64_t max_batches, int64_t *run_id, int64_t *wait_id, int64_t id_base,
                    double *first_token_time);

/* orc_advance_ids under per-instance KV-cache limits (block_size, num_blocks, max_ctx
 * [I]): each executed batch follows the KV step rule of orc_sfs_candidate_kv (blocks
 * found in running order with preemption of the last running request, admission only
 * with the first chunk's blocks, the context limit ending a request).  ORC_EINVAL for a
 * routed query that could never run (prompt at max_ctx, or its capped whole context
 * needing more blocks than the instance has). */
int orc_advance_kv(int32_t I, const int32_t *model_of_instance, const float *coef, const int32_t *B,
                   const int32_t *S, int32_t cap_running, int32_t cap_waiting, int32_t *n_run,
                   int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre,
                   int32_t *wait_dec, double *clock, int32_t Q, const int32_t *assign,
                   const int32_t *prompt_len, const int32_t *dec, int32_t mode, double t_now,
                   int64_t max_batches, const int32_t *block_size, const int64_t *num_blocks,
                   const int64_t *max_ctx, int64_t *run_id, int64_t *wait_id, int64_t id_base,
                   double *first_token_time);

/* Utility of Eq. 2 with the cost of App. B.4 in canonical fp32. */
float orc_utility(float acc, float lambda, int32_t p, int32_t dec_hat, float price_in, float price_out);

/* ---- Average-case TTFT estimators (Sec. 4, average-case TTFT estimation; App. E) ---- */

/* x^k for an integer k >= 0 by binary exponentiation (bits of k from the least
 * significant; a fixed sequence of IEEE products). */
double orc_pow_int(double x, int32_t k);

/* Expected LPS queueing delay (App. E, boxed result; G/G/k correction at its end):
 * rho = alpha / mu, E[W] = ((ca2 + cs2) / 2) * rho^k / (mu - alpha).  NaN unless
 * 0 <= alpha < mu, k >= 1. */
double orc_lps_wait(double alpha, double mu, int32_t k, double ca2, double cs2);

/* Throughput-based waiting time (Sec. 4, prefill-throughput estimator): remaining
 * prefill tokens of every resident request / theta. */
double orc_throughput_wait(const orc_instance *inst, double theta);

/* TTFT = W_j + p_i / theta_j + Tdec_j for every query i and instance j (outputs [Q][I]):
 * canonical fp32 fmaf((float)p, (float)(1 / theta), (float)(W + Tdec)) and fp64. */
int orc_avgcase_ttft(int32_t I, int32_t Q, const double *W, const double *theta, const double *tdec,
                     const int32_t *prompt_len, float *t32, double *t64);

/* ---- Baseline routing policies and stream metrics (Sec. 6 baselines; Eq. 4) ---- */

/* Round Robin: query q goes to instance (start + q) mod I, whatever the load,
 * utility or latency. */
int orc_round_robin(int32_t Q, int32_t I, int64_t start, int32_t *assign);

/* Shortest Queue: the queries in order each go to the instance with the fewest
 * resident requests, counting the queries routed before them (ties to the lowest
 * index).  counts[I] are the resident requests (running + waiting) at the start. */
int orc_shortest_queue(int32_t Q, int32_t I, const int32_t *counts, int32_t *assign);

/* Latency-Agnostic: argmax over instances of the utility of Eq. 2 (ties to the lowest
 * index), i.e. Eq. 5 with mu = 0. */
int orc_latency_agnostic(int32_t Q, int32_t I, int32_t M, const int32_t *model_of_instance,
                         const float *price_in, const float *price_out, const int32_t *prompt_len,
                         const int32_t *dec_hat, const float *acc, float lambda, int32_t *assign);

/* OnTimeUtility (Eq. 4) and SLO attainment over Q routed queries.  The realized TTFT
 * of query i is the fp32 sum delay_i + ttft_i (delay NULL: 0); it is on time if that
 * is <= tau_i (NaN never is).  out[0] = (1/Q) sum of util_i over on-time queries,
 * out[1] = (on-time count) / Q; fp64 sums in index order. */
int orc_on_time_utility(int32_t Q, const float *util, const float *ttft, const float *tau,
                        const float *delay, double *out);

#ifdef __cplusplus
}
#endif
#endif
