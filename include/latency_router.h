/*
 * latency_router.h -- C ABI of the GB300 latency-aware router hot path.
 *
 * The library estimates, for every (query, model instance) candidate, the
 * time to first token by the Serving Framework Simulation of Sec. 4.1: the
 * instance's resident requests plus the new query at the tail of its FCFS
 * waiting queue are stepped through token batches (chunked prefill under a
 * token budget and a sequence cap) until the query's first output token
 * (Eq. 7); the estimate is the sum over those batches (Eq. 8) of the batch
 * time model of Eq. 9.  It then scores each candidate with the accuracy-cost
 * utility of Eq. 2 and picks one instance per query by the Lagrangian
 * objective of Eq. 5 or the latency-constrained objective of Eq. 3.
 * Also: the online stream (lr_advance), the average-case TTFT sources of Sec. 4 /
 * App. E (lr_set_queue_params, lr_set_ttft_source), KV-cache block and context
 * limits with preemption (lr_set_kv_limits), least-squares calibration of the
 * batch-time coefficients (lr_calibrate), and the baseline routers with
 * OnTimeUtility (lr_route_baseline, lr_on_time_utility).
 *
 * Conventions for every call:
 *  - All integers are int32 unless stated; all arrays are dense, row-major.
 *  - Configuration arrays passed to lr_create are host pointers, copied.
 *  - Per-call arrays are DEVICE pointers owned by the caller; the library
 *    reads or writes them only inside work enqueued on `cuda_stream`
 *    (a cudaStream_t; NULL means the legacy default stream).
 *  - Calls are asynchronous on that stream.  Calls on one context must be
 *    ordered by the caller (one stream, or events between streams).
 *  - Errors a host can see (null pointers, sizes beyond capacity, invalid
 *    limits) are returned immediately and nothing is enqueued.  Errors found
 *    on the device (an invalid snapshot, a trajectory longer than max_iters,
 *    a prompt length out of range) are recorded in a device status word that
 *    lr_status() returns; affected outputs are NaN (times) or -1 (indices).
 *  - The library never aborts, throws or leaves a device loop unbounded.
 */
#ifndef LATENCY_ROUTER_H
#define LATENCY_ROUTER_H

#include <stdint.h>

#if defined(__GNUC__)
#define LR_API __attribute__((visibility("default")))
#else
#define LR_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

/* Return codes. */
enum lr_code {
    LR_OK = 0,
    LR_EINVAL = 1,      /* invalid argument or invalid input value */
    LR_ENOMEM = 2,      /* device or host allocation failed */
    LR_ECUDA = 3,       /* a CUDA runtime call failed (see lr_last_error) */
    LR_ECAPACITY = 4,   /* a size exceeds what the context was created for */
    LR_ETRAJ = 5,       /* a simulated trajectory exceeded max_iters (device) */
    LR_ESTATE = 6,      /* a snapshot violates the state preconditions (device) */
    LR_ENOSTATE = 7     /* no snapshot has been loaded successfully yet (device) */
};

/* When the first output token is produced (Sec. 4.1: decoding starts once every
 * prompt token has been processed). */
enum lr_first_token_mode {
    LR_FIRST_TOKEN_SEPARATE_DECODE = 0,  /* its own decode batch after the last prefill chunk (default) */
    LR_FIRST_TOKEN_WITH_LAST_CHUNK = 1   /* sampled in the batch that completes the prompt */
};

/* Pool description (Sec. 3, the system model; Eq. 9 coefficients; App. B.4 prices). */
typedef struct {
    int32_t num_instances;             /* I >= 1 model instances j */
    int32_t num_models;                /* M >= 1 distinct models */
    const int32_t *model_of_instance;  /* [I] in [0, M) */
    const float *coef;                 /* [M][5] Eq. 9 coefficients in seconds:
                                          beta0 (per batch), beta1p (per prefill token),
                                          beta1d (per decode token), beta2 (per decode token
                                          and token of context), beta3 (per prefill attention
                                          pair); the paper's form has beta1p == beta1d.
                                          Finite and >= 0. */
    const float *price_in;             /* [M] $ per prompt token, finite >= 0 */
    const float *price_out;            /* [M] $ per response token, finite >= 0 */
    const int32_t *max_batched_tokens; /* [I] token budget B_j per batch, 1..2^24 */
    const int32_t *max_seqs;           /* [I] sequence cap S_j, 1 <= S_j <= B_j */
    int32_t cap_running;               /* row stride of the running arrays (>= 1) */
    int32_t cap_waiting;               /* row stride of the waiting arrays (>= 1) */
    int32_t max_queries;               /* largest Q of any call, 1 .. 2^30 */
    int32_t max_pairs;                 /* largest P of lr_route, 1..64 */
    int32_t max_prompt_len;            /* largest prompt length of any query, 1..2^20 */
    int32_t first_token_mode;          /* enum lr_first_token_mode */
    int32_t max_iters;                 /* bound on simulation steps per instance and load */
} lr_config;

/* One snapshot of every instance (Sec. 4 setup: resident set R_j = Q_j u A_j with
 * remaining prefill and predicted decode tokens; App. F on workload snapshots).
 * DEVICE pointers.  Per-instance arrays are [I]; per-request arrays are
 * [I][cap] with row stride cap_running / cap_waiting; entries beyond a row's
 * count are ignored.
 * Preconditions, checked on the device (LR_ESTATE): 0 <= n_run[j] <= min(cap_running,
 * S_j); 0 <= n_wait[j] <= cap_waiting; run_ctx in [0, 2^28]; run_pre in [0, 2^24];
 * run_dec and wait_dec in [1, 2^24]; wait_pre in [1, 2^24] and at most 2^30 in total per
 * instance; only the LAST running request of a row may have run_pre > 0 (the state a
 * chunked-prefill FCFS engine is in after any batch). */
typedef struct {
    const int32_t *n_run;      /* [I] running requests (admission order) */
    const int32_t *run_ctx;    /* [I][cap_running] tokens already in the KV cache */
    const int32_t *run_pre;    /* [I][cap_running] remaining prefill tokens */
    const int32_t *run_dec;    /* [I][cap_running] remaining predicted decode tokens */
    const int32_t *n_wait;     /* [I] waiting requests (FCFS order) */
    const int32_t *wait_pre;   /* [I][cap_waiting] prompt tokens */
    const int32_t *wait_dec;   /* [I][cap_waiting] predicted decode tokens */
} lr_state_view;

typedef struct lr_ctx lr_ctx;  /* opaque, owned by the library */

/* Create a context on the current CUDA device.  Copies the configuration and
 * allocates all device memory the other calls need.  *out is set on LR_OK. */
LR_API int lr_create(const lr_config *cfg, lr_ctx **out);

/* Free everything lr_create allocated.  Synchronizes the device first.  NULL is a no-op. */
LR_API int lr_destroy(lr_ctx *ctx);

/* Ingest a snapshot (App. F): copies it into library memory and summarizes, per
 * instance, the query-independent part of the simulation -- the batch at which a
 * query appended now would be admitted, the budget left to it in that and the
 * following batches, and the resident batch features up to each of them.  The
 * snapshot is written to a back buffer and becomes the live one only if every
 * instance is valid and simulates within max_iters; otherwise the previous live
 * snapshot stays in use (App. F: the router keeps its last complete copy) and the
 * status word records LR_ESTATE or LR_ETRAJ.
 * Overlap: a load (or lr_advance) may run on one stream while lr_estimate_ttft /
 * lr_route run on another; each CTA of those calls uses the snapshot that is live
 * when it starts, so every query row is computed against one complete snapshot, the
 * previous or the new one (App. F: the router estimates from its most recent complete
 * copy while the next is prepared).  The back buffer a load writes is the one the
 * snapshot before the live one occupied, so order the next load after every
 * estimate or route call issued before the previous load finished (at most one load
 * in flight). */
LR_API int lr_load_state(lr_ctx *ctx, const lr_state_view *state, void *cuda_stream);

/* SFS TTFT estimates (Eq. 8 with Eq. 9) for every candidate of Q queries.
 * prompt_len: [Q] device, each in [1, max_prompt_len] (else that row is NaN and the
 * status word records LR_EINVAL).  ttft_out: [Q][I] device fp32 seconds.
 * first_batch_out: [Q][I] device int32 index of the first-token batch (Eq. 7), or NULL.
 * Q may be 0. */
LR_API int lr_estimate_ttft(lr_ctx *ctx, int32_t Q, const int32_t *prompt_len, float *ttft_out,
                     int32_t *first_batch_out, void *cuda_stream);

/* The integer batch features behind each estimate: features_out [Q][I][5] int64 device,
 * F = (batches, prefill tokens, decode tokens, sum of decode-token context, sum over
 * prefill chunks of x*c + x(x+1)/2) summed over batches 1..l_TTFT (Eq. 7-9), so that
 * TTFT = beta . F.  Rows with an invalid prompt length are -1. */
LR_API int lr_estimate_features(lr_ctx *ctx, int32_t Q, const int32_t *prompt_len, int64_t *features_out,
                         void *cuda_stream);

/* Route Q queries for each of P trade-off pairs.
 *  prompt_len [Q], dec_hat [Q][M] (predicted response tokens, >= 0), acc [Q][M]
 *  (predicted accuracy, finite): device.
 *  cost_{i,j} = p_i * price_in_m + dec_hat_{i,m} * price_out_m (App. B.4),
 *  U = acc - lambda * cost (Eq. 2).
 *  tau == NULL: Lagrangian objective (Eq. 5), argmax_j U - mu * TTFT.
 *  tau != NULL ([Q] device, seconds): constrained objective (Eq. 3), argmax U over
 *  {j : TTFT <= tau_i}, or the least TTFT when that set is empty; it takes one
 *  lambda (P == 1, else LR_EINVAL), and mu is then unused and may be NULL.
 *  Ties go to the lowest instance index.  A candidate whose TTFT is NaN (no
 *  estimate: an invalid prompt, or an instance that cannot take the query under
 *  KV limits) is never chosen; a query with no eligible instance gets assign -1
 *  and NaN utility and TTFT.
 *  lambda, mu: [P] HOST arrays, finite and >= 0, 1 <= P <= max_pairs.
 *  Outputs, device: assign_out [P][Q] int32, util_out [P][Q] fp32 U of the chosen
 *  instance, ttft_chosen_out [P][Q] fp32 or NULL, frontier_out [P][3] fp64 means of
 *  (accuracy, cost, TTFT) of the chosen instances or NULL, ttft_matrix_out [Q][I] fp32
 *  (the full estimate matrix, as lr_estimate_ttft writes it) or NULL.
 *  Requires I <= 1024. */
LR_API int lr_route(lr_ctx *ctx, int32_t Q, const int32_t *prompt_len, const int32_t *dec_hat, const float *acc,
             const float *tau, int32_t P, const float *lambda, const float *mu, int32_t *assign_out,
             float *util_out, float *ttft_chosen_out, double *frontier_out, float *ttft_matrix_out,
             void *cuda_stream);

/* lr_route with the frontier, for callers that must not allocate device memory while
 * serving (the paper has no counterpart: it is a memory-management variant of lr_route).
 * A serving loop that runs inside a fixed device-memory reservation, or that cannot let
 * an allocation synchronize the device between its launches, cannot call cudaMalloc (or
 * an allocating library routine) on the request path.  This call allocates nothing: the
 * per-(pair, query) chosen-TTFT values that the frontier averages live in one fixed array
 * of the library's static device memory (LR_STATIC_ROUTE_CAP fp32 entries, 1 MiB) instead
 * of memory taken from the context.  Arguments and outputs are those of lr_route with
 * ttft_chosen_out and ttft_matrix_out absent; frontier_out is required.
 *  - Requires P * Q <= LR_STATIC_ROUTE_CAP, else LR_ECAPACITY before any launch.
 *  - Set-up: lr_create (the context's device current) looks up the array's device
 *    address once and keeps it in the context; this call itself makes no runtime
 *    query of it, so a capture may begin at any point after lr_create.
 *  - Nothing in the array needs to start at zero: every entry the frontier reads is
 *    written earlier in the same call, in stream order.
 *  - The array is shared by every context on a device: two of these calls in flight at
 *    once on one device (different streams, or different contexts) race on it, so order
 *    them (one stream, or events). */
#define LR_STATIC_ROUTE_CAP (1 << 18)
LR_API int lr_route_frontier_static(lr_ctx *ctx, int32_t Q, const int32_t *prompt_len, const int32_t *dec_hat,
                                    const float *acc, const float *tau, int32_t P, const float *lambda,
                                    const float *mu, int32_t *assign_out, float *util_out, double *frontier_out,
                                    void *cuda_stream);

/* Where the TTFT of lr_estimate_ttft and lr_route (and lr_route_frontier_static) comes from. */
enum lr_ttft_source {
    LR_TTFT_SFS = 0,         /* Serving Framework Simulation of the live snapshot (Sec. 4.1), the default */
    LR_TTFT_THROUGHPUT = 1,  /* prefill-throughput estimator (Sec. 4): W_j = remaining prefill tokens of
                                the snapshot's residents / theta_j */
    LR_TTFT_LPS = 2          /* average-case estimator (Sec. 4, App. E): W_j = ((ca2 + cs2) / 2) *
                                (alpha_j / mu_j)^k_j / (mu_j - alpha_j); needs no snapshot */
};

/* Per-instance parameters of the average-case sources; host arrays of length I, copied.
 * TTFT_ij = W_j + p_i / theta_j + Tdec_j, evaluated as
 * fmaf((float)p, fp32(1 / theta_j), fp32(W_j + Tdec_j)) with W_j and the divisions in fp64
 * ((alpha/mu)^k by binary exponentiation over the bits of k from the least significant). */
typedef struct {
    const double *prefill_tput;       /* theta_j, prefill tokens per second, finite > 0 */
    const double *decode_batch_time;  /* Tdec_j, average decode-batch time (s), finite >= 0 */
    const double *arrival_rate;       /* alpha_j, queries/s, 0 <= alpha_j < mu_j; NULL: no LPS source */
    const double *service_rate;       /* mu_j, queries/s (App. E: from peak output throughput) */
    const int32_t *parallelism;       /* k_j, concurrent sequences, 1 .. 2^20 */
    const double *arrival_scv;        /* ca^2_j >= 0 of inter-arrival times, NULL: 1 (Poisson) */
    const double *service_scv;        /* cs^2_j >= 0 of service requirements, NULL: 1 (exponential) */
} lr_queue_params;

/* Validate and upload the queue parameters (LR_EINVAL, nothing changed, on a bad value);
 * ordered on cuda_stream like the other calls. */
LR_API int lr_set_queue_params(lr_ctx *ctx, const lr_queue_params *params, void *cuda_stream);

/* Select the TTFT source (lr_ttft_source).  The average-case sources need
 * lr_set_queue_params first (LPS: with rates), else LR_EINVAL.  first_batch_out of
 * lr_estimate_ttft and lr_estimate_features describe the SFS only; first_batch_out with
 * another source is LR_EINVAL.  The throughput source reads the live snapshot
 * (LR_ENOSTATE before one is loaded); the LPS source reads none. */
LR_API int lr_set_ttft_source(lr_ctx *ctx, int32_t source);

/* KV-cache limits in the simulated step rule (App. F counts context limits, the
 * state of KV-cache allocation and preemption among what the simulation models,
 * without a rule).  Reading:
 * instance j has num_blocks[j] blocks of block_size[j] tokens, a request with c
 * tokens in the cache holds ceil(c / block_size) of them; a running request whose
 * tokens of a batch need blocks that are not free preempts the last running request
 * (its blocks return, its whole context becomes prefill again and it goes to the
 * front of the waiting queue), preempting itself if it is the last; the waiting
 * head is admitted only if its first chunk's blocks are free; a request whose
 * context reaches max_ctx[j] ends there.  The query appended at the waiting tail
 * never changes the residents' batches, so every later lr_load_state simulates
 * each instance's residents once, recording up to `horizon` batches from the first
 * one in which a query could be admitted, and lr_estimate_ttft /
 * lr_estimate_features follow each query through those records.
 * block_size [I] int32 in [1, 4096], num_blocks [I] int64 in [1, 2^40], max_ctx [I]
 * int64 in [2, 2^40]: host arrays, copied.  horizon in [1, 2^16].  All three arrays
 * NULL turns the limits off (the default).  The call synchronizes the device and drops
 * the live snapshot: estimates return LR_ENOSTATE until the next lr_load_state.
 * With limits on, lr_route and lr_route_frontier_static first write the KV-limited
 * estimate matrix (to ttft_matrix_out if given, else to library memory) and score
 * and pick over it; lr_route_baseline reports the chosen instance's KV-limited time;
 * lr_advance executes the same rule; the average-case sources return LR_EINVAL.  Each estimate call
 * runs one walk per distinct prompt length (the queries are counting-sorted by
 * length in library memory sized by max_queries).  Memory taken here: per buffer
 * 68 B x I x horizon of records, and max_queries x (8 B + 4 B x I) for the sort
 * and the routed matrix (LR_ENOMEM if it cannot be had; nothing is allocated
 * later, so routing stays allocation-free).  Device errors: a snapshot in which a running request other than the last is
 * in prefill, a context has reached max_ctx, the residents hold more blocks than the
 * instance has, or a request's whole context (capped at max_ctx) needs more blocks than
 * the instance has, is LR_ESTATE; a query whose prompt is not below max_ctx, or whose
 * prompt and first token need more blocks than the instance has, gets NaN (features -1)
 * and LR_EINVAL; one that needs batches past the recorded horizon gets NaN and
 * LR_ETRAJ. */
LR_API int lr_set_kv_limits(lr_ctx *ctx, const int32_t *block_size, const int64_t *num_blocks,
                            const int64_t *max_ctx, int32_t horizon);

/* Least-squares calibration of the Eq. 9 coefficients per model from a log of executed
 * token batches (Sec. 4.1: calibrated from observed token-batch processing times).
 * features: [N][5] int64 device, each batch's (F0 = 1, prefill tokens, decode tokens, sum of
 * decode-token contexts, sum over prefill chunks of x*c + x(x+1)/2); model: [N] int32 device
 * in [0, M); time: [N] fp64 device, observed seconds.  shared_beta1 != 0 fits the paper's
 * four-coefficient form (one beta1, regressor F1 + F2), otherwise five coefficients.
 * coef_out: [M][5] fp64 device (beta0, beta1p, beta1d, beta2, beta3), NaN for a model with
 * fewer rows than unknowns or a rank-deficient design.  The sums are exact integers
 * (features must lie in [0, 2^32), times in [0, 2^19) s, kept to 2^-44 s, N < 2^32); rows
 * outside those ranges or with a model outside [0, M) are skipped and record LR_EINVAL.
 * Rows grouped by model are the fast case.  Requires num_models <= 128. */
LR_API int lr_calibrate(lr_ctx *ctx, int64_t N, const int64_t *features, const int32_t *model, const double *time,
                        int32_t shared_beta1, double *coef_out, void *cuda_stream);

/* Online stream step (Sec. 5: queries arrive over time and are routed as they come;
 * App. F: every instance keeps executing token batches and publishes its state after each).
 * The queries with assign[i] >= 0 join instance assign[i]'s waiting tail in query order
 * (prompt_len[i] prompt tokens, dec[i] output tokens, both in [1, 2^24]); then every
 * instance executes the whole token batches -- the scheduler step the estimator simulates --
 * that end by t_now (seconds), each taking the Eq. 9 time of its own composition, evaluated
 * in fp32 and accumulated into a per-instance fp64 clock (an instance with nothing to run
 * jumps to t_now; no clock ever runs backwards).  Entries of assign outside [0, I), e.g. -1
 * for a query routed elsewhere, are skipped.  The advanced snapshot is then summarized and published as by
 * lr_load_state; clocks start at 0 when a snapshot is loaded.  assign, prompt_len: [Q]
 * device arrays (Q may be 0); dec: [Q][dec_cols] device, dec_cols 1 (one length per query)
 * or num_models (the column of the chosen instance's model is used, e.g. the dec_hat
 * matrix given to lr_route).  Requires cap_running >= every max_seqs (LR_ECAPACITY
 * otherwise).  A waiting queue that would exceed cap_waiting records LR_ECAPACITY, an
 * out-of-range length LR_EINVAL; either leaves the previous snapshot live.
 * With KV-cache limits on (lr_set_kv_limits) every executed batch follows the KV step
 * rule described there (blocks found in running order with preemption of the last running
 * request, admission only with the first chunk's blocks, the context limit ending a
 * request), and the advanced snapshot is summarized and published as a loaded one under
 * those limits.  There a query whose prompt is not below max_ctx, or whose whole context
 * (capped at max_ctx) needs more blocks than the instance has, records LR_EINVAL; a
 * waiting queue that preemptions grow past cap_waiting records LR_ECAPACITY; either keeps
 * the previous snapshot live.  The KV step needs 4 x (11 cap_running + 3 cap_waiting + 32)
 * bytes of shared memory per instance, at most 200 KB for 4 (LR_ECAPACITY otherwise). */
LR_API int lr_advance(lr_ctx *ctx, int32_t Q, const int32_t *assign, const int32_t *prompt_len,
                      const int32_t *dec, int32_t dec_cols, double t_now, void *cuda_stream);

/* Record when tracked queries emit their first output token in the executed stream
 * (Sec. 4.1: the TTFT ends with the first output token; Eq. 4 scores each query by its
 * realized TTFT).  first_token_time: [capacity] fp64 device array owned by the caller,
 * 1 <= capacity < 2^31; NULL turns tracking off.  Queries appended by
 * lr_advance_tracked with ids become tracked; when a tracked request's first output token
 * comes out of a batch that a stream step executes -- its first decode token, or, with
 * LR_FIRST_TOKEN_WITH_LAST_CHUNK, the token of the batch that completes its prompt --
 * first_token_time[id] receives that batch's end time (the instance's fp64 clock after
 * it) and the request stops being tracked.  Entries of ids that have not produced their
 * first token yet are left as they are (e.g. NaN set by the caller).  Requests of a
 * snapshot given to lr_load_state are untracked.  Synchronizes the device and makes every
 * resident request untracked.  An advance whose snapshot is then rejected (LR_ETRAJ) may
 * already have written entries for the batches it executed. */
LR_API int lr_track_first_tokens(lr_ctx *ctx, double *first_token_time, int64_t capacity);

/* lr_advance that tracks the appended queries: query i of this call (if assign[i] is an
 * instance) gets id id_base + i.  id_base >= 0 needs tracking on (LR_EINVAL otherwise) and
 * id_base + Q <= capacity (LR_ECAPACITY); id_base < 0 appends untracked queries, exactly
 * like lr_advance.  Either call records the first tokens of tracked requests already
 * queued. */
LR_API int lr_advance_tracked(lr_ctx *ctx, int32_t Q, const int32_t *assign, const int32_t *prompt_len,
                              const int32_t *dec, int32_t dec_cols, int64_t id_base, double t_now,
                              void *cuda_stream);

/* Copy the live snapshot (as advanced so far) into caller arrays: device pointers with the
 * shapes of lr_state_view plus clock [I] fp64; any pointer may be NULL to skip it. */
LR_API int lr_read_state(const lr_ctx *ctx, int32_t *n_run, int32_t *run_ctx, int32_t *run_pre,
                         int32_t *run_dec, int32_t *n_wait, int32_t *wait_pre, int32_t *wait_dec,
                         double *clock, void *cuda_stream);

/* Synchronize `cuda_stream`, return the first device-side error code recorded since
 * the last call (LR_OK if none) and clear it. */
LR_API int lr_status(lr_ctx *ctx, void *cuda_stream);

/* Static description of a return code. */
LR_API const char *lr_strerror(int code);

/* Text of the last host-side failure on this context (CUDA error string or the
 * validation that failed); empty if none.  Valid until the next call on ctx. */
LR_API const char *lr_last_error(const lr_ctx *ctx);

/* ---- Baseline routing policies and stream metrics (Sec. 6 baselines; Eq. 4) ---- */

enum lr_policy {
    LR_POLICY_ROUND_ROBIN = 0,      /* query i -> instance (rr_start + i) mod I */
    LR_POLICY_SHORTEST_QUEUE = 1,   /* fewest resident requests (running + waiting) */
    LR_POLICY_LATENCY_AGNOSTIC = 2  /* largest utility U (Eq. 2), latency ignored */
};

/* The paper's baseline routers (Sec. 6), for comparison with lr_route.
 * Round Robin assigns cyclically; Shortest Queue lets the Q queries, in order, each
 * join the instance with the fewest resident requests of the live snapshot, counting
 * the queries routed before it in this call (ties: lowest index); Latency-Agnostic
 * picks the largest utility (ties: lowest index), i.e. Eq. 5 with mu = 0.  For each
 * query the chosen instance, its utility U (Eq. 2, cost as in lr_route, one lambda)
 * and its SFS TTFT estimate (the value lr_estimate_ttft gives for that candidate,
 * whatever TTFT source is selected) are written.
 * prompt_len [Q], dec_hat [Q][M], acc [Q][M]: device, as in lr_route.  lambda: host
 * value, finite and >= 0.  rr_start >= 0: Round Robin's first index.
 * assign_out [Q] int32, util_out [Q] fp32, ttft_chosen_out [Q] fp32 or NULL: device.
 * Needs a live snapshot (else the rows are -1 / NaN and the status word records
 * LR_ENOSTATE); a prompt out of range gives that row -1 / NaN (LR_EINVAL recorded).
 * LR_ECAPACITY if the per-CTA sort of the instances' queue counts does not fit in
 * shared memory (about 10,000 instances or more). */
LR_API int lr_route_baseline(lr_ctx *ctx, int32_t policy, int32_t Q, const int32_t *prompt_len,
                             const int32_t *dec_hat, const float *acc, float lambda, int64_t rr_start,
                             int32_t *assign_out, float *util_out, float *ttft_chosen_out, void *cuda_stream);

/* OnTimeUtility (Eq. 4) and SLO attainment over Q >= 1 routed queries.  The
 * realized TTFT of query i is the fp32 sum delay[i] + ttft[i] (delay NULL: 0), e.g.
 * the time the query waited for its routing decision plus the chosen instance's
 * TTFT; it is on time if it is <= tau[i] (NaN never is).
 * out[0] = (1/Q) * sum of util[i] over on-time queries, out[1] = on-time count / Q.
 * util, ttft, tau, delay: [Q] device fp32; out: [2] device fp64.  The sums are fp64
 * in a fixed order (the same result on every run). */
LR_API int lr_on_time_utility(lr_ctx *ctx, int32_t Q, const float *util, const float *ttft, const float *tau,
                              const float *delay, double *out, void *cuda_stream);

#ifdef __cplusplus
}
#endif
#endif /* LATENCY_ROUTER_H */
