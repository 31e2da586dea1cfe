// Library-internal layout shared by the host API and the kernels.
//
// Data layout in HBM (all per-instance tables are [row][I], instance-minor, so
// that consecutive threads of a CTA -- which own consecutive instances -- read
// consecutive words):
//
//   config      : model_of_instance[I], B[I], S[I], shift[I], nb[I], coef[M][5],
//                 price_in[M], price_out[M]
//   buffer 0/1  : a snapshot copy (SoA, row stride cap) plus its summary:
//                 inst[I]           InstParams (admission batch, totals, splits)
//                 bkt[NBH][I]       int2 (in-bucket boundary, boundaries below)
//                 f2[KPH][I], f3[KPH][I], rcum[KPH][I]
//                 tile[T]           per tile of 4*tgp instances, the candidate
//                                   kernel's shared-memory image (see below)
//   control     : live buffer index, sticky status word, load error, CTA counter
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace lr {

constexpr int kKMax = 64;               // table entries per instance (k = 0..kp-1)
constexpr int kNBMax = 2 * kKMax + 2;   // prompt-length buckets per instance
constexpr int kBig = 0x7fffffff;        // "never" / "no boundary"
constexpr int kSplitBits = 20;          // low part of the exact fp32 splits
constexpr long long kFastLimit = 1LL << 44;  // integers below this split exactly
constexpr int kMaxPairs = 64;

// Return codes (mirror include/latency_router.h).
enum : int { kOk = 0, kEInval = 1, kENoMem = 2, kECuda = 3, kECapacity = 4, kETraj = 5, kEState = 6,
             kENoState = 7 };

struct InstParams {      // 64 bytes
    int32_t la;          // batch at which a query appended now is admitted
    int32_t kp;          // number of table entries
    int32_t shift;       // log2 of the bucket width
    int32_t fast;        // 1: every feature of this instance splits exactly into fp32
    long long f1tot;     // prefill tokens of all residents
    long long f4tot;     // prefill attention pairs of all residents
    float h1, l1, h4, l4;  // exact fp32 high/low parts of f1tot and f4tot
    int32_t r0;          // budget left to the query in its admission batch
    int32_t pad[3];
};

struct DevConfig {
    int32_t I, M, capR, capW;
    int32_t pmax, mode, max_iters, tgp;     // tgp: thread groups per instance tile of the candidate kernel
    int32_t kph, nbh;                       // table row counts (host bounds over instances)
    const int32_t *moi, *B, *S, *shift, *nb;
    const float *coef, *pin, *pout;
};

// KV-limited simulation (App. F): one batch of an instance's residents alone, from
// the first batch in which a query could be admitted (the waiting queue empty after
// admissions, budget and a seat left).  64 bytes.
struct __align__(16) KvRec {
    long long cf[4];   // residents' features 1..4 summed from the first record through this one
    long long slack;   // least (free blocks - blocks needed) over the running scan; < 0: a preemption
    long long far;     // free blocks after the running scan
    long long thr;     // a waiting query with prompt p is admitted in this batch iff p <= thr
    int32_t bar, bl;   // budget left after the running scan, after admissions
};
// Per instance: the residents' features before the first record, and the records' extent.
struct __align__(16) KvInst {
    long long fcum[5];
    int32_t la0;   // batch of record 0
    int32_t nrec;  // records written
    int32_t done;  // 1: no resident is left after the last record (later batches are empty)
    int32_t pad;
};
struct KvLimits {
    const int32_t *bs;     // [I] block size (tokens), at most kKvMaxBlock
    const long long *nb;   // [I] blocks
    const long long *mctx; // [I] context limit
    int32_t horizon;       // records per instance
    int32_t hist;          // the largest block size: entries of the load's residue histogram
};
constexpr int kKvMaxBlock = 4096;
constexpr int kKvCal = 1024;  // batches covered by the load's end calendar

struct StateBuf {
    int32_t *n_run, *run_ctx, *run_pre, *run_dec, *n_wait, *wait_pre, *wait_dec;
    double *clock;  // [I] end time of the instance's last completed batch (s)
    InstParams *inst;
    int2 *bkt;
    unsigned char *tile;  // candidate-kernel tile blocks
    long long *f2, *f3;
    int32_t *rcum;
    KvInst *kvi;   // [I], with KV limits
    KvRec *kvr;    // [I][horizon], with KV limits
    int32_t *kvp;  // [I][horizon] running maximum of the records' thr (clamped to int32), with KV limits
    // first-token tracking (lr_track_first_tokens): each request's id until its first output
    // token, else -1; written by the stream step only (a snapshot load makes every request -1)
    int32_t *run_id, *wait_id;  // [I][capR], [I][capW]
};

// Copies of the live-buffer index, each in its own 128-byte line: the CTAs of a
// candidate-kernel launch (hundreds, all starting at once) read different copies
// instead of queueing on one line.
constexpr int kLiveReps = 64;
struct __align__(128) DevCtl {
    int32_t active;      // live buffer, -1 before the first successful load
    int32_t status;      // first error since the last lr_status
    int32_t load_err;    // error of the load in progress
    uint32_t done_ctas;  // K1 completion counter
    int32_t pad[28];
    int32_t live[kLiveReps][32];  // live[r][0]: copies of active
};

struct StateIn {
    const int32_t *n_run, *run_ctx, *run_pre, *run_dec, *n_wait, *wait_pre, *wait_dec;
    const double *clock;  // may be null: clocks start at 0
};

// The live-buffer index with acquire ordering: reads of the buffer it names see
// everything the load that published it wrote (it may have finished on another stream).
__device__ __forceinline__ int32_t load_acquire(const int32_t *p) {
    int32_t v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Publish a new live buffer (after a __threadfence of the writes that made it): the
// index and its copies, which readers take with acquire loads.
__device__ __forceinline__ void publish_live(DevCtl *ctl, int32_t v) {
    atomicExch(&ctl->active, v);
    for (int r = 0; r < kLiveReps; ++r)
        asm volatile("st.relaxed.gpu.global.b32 [%0], %1;" ::"l"(&ctl->live[r][0]), "r"(v) : "memory");
}

// The live-buffer index from this CTA's copy, with acquire ordering.
__device__ __forceinline__ int32_t load_live(const DevCtl *ctl) {
    return load_acquire(&ctl->live[blockIdx.x % kLiveReps][0]);
}

__device__ __forceinline__ void record_status(DevCtl *ctl, int code) {
    atomicCAS(&ctl->status, 0, code);
}

__device__ __forceinline__ unsigned lanemask_lt() {
    unsigned m;
    asm volatile("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

__device__ __forceinline__ long long warp_sum64(long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Candidate-kernel tile block: everything one CTA of the candidate kernel needs about
// its tile of 4 * tgp instances, laid out as that CTA's shared memory so that a single
// bulk copy brings it in.  Instance j0 + 4g + u of the tile sits in column u * tgp + g:
//   entA [kph][4][tgp]    8 bytes: T_k (fp32) and X_k, which is f3_k (fp32) when the
//                         first token comes with the last chunk, else F3_k as an int32
//                         (valid when the instance is compact: F3_k + pmax < 2^31)
//   entB [kph][4][tgp]    8 bytes: H3_k, L3_k, the exact fp32 split of F3_k
//   bkt  [nbh][tgp][4]    uint32: (in-bucket boundary << 7) | boundaries below, the
//                         boundary 2^24 - 1 when the bucket holds none; a thread's four
//                         instances are adjacent (one 16-byte load when they share the
//                         bucket width)
//   scal [kScal][4][tgp]  32-bit scalars, fields kSc*
// A warp reads a table as one dense 4- or 8-byte word per lane (1 or 2 shared-memory
// wavefronts); a compact CTA reads only entA.
constexpr int kScal = 12;
enum : int { kScShift = 0, kScH1, kScL1, kScH4, kScL4, kScB1p, kScB2, kScB3, kScModel, kScLa, kScFast, kScCompact };
constexpr uint32_t kBktNone = (1u << 24) - 1;  // bucket boundary field of a bucket without one
__host__ __device__ inline size_t tile_enta_bytes(const DevConfig &c) { return (size_t)c.kph * 4 * c.tgp * 8; }
__host__ __device__ inline size_t tile_ent_bytes(const DevConfig &c) { return 2 * tile_enta_bytes(c); }
__host__ __device__ inline size_t tile_bkt_bytes(const DevConfig &c) {
    return ((size_t)c.nbh * 4 * c.tgp * 4 + 15) & ~(size_t)15;
}
__host__ __device__ inline size_t tile_bytes(const DevConfig &c) {
    return tile_ent_bytes(c) + tile_bkt_bytes(c) + (size_t)kScal * 4 * c.tgp * 4;
}
__host__ __device__ inline int tile_count(const DevConfig &c) { return (c.I + 4 * c.tgp - 1) / (4 * c.tgp); }
// Byte offset of instance j's column within its tile block, and the tile's base.
__host__ __device__ inline size_t tile_base(const DevConfig &c, int j) { return (size_t)(j / (4 * c.tgp)) * tile_bytes(c); }
__host__ __device__ inline int tile_col(const DevConfig &c, int j) {
    const int jj = j % (4 * c.tgp);
    return (jj & 3) * c.tgp + (jj >> 2);
}
// Columns past the last instance, written once so that they read as empty instances.
cudaError_t launch_tile_pad(const DevConfig &c, unsigned char *tile, cudaStream_t st);

// Calibration of the batch-time coefficients (lr_calibrate.cu).
constexpr int kCalCols = 5;
constexpr int kCalAcc = 21;        // per model: 15 sums of the upper triangle of G, 5 of b, the row count
constexpr int kCalMaxModels = 128;  // shared-memory sums of one CTA (128-bit each)
constexpr double kCalTimeScale = 17592186044416.0;  // 2^44: times in 2^-44 s fixed point
constexpr double kCalTimeMax = 524288.0;            // 2^19 s
constexpr int kCalThreads = 512;                    // one CTA per SM
constexpr int kCalConsumerWarps = kCalThreads / 32 - 1;  // the last warp issues the copies
constexpr int kCalTile = 2 * 32 * kCalConsumerWarps;     // rows per staged tile, two a consumer lane (16-byte copies)
constexpr int kCalStagesMax = 3;                    // tiles in flight per CTA
constexpr int kCalFlushRows = 128;                  // rows a lane sums in 64 bits between flushes
constexpr size_t kCalSmemMax = 227 * 1024;
constexpr size_t kCalStageBytes = (size_t)kCalTile * (kCalCols * 8 + 8 + 4);
constexpr int kCalFlushSums = 26;  // a warp flush's sums: 15 of G, 5 + 5 halves of b, the row count
// the CTA's shared sums: 128-bit [M][kCalAcc] and the flushes' carry-save words [M][kCalFlushSums]
__host__ __device__ inline size_t cal_sums_bytes(int M) { return (size_t)M * (kCalAcc + kCalFlushSums) * 16; }
// the calibration's device words: the sums [M][kCalAcc][2] and the CTA counter of the
// last-CTA solve (zero between calls)
__host__ __device__ inline size_t cal_acc_words(int M) { return (size_t)M * kCalAcc * 2 + 2; }
cudaError_t launch_calibrate(long long N, const long long *F, const int32_t *model, const double *time, int M,
                             int shared_beta1, unsigned long long *acc, double *coef, DevCtl *ctl, int grid,
                             cudaStream_t st);
cudaError_t set_calib_smem(int M);

// Launch helpers implemented in the kernel translation units.
struct K1Launch {
    DevConfig cfg;
    StateBuf buf0, buf1;
    DevCtl *ctl;
    StateIn in;
};
cudaError_t launch_trajectory(const K1Launch &a, int grid, int block, size_t smem, cudaStream_t st);
cudaError_t set_k1_smem(size_t bytes);
constexpr int kK1Warps = 4;

// KV-limited load (residents alone, records) and estimate (per-candidate walk).
struct KvLoad {
    DevConfig cfg;
    KvLimits kv;
    StateBuf buf0, buf1;
    DevCtl *ctl;
    StateIn in;
};
constexpr int kKvWarps = 4;
// shared memory per warp of the KV load: the running list (context, prefill, decode,
// blocks) and the waiting ring (prefill, decode) over capR + capW requests, the end
// calendar (links and blocks at the end per request, kKvCal heads) and the residue
// histogram, 16-byte aligned
__host__ __device__ inline size_t kv_smem_per_warp(const DevConfig &c, int hist) {
    return (sizeof(int32_t) * (8 * (size_t)(c.capR + c.capW) + kKvCal + hist + 16) + 15) & ~(size_t)15;
}
// warps: instances per CTA, 1 .. kKvWarps
cudaError_t launch_kv_load(const KvLoad &a, int grid, int warps, size_t smem, cudaStream_t st);
cudaError_t set_kv_smem(size_t bytes);
struct KvEst {
    DevConfig cfg;
    KvLimits kv;
    StateBuf buf0, buf1;
    DevCtl *ctl;
    int32_t Q;
    const int32_t *prompt;
    float *ttft;
    int32_t *first_batch;
    long long *features;
    // the call's queries sorted by prompt length (counting sort over kKvBuckets
    // buckets: invalid lengths, then valid ones >> shift); with shift 0 one
    // query per length is estimated and the others copy its rows
    int32_t *cnt, *start, *run, *uid;  // [kKvBuckets]
    int32_t *nu;                       // [1] distinct lengths
    int32_t *tsum;                     // [2][kKvScanTiles] per-tile bucket sums of the scan
    int32_t *order, *leaders;          // [max_queries]
    int32_t *claim;                    // [ceil(I / 8)] the estimate's block counters per instance group
};
constexpr int kKvBuckets = 1 << 16;
constexpr int kKvScanTiles = kKvBuckets / 4096;  // the bucket scan's tiles, one CTA each
cudaError_t launch_kv_estimate(const KvEst &a, int sms, cudaStream_t st);

// Batches covered by K1's completion calendar; decoders ending later are
// tracked by scanning the decoder list.
constexpr int kCalendar = 2048;

// Shared memory of one K1 warp (in int32 words, a multiple of 4): calendar and
// its bitmap, the decoder list (first batch, last batch, context offset, pad),
// the waiting queue's prompt prefix sums and decode lengths, and the budgets.
__host__ __device__ inline size_t trajectory_smem_per_warp(const DevConfig &c) {
    const size_t words = (size_t)kCalendar + kCalendar / 32 + 4 * (size_t)(c.capR + c.capW) +
                         (size_t)(c.capW + 2) + (size_t)(c.capW + 1) + (size_t)c.kph + 32;
    return sizeof(int32_t) * ((words + 3) & ~(size_t)3);
}

// Average-case TTFT sources (Sec. 4, App. E): per-instance parameters as given
// and the derived constants of t = fma(p, g, C).
// kSrcMatrix (internal): the times come from a [Q][I] matrix already computed (the
// KV-limited estimate), read by the candidate kernel's affine mode
enum : int { kSrcSfs = 0, kSrcThroughput = 1, kSrcLps = 2, kSrcMatrix = 3 };
struct QueueRaw {      // 64 bytes, copied from the caller's arrays
    double theta, tdec, alpha, mu, ca2, cs2;
    int32_t k, has_lps;
    int32_t pad[2];
};
struct QueueDev {      // 32 bytes
    double theta, tdec;
    double wlps;       // LPS expected wait (NaN without queue rates)
    float g;           // fp32(1 / theta)
    float clps;        // fp32(wlps + tdec)
};
cudaError_t launch_queue_params(int I, const QueueRaw *raw, QueueDev *qd, cudaStream_t st);

struct K2Launch {
    DevConfig cfg;
    StateBuf buf0, buf1;
    DevCtl *ctl;
    int32_t Q;
    const int32_t *prompt;
    // estimate outputs
    float *ttft;
    int32_t *first_batch;
    long long *features;
    // route inputs / outputs
    const int32_t *dec_hat;
    const float *acc;
    const float *tau;
    int32_t P;
    float lam[kMaxPairs];
    float mu[kMaxPairs];
    int32_t *assign;
    float *util;
    float *ttft_chosen;
    // launch shape: Gp thread groups of four instances per row (a power of two up
    // to 32, else a multiple of 32), QS rows in flight, QT rows per staged chunk
    int32_t Gp, QS, QT, vec_ok;
    // TTFT source (kSrc*) and, for the average-case ones, the instance constants
    int32_t src;
    const QueueDev *qd;
    const float *ttft_in;  // kSrcMatrix: [Q][I]
    // [0]: CTAs finished; [1 + tile]: query rows of the tile claimed past the static
    // ones.  Zero before a launch; the last CTA to finish clears them for the next.
    uint32_t *work;
    // CTAs (per tile) that start with a static chunk of first_rows query rows
    int32_t first_ctas, first_rows;
};
// Entries of the candidate kernel's work counters for I instances.
inline int k2_work_words(int I) { return (I + 1023) / 1024 + 2; }
int cand_out_flags(bool matrix, bool iters, bool route, bool constrained, int P);
cudaError_t launch_cand(const K2Launch &a, int out, dim3 grid, int block, size_t smem, cudaStream_t st);
cudaError_t launch_features(const K2Launch &a, int sms, cudaStream_t st);
cudaError_t launch_frontier(const K2Launch &a, double *out, cudaStream_t st);
// Baseline routing policies (0 Round Robin, 1 Shortest Queue, 2 Latency-Agnostic) and
// the stream metrics (OnTimeUtility, SLO attainment) over routed queries.
size_t baseline_smem(const DevConfig &c);
cudaError_t set_baseline_smem(size_t bytes);
cudaError_t launch_baseline(const K2Launch &a, int policy, long long rr_start, float lam, int sms, cudaStream_t st);
constexpr int kOnTimeParts = 1024;
cudaError_t launch_on_time(int Q, const float *util, const float *ttft, const float *tau, const float *delay,
                           double *part, int max_parts, double *out, cudaStream_t st);
cudaError_t cand_occupancy(int mode, bool route, int block, size_t smem, int *blocks_per_sm);
cudaError_t set_k2_smem(size_t bytes);
constexpr int kK2Block = 256;                // route: three CTAs per SM, one fits beside a load's CTA
constexpr size_t kK2SmemTarget = 72 * 1024;  // three CTAs per SM
constexpr int kK2EstBlock = 768;             // estimate alone: one CTA per SM, one tile copy per SM
constexpr size_t kK2EstSmemTarget = 120 * 1024;

// K3: append routed queries and advance every instance to t_now (online stream).
struct K3Launch {
    DevConfig cfg;
    StateBuf buf0, buf1;  // the live one is read
    StateBuf scratch;     // receives the advanced snapshot (then summarized by K1)
    DevCtl *ctl;
    int32_t Q;
    int32_t dec_cols;  // 1: dec[i]; M: dec[i][model of the chosen instance]
    const int32_t *assign, *prompt, *dec;
    double t_now;
    // first-token tracking: the appended query i gets id id_base + i (id_base < 0: -1);
    // ftt[id] receives the end time of the batch with its first output token
    int32_t track;
    long long id_base;
    double *ftt;
    KvLimits kv;  // the KV stream step (launch_advance_kv) only
};
constexpr int kK3Warps = 4;
// Shared memory of one K3 warp: the running list twice (ctx, pre, dec, id; the
// batch's survivors are compacted into the other copy) and the waiting queue (pre,
// dec, id).
__host__ __device__ inline size_t advance_smem_per_warp(const DevConfig &c) {
    return sizeof(int32_t) * ((size_t)8 * c.capR + (size_t)3 * c.capW + 32);
}
// The KV stream step's waiting queue is a ring of capW + capR entries: preempted
// requests return to its front.
__host__ __device__ inline size_t advance_kv_smem_per_warp(const DevConfig &c) {
    return sizeof(int32_t) * ((size_t)8 * c.capR + (size_t)3 * ((size_t)c.capW + c.capR) + 32);
}
cudaError_t launch_advance(const K3Launch &a, int grid, size_t smem, cudaStream_t st);
cudaError_t launch_advance_kv(const K3Launch &a, int grid, size_t smem, cudaStream_t st);
cudaError_t set_k3_kv_smem(size_t bytes);
cudaError_t set_k3_smem(size_t bytes);
struct StateOut {
    int32_t *n_run, *run_ctx, *run_pre, *run_dec, *n_wait, *wait_pre, *wait_dec;
    double *clock;
};
cudaError_t launch_read_state(const DevConfig &c, const StateBuf &b0, const StateBuf &b1, DevCtl *ctl,
                              const StateOut &o, cudaStream_t st);

}  // namespace lr
