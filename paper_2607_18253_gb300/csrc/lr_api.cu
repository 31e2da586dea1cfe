// Host side of the C ABI declared in include/latency_router.h: validation,
// device memory, launch shapes and the status word.
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "latency_router.h"
#include "lr_internal.cuh"

// Chosen-TTFT intermediate of lr_route_frontier_static: [P][Q] fp32 in static
// device memory, so that the call itself allocates nothing.  In host code this
// name is a host-side stand-in, not a device address: lr_create looks the
// device address up (cudaGetSymbolAddress, the context's device current) and
// keeps it in the context.
static __device__ __align__(256) float g_static_route_tch[LR_STATIC_ROUTE_CAP];

struct lr_ctx {
    int device = 0;
    int sms = 0;
    float *static_tch = nullptr;  // device address of g_static_route_tch on this context's device
    double *ftt = nullptr;        // first-token times of tracked queries (caller's array), or none
    int64_t ftt_cap = 0;
    lr::DevConfig cfg{};
    lr::StateBuf buf[2]{};
    lr::StateBuf scratch{};  // advanced snapshot before it is summarized
    lr::DevCtl *ctl = nullptr;
    int max_seqs = 0;
    size_t k3_smem = 0;
    float *scratch_tch = nullptr;
    uint32_t *k2_work = nullptr;  // the candidate kernel's row counters
    double *ontime_part = nullptr;  // per-CTA partial sums of lr_on_time_utility
    bool bl_ok = false;             // the baseline policies' shared memory fits
    // stream of the last snapshot load (lr_load_state or lr_advance): a candidate-kernel
    // call on another stream may run beside it
    void *load_stream = nullptr;
    bool loaded_any = false;
    // average-case TTFT sources
    lr::QueueRaw *qraw = nullptr;
    lr::QueueDev *qd = nullptr;
    unsigned long long *cal_acc = nullptr;  // calibration sums [M][kCalAcc][2] (128-bit) and counter
    int source = lr::kSrcSfs;
    bool have_qp = false, have_lps = false;
    // KV-cache limits (lr_set_kv_limits): per-instance arrays, the records of both
    // buffers, and the load's launch shape
    bool kv_on = false;
    lr::KvLimits kv{};
    int kv_warps = 0;
    size_t kv_smem = 0;
    size_t k3_kv_smem = 0;  // the KV stream step's shared memory (all warps of a CTA)
    int32_t *kv_order = nullptr;  // [max_queries] the estimate's query order
    int32_t *kv_leaders = nullptr, *kv_sort = nullptr;  // [max_queries]; [4][kKvBuckets] + 4 + [2][tiles] + [ceil(I/8)]
    float *kv_mat = nullptr;  // [max_queries][I] the KV estimate matrix a route scores
    std::vector<void *> kv_allocs;
    std::vector<void *> allocs;
    std::string err;
    int max_queries = 0, max_pairs = 0;
    // K1
    size_t k1_smem = 0;
    // candidate kernel shapes: estimate (instances may span several tiles) and
    // route (all instances of a row in one CTA)
    struct Shape {
        int Gp = 0, QS = 0, QT = 0, tiles = 1, occ = 1, block = 0;
        size_t smem = 0;
        bool ok = false;
    } est, rt;
};

namespace {

int fail(lr_ctx *c, int code, const std::string &msg) {
    if (c) c->err = msg;
    return code;
}

int cuda_fail(lr_ctx *c, cudaError_t e, const char *what) {
    if (c) c->err = std::string(what) + ": " + cudaGetErrorString(e);
    return LR_ECUDA;
}

template <typename T>
cudaError_t dev_alloc(lr_ctx *c, T **p, size_t count) {
    void *v = nullptr;
    const size_t bytes = count * sizeof(T) > 0 ? count * sizeof(T) : 16;
    cudaError_t e = cudaMalloc(&v, bytes);
    if (e != cudaSuccess) return e;
    c->allocs.push_back(v);
    e = cudaMemset(v, 0, bytes);
    *p = static_cast<T *>(v);
    return e;
}

int floor_log2(long long x) {
    int s = 0;
    while ((2LL << s) <= x) ++s;
    return s;
}

int round_up(int x, int m) { return ((x + m - 1) / m) * m; }

bool finite_nonneg(float v) { return std::isfinite(v) && v >= 0.0f; }

// Every request of both snapshot buffers untracked (-1), on `stream` (nullptr: the
// legacy stream).
cudaError_t reset_ids(lr_ctx *c, void *stream) {
    const size_t R = (size_t)c->cfg.I * c->cfg.capR, W = (size_t)c->cfg.I * c->cfg.capW;
    cudaError_t e = cudaSuccess;
    for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
        e = cudaMemsetAsync(c->buf[b].run_id, 0xff, R * sizeof(int32_t), (cudaStream_t)stream);
        if (e == cudaSuccess) e = cudaMemsetAsync(c->buf[b].wait_id, 0xff, W * sizeof(int32_t), (cudaStream_t)stream);
    }
    return e;
}

// The live-buffer index and its copies, from the host (no kernel of the context may
// be running); the other control words start at zero.
cudaError_t set_live_host(lr_ctx *c, int32_t v) {
    lr::DevCtl h;
    std::memset(&h, 0, sizeof(h));
    h.active = v;
    for (int r = 0; r < lr::kLiveReps; ++r) h.live[r][0] = v;
    // only the index and its copies change: the status words stay as they are
    cudaError_t e = cudaMemcpy(&c->ctl->active, &h.active, sizeof(int32_t), cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(&c->ctl->live[0][0], &h.live[0][0], sizeof(h.live), cudaMemcpyHostToDevice);
    return e;
}

void free_kv(lr_ctx *c) {
    for (void *p : c->kv_allocs) cudaFree(p);
    c->kv_allocs.clear();
    c->kv = lr::KvLimits{};
    c->kv_on = false;
    c->kv_order = nullptr;
    c->kv_leaders = nullptr;
    c->kv_sort = nullptr;
    c->kv_mat = nullptr;
    for (int b = 0; b < 2; ++b) {
        c->buf[b].kvi = nullptr;
        c->buf[b].kvr = nullptr;
        c->buf[b].kvp = nullptr;
    }
}

void free_all(lr_ctx *c) {
    free_kv(c);
    for (void *p : c->allocs) cudaFree(p);
    c->allocs.clear();
}

int pow2_ceil(int x) {
    int p = 1;
    while (p < x) p *= 2;
    return p;
}

// Launch shape of the candidate kernel: threads own four consecutive instances;
// Gp groups per row (power of two up to 32, else a multiple of 32); the
// summary tables of the tile and QT staged query rows fit the shared-memory
// target.  Routing runs three 256-thread CTAs per SM (one of them fits beside a
// snapshot load's CTA); the estimate alone runs one 768-thread CTA per SM, so
// that each SM copies its tile block once.
lr_ctx::Shape make_shape(const lr::DevConfig &d, bool route, int max_pairs) {
    lr_ctx::Shape s;
    s.block = route ? lr::kK2Block : lr::kK2EstBlock;
    const int G = (d.I + 3) / 4;
    s.Gp = G <= 32 ? pow2_ceil(G) : round_up(G, 32);
    if (s.Gp > lr::kK2Block) {
        if (route) return s;
        s.Gp = lr::kK2Block;
    }
    s.tiles = (d.I + 4 * s.Gp - 1) / (4 * s.Gp);
    s.QS = s.block / s.Gp;
    const int wpr = s.Gp > 32 ? s.Gp / 32 : 1;
    // the tile block (tables and per-instance scalars), brought in by one bulk copy
    lr::DevConfig dt = d;
    dt.tgp = s.Gp;
    const size_t tables = lr::tile_bytes(dt);
    const size_t part = s.Gp > 32 ? 2 * (size_t)wpr * 16 * max_pairs : 0;  // wide-row partials per pair
    // staged row (16 B) and two raw copies of its prompt; routing adds the wide-row
    // partials, (cost, acc) per model, tau, and two raw copies of tau, dec_hat and acc
    const size_t per_row = 16 + 8 + (route ? part + (size_t)d.M * 8 + 4 + 8 + (size_t)d.M * 16 : 0);
    const size_t target = route ? lr::kK2SmemTarget : lr::kK2EstSmemTarget;
    const size_t room = target > tables ? target - tables : 0;
    int qt = (int)std::min<size_t>(route ? 256 : 1024, room / per_row);
    if (route && (size_t)qt * per_row + tables > 200 * 1024) qt = 0;
    qt = std::max(s.QS, (qt / s.QS) * s.QS);
    s.QT = qt;
    s.smem = tables + (size_t)qt * per_row;
    s.ok = s.smem <= 200 * 1024;
    return s;
}

// Row split of a candidate-kernel launch of `ctas` CTAs per tile.  Calls on one
// context are ordered except a snapshot load beside an estimate or route on another
// stream, so a call on the last load's stream runs alone: every CTA takes an equal
// static range.  Otherwise the CTAs that fit beside the load's K1 CTAs (one
// candidate-kernel slot each) start with a static range of 90% of their share, and
// the other rows are claimed as they run out, by the remaining CTAs and by whichever
// finish early, so that every CTA ends on small claimed chunks.
void set_row_split(lr::K2Launch &a, const lr_ctx *c, int ctas, int tiles, int occ, void *stream) {
    if (!c->loaded_any || stream == c->load_stream) {
        a.first_ctas = ctas;
        a.first_rows = std::max(1, (a.Q + ctas - 1) / std::max(1, ctas));
        return;
    }
    const int k1 = (c->cfg.I + lr::kK1Warps - 1) / lr::kK1Warps;
    a.first_ctas = tiles == 1 ? std::max(0, std::min(ctas, c->sms * occ - k1)) : 0;
    const int f = (int)((long long)a.Q * 9 / (10LL * std::max(1, ctas)));
    a.first_rows = std::max(a.QS, f - f % a.QS);
}

lr::K2Launch k2_base(const lr_ctx *c) {
    lr::K2Launch a;
    std::memset(&a, 0, sizeof(a));
    a.cfg = c->cfg;
    a.buf0 = c->buf[0];
    a.buf1 = c->buf[1];
    a.ctl = c->ctl;
    a.src = c->source;
    a.qd = c->qd;
    a.work = c->k2_work;
    return a;
}

}  // namespace

extern "C" {

int lr_create(const lr_config *cfg, lr_ctx **out) {
    if (!cfg || !out) return LR_EINVAL;
    *out = nullptr;
    lr_ctx *c = new (std::nothrow) lr_ctx();
    if (!c) return LR_ENOMEM;
    auto bail = [&](int code, const std::string &msg) {
        std::fprintf(stderr, "lr_create: %s\n", msg.c_str());
        free_all(c);
        delete c;
        return code;
    };
    const int I = cfg->num_instances, M = cfg->num_models;
    if (I < 1 || I > (1 << 16) || M < 1 || M > 1024) return bail(LR_EINVAL, "num_instances or num_models out of range");
    if (!cfg->model_of_instance || !cfg->coef || !cfg->price_in || !cfg->price_out || !cfg->max_batched_tokens ||
        !cfg->max_seqs)
        return bail(LR_EINVAL, "null configuration array");
    if (cfg->cap_running < 1 || cfg->cap_waiting < 1 || cfg->cap_running > 4096 || cfg->cap_waiting > 4096)
        return bail(LR_EINVAL, "cap_running / cap_waiting out of range");
    if (cfg->max_queries < 1 || cfg->max_queries > (1 << 30) || cfg->max_pairs < 1 || cfg->max_pairs > lr::kMaxPairs)
        return bail(LR_EINVAL, "max_queries / max_pairs out of range");
    if (cfg->max_prompt_len < 1 || cfg->max_prompt_len > (1 << 20)) return bail(LR_EINVAL, "max_prompt_len out of range");
    if (cfg->first_token_mode != LR_FIRST_TOKEN_SEPARATE_DECODE && cfg->first_token_mode != LR_FIRST_TOKEN_WITH_LAST_CHUNK)
        return bail(LR_EINVAL, "first_token_mode");
    if (cfg->max_iters < 1) return bail(LR_EINVAL, "max_iters");
    for (int m = 0; m < M; ++m) {
        for (int k = 0; k < 5; ++k)
            if (!finite_nonneg(cfg->coef[m * 5 + k])) return bail(LR_EINVAL, "coefficients must be finite and >= 0");
        if (!finite_nonneg(cfg->price_in[m]) || !finite_nonneg(cfg->price_out[m]))
            return bail(LR_EINVAL, "prices must be finite and >= 0");
    }
    std::vector<int32_t> shift(I), nb(I);
    int kph = 1, nbh = 1;
    for (int j = 0; j < I; ++j) {
        const int B = cfg->max_batched_tokens[j], S = cfg->max_seqs[j], m = cfg->model_of_instance[j];
        if (m < 0 || m >= M) return bail(LR_EINVAL, "model_of_instance out of range");
        if (B < 1 || B > (1 << 24) || S < 1 || S > B) return bail(LR_EINVAL, "need 1 <= max_seqs <= max_batched_tokens <= 2^24");
        const long long gap = (long long)B - S + 1;  // least budget a query gets after admission
        shift[j] = floor_log2(gap);
        nb[j] = (cfg->max_prompt_len >> shift[j]) + 1;
        const long long kp = (cfg->max_prompt_len - 1 + gap - 1) / gap + 1;
        if (kp > lr::kKMax || nb[j] > lr::kNBMax)
            return bail(LR_ECAPACITY, "max_prompt_len too large for max_batched_tokens - max_seqs + 1 of instance " +
                                          std::to_string(j));
        kph = std::max(kph, (int)kp);
        nbh = std::max(nbh, nb[j]);
        c->max_seqs = std::max(c->max_seqs, S);
    }
    cudaError_t e = cudaGetDevice(&c->device);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&c->sms, cudaDevAttrMultiProcessorCount, c->device);
    if (e != cudaSuccess) return bail(LR_ECUDA, std::string("cuda device: ") + cudaGetErrorString(e));
    {
        // the static array of lr_route_frontier_static on this device (the device is
        // current here, and lr_create runs before any capture of the context's calls)
        void *sp = nullptr;
        e = cudaGetSymbolAddress(&sp, g_static_route_tch);
        if (e != cudaSuccess) return bail(LR_ECUDA, std::string("cudaGetSymbolAddress: ") + cudaGetErrorString(e));
        c->static_tch = static_cast<float *>(sp);
    }

    lr::DevConfig &d = c->cfg;
    d.I = I;
    d.M = M;
    d.capR = cfg->cap_running;
    d.capW = cfg->cap_waiting;
    d.pmax = cfg->max_prompt_len;
    d.mode = cfg->first_token_mode;
    d.max_iters = cfg->max_iters;
    d.kph = kph;
    d.nbh = nbh;
    {
        // thread groups per instance tile of the candidate kernel (as make_shape chooses)
        const int G = (I + 3) / 4;
        d.tgp = std::min(G <= 32 ? pow2_ceil(G) : round_up(G, 32), lr::kK2Block);
    }
    c->max_queries = cfg->max_queries;
    c->max_pairs = cfg->max_pairs;

    int32_t *moi, *B, *S, *sh, *nbd;
    float *coef, *pin, *pout;
    const size_t R = (size_t)I * d.capR, W = (size_t)I * d.capW;
#define LR_ALLOC(ptr, n)                                                            \
    do {                                                                            \
        cudaError_t ee = dev_alloc(c, &(ptr), (n));                                 \
        if (ee != cudaSuccess) return bail(LR_ENOMEM, cudaGetErrorString(ee));      \
    } while (0)
    LR_ALLOC(moi, I);
    LR_ALLOC(B, I);
    LR_ALLOC(S, I);
    LR_ALLOC(sh, I);
    LR_ALLOC(nbd, I);
    LR_ALLOC(coef, (size_t)M * 5);
    LR_ALLOC(pin, M);
    LR_ALLOC(pout, M);
    for (int b = 0; b < 2; ++b) {
        lr::StateBuf &s = c->buf[b];
        LR_ALLOC(s.n_run, I);
        LR_ALLOC(s.run_ctx, R);
        LR_ALLOC(s.run_pre, R);
        LR_ALLOC(s.run_dec, R);
        LR_ALLOC(s.n_wait, I);
        LR_ALLOC(s.wait_pre, W);
        LR_ALLOC(s.wait_dec, W);
        LR_ALLOC(s.clock, I);
        LR_ALLOC(s.inst, I);
        LR_ALLOC(s.bkt, (size_t)nbh * I);
        LR_ALLOC(s.tile, (size_t)lr::tile_count(d) * lr::tile_bytes(d));
        LR_ALLOC(s.f2, (size_t)kph * I);
        LR_ALLOC(s.f3, (size_t)kph * I);
        LR_ALLOC(s.rcum, (size_t)kph * I);
        LR_ALLOC(s.run_id, R);
        LR_ALLOC(s.wait_id, W);
    }
    {
        lr::StateBuf &s = c->scratch;
        LR_ALLOC(s.n_run, I);
        LR_ALLOC(s.run_ctx, R);
        LR_ALLOC(s.run_pre, R);
        LR_ALLOC(s.run_dec, R);
        LR_ALLOC(s.n_wait, I);
        LR_ALLOC(s.wait_pre, W);
        LR_ALLOC(s.wait_dec, W);
        LR_ALLOC(s.clock, I);
    }
    LR_ALLOC(c->ctl, 1);
    LR_ALLOC(c->scratch_tch, (size_t)cfg->max_pairs * cfg->max_queries);
    LR_ALLOC(c->k2_work, lr::k2_work_words(I));
    LR_ALLOC(c->ontime_part, 2 * (size_t)lr::kOnTimeParts);
    LR_ALLOC(c->qraw, I);
    LR_ALLOC(c->qd, I);
    LR_ALLOC(c->cal_acc, lr::cal_acc_words(M));
#undef LR_ALLOC
    e = cudaMemcpy(moi, cfg->model_of_instance, I * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(B, cfg->max_batched_tokens, I * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(S, cfg->max_seqs, I * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(sh, shift.data(), I * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(nbd, nb.data(), I * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(coef, cfg->coef, (size_t)M * 20, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(pin, cfg->price_in, M * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(pout, cfg->price_out, M * 4, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = set_live_host(c, -1);
    if (e == cudaSuccess) e = cudaMemset(c->k2_work, 0, sizeof(uint32_t) * lr::k2_work_words(I));
    if (e != cudaSuccess) return bail(LR_ECUDA, cudaGetErrorString(e));
    d.moi = moi;
    d.B = B;
    d.S = S;
    d.shift = sh;
    d.nb = nbd;
    d.coef = coef;
    d.pin = pin;
    d.pout = pout;
    if (I % (4 * d.tgp) != 0) {
        e = lr::launch_tile_pad(d, c->buf[0].tile, 0);
        if (e == cudaSuccess) e = lr::launch_tile_pad(d, c->buf[1].tile, 0);
        if (e == cudaSuccess) e = cudaDeviceSynchronize();
        if (e != cudaSuccess) return bail(LR_ECUDA, cudaGetErrorString(e));
    }

    // K1: one warp per instance.
    c->k1_smem = lr::kK1Warps * lr::trajectory_smem_per_warp(d);
    if (c->k1_smem > 200 * 1024) return bail(LR_ECAPACITY, "snapshot capacities too large for one K1 warp");
    c->est = make_shape(d, false, 1);
    c->rt = make_shape(d, true, cfg->max_pairs);
    if (!c->est.ok) return bail(LR_ECAPACITY, "summary tables too large for shared memory");
    c->k3_smem = lr::kK3Warps * lr::advance_smem_per_warp(d);
    e = lr::set_k1_smem(c->k1_smem);
    if (e == cudaSuccess && c->k3_smem <= 200 * 1024) e = lr::set_k3_smem(c->k3_smem);
    if (e == cudaSuccess && M <= lr::kCalMaxModels) e = lr::set_calib_smem(M);
    if (e == cudaSuccess) e = lr::set_k2_smem(std::max(c->est.smem, c->rt.ok ? c->rt.smem : 0));
    c->bl_ok = lr::baseline_smem(d) <= 200 * 1024;
    if (e == cudaSuccess && c->bl_ok) e = lr::set_baseline_smem(lr::baseline_smem(d));
    if (e == cudaSuccess) e = lr::cand_occupancy(d.mode, false, c->est.block, c->est.smem, &c->est.occ);
    if (e == cudaSuccess && c->rt.ok) e = lr::cand_occupancy(d.mode, true, c->rt.block, c->rt.smem, &c->rt.occ);
    if (e != cudaSuccess) return bail(LR_ECUDA, cudaGetErrorString(e));
    c->est.occ = std::max(1, c->est.occ);
    c->rt.occ = std::max(1, c->rt.occ);
    *out = c;
    return LR_OK;
}

int lr_destroy(lr_ctx *c) {
    if (!c) return LR_OK;
    cudaDeviceSynchronize();
    free_all(c);
    delete c;
    return LR_OK;
}

int lr_load_state(lr_ctx *c, const lr_state_view *v, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (!v || !v->n_run || !v->run_ctx || !v->run_pre || !v->run_dec || !v->n_wait || !v->wait_pre || !v->wait_dec)
        return fail(c, LR_EINVAL, "null snapshot array");
    if (c->kv_on) {
        lr::KvLoad k;
        std::memset(&k, 0, sizeof(k));
        k.cfg = c->cfg;
        k.kv = c->kv;
        k.buf0 = c->buf[0];
        k.buf1 = c->buf[1];
        k.ctl = c->ctl;
        k.in = lr::StateIn{v->n_run, v->run_ctx, v->run_pre, v->run_dec, v->n_wait, v->wait_pre, v->wait_dec, nullptr};
        const int grid = (c->cfg.I + c->kv_warps - 1) / c->kv_warps;
        // a loaded snapshot's requests are untracked (only the stream step assigns ids)
        cudaError_t e = c->ftt ? reset_ids(c, stream) : cudaSuccess;
        if (e != cudaSuccess) return cuda_fail(c, e, "tracking reset");
        e = lr::launch_kv_load(k, grid, c->kv_warps, c->kv_smem, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(c, e, "KV load launch");
        c->load_stream = stream;
        c->loaded_any = true;
        return LR_OK;
    }
    lr::K1Launch a;
    std::memset(&a, 0, sizeof(a));
    a.cfg = c->cfg;
    a.buf0 = c->buf[0];
    a.buf1 = c->buf[1];
    a.ctl = c->ctl;
    a.in = lr::StateIn{v->n_run, v->run_ctx, v->run_pre, v->run_dec, v->n_wait, v->wait_pre, v->wait_dec, nullptr};
    const int grid = (c->cfg.I + lr::kK1Warps - 1) / lr::kK1Warps;
    // a loaded snapshot's requests are untracked (only the stream step assigns ids)
    cudaError_t e = c->ftt ? reset_ids(c, stream) : cudaSuccess;
    if (e != cudaSuccess) return cuda_fail(c, e, "tracking reset");
    e = lr::launch_trajectory(a, grid, lr::kK1Warps * 32, c->k1_smem, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "trajectory launch");
    c->load_stream = stream;
    c->loaded_any = true;
    return LR_OK;
}

static int estimate_common(lr_ctx *c, int32_t Q, const int32_t *p, float *ttft, int32_t *iters, int64_t *feat,
                           void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (Q < 0) return fail(c, LR_EINVAL, "Q < 0");
    if (Q > c->max_queries) return fail(c, LR_ECAPACITY, "Q exceeds max_queries");
    if (Q == 0) return LR_OK;
    if (!p || (!ttft && !feat)) return fail(c, LR_EINVAL, "null array");
    if (iters && c->source != lr::kSrcSfs)
        return fail(c, LR_EINVAL, "first_batch_out exists only for the SFS source");
    if (c->kv_on) {
        lr::KvEst k;
        std::memset(&k, 0, sizeof(k));
        k.cfg = c->cfg;
        k.kv = c->kv;
        k.buf0 = c->buf[0];
        k.buf1 = c->buf[1];
        k.ctl = c->ctl;
        k.Q = Q;
        k.prompt = p;
        k.ttft = ttft;
        k.first_batch = iters;
        k.features = reinterpret_cast<long long *>(feat);
        k.order = c->kv_order;
        k.leaders = c->kv_leaders;
        k.cnt = c->kv_sort;
        k.start = k.cnt + lr::kKvBuckets;
        k.run = k.start + lr::kKvBuckets;
        k.uid = k.run + lr::kKvBuckets;
        k.nu = k.uid + lr::kKvBuckets;
        k.tsum = k.nu + 4;
        k.claim = k.tsum + 2 * lr::kKvScanTiles;
        cudaError_t e = lr::launch_kv_estimate(k, c->sms, (cudaStream_t)stream);
        return e == cudaSuccess ? LR_OK : cuda_fail(c, e, "KV estimate launch");
    }
    lr::K2Launch a = k2_base(c);
    a.Q = Q;
    a.prompt = p;
    cudaError_t e;
    if (feat) {
        a.features = reinterpret_cast<long long *>(feat);
        e = lr::launch_features(a, c->sms, (cudaStream_t)stream);
        return e == cudaSuccess ? LR_OK : cuda_fail(c, e, "features launch");
    }
    a.ttft = ttft;
    a.first_batch = iters;
    a.Gp = c->est.Gp;
    a.QS = c->est.QS;
    a.QT = c->est.QT;
    a.vec_ok = (c->cfg.I % 4 == 0) && ((uintptr_t)ttft % 16 == 0);
    dim3 grid(std::min(c->sms * c->est.occ, (Q + a.QS - 1) / a.QS), c->est.tiles);
    set_row_split(a, c, (int)grid.x, (int)grid.y, c->est.occ, stream);
    e = lr::launch_cand(a, lr::cand_out_flags(true, iters != nullptr, false, false, 1), grid, c->est.block,
                        c->est.smem, (cudaStream_t)stream);
    return e == cudaSuccess ? LR_OK : cuda_fail(c, e, "estimate launch");
}

int lr_estimate_ttft(lr_ctx *c, int32_t Q, const int32_t *prompt_len, float *ttft_out, int32_t *first_batch_out,
                     void *stream) {
    if (c && Q > 0 && !ttft_out) return fail(c, LR_EINVAL, "null ttft_out");
    return estimate_common(c, Q, prompt_len, ttft_out, first_batch_out, nullptr, stream);
}

int lr_estimate_features(lr_ctx *c, int32_t Q, const int32_t *prompt_len, int64_t *features_out, void *stream) {
    if (c && Q > 0 && !features_out) return fail(c, LR_EINVAL, "null features_out");
    return estimate_common(c, Q, prompt_len, nullptr, nullptr, features_out, stream);
}

int lr_route(lr_ctx *c, int32_t Q, const int32_t *prompt_len, const int32_t *dec_hat, const float *acc, const float *tau,
             int32_t P, const float *lambda, const float *mu, int32_t *assign_out, float *util_out,
             float *ttft_chosen_out, double *frontier_out, float *ttft_matrix_out, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (Q < 0) return fail(c, LR_EINVAL, "Q < 0");
    if (Q > c->max_queries) return fail(c, LR_ECAPACITY, "Q exceeds max_queries");
    if (P < 1) return fail(c, LR_EINVAL, "P < 1");
    if (P > c->max_pairs) return fail(c, LR_ECAPACITY, "P exceeds max_pairs");
    if (!c->rt.ok) return fail(c, LR_ECAPACITY, "routing needs num_instances <= 1024 and its tiles in shared memory");
    if (!lambda || (!tau && !mu)) return fail(c, LR_EINVAL, "null lambda / mu");
    if (tau && P != 1) return fail(c, LR_EINVAL, "the constrained objective takes one lambda (P == 1)");
    for (int k = 0; k < P; ++k) {
        if (!finite_nonneg(lambda[k])) return fail(c, LR_EINVAL, "lambda must be finite and >= 0");
        if (!tau && !finite_nonneg(mu[k])) return fail(c, LR_EINVAL, "mu must be finite and >= 0");
    }
    if (Q == 0) return LR_OK;
    if (!prompt_len || !dec_hat || !acc || !assign_out || !util_out) return fail(c, LR_EINVAL, "null array");
    float *kv_matrix = nullptr;
    if (c->kv_on) {
        // KV limits: the estimate matrix first (into the caller's matrix if asked
        // for, else library memory), then utility and argmax over it
        kv_matrix = ttft_matrix_out ? ttft_matrix_out : c->kv_mat;
        const int rc = estimate_common(c, Q, prompt_len, kv_matrix, nullptr, nullptr, stream);
        if (rc != LR_OK) return rc;
    }
    lr::K2Launch a = k2_base(c);
    a.Q = Q;
    a.prompt = prompt_len;
    a.dec_hat = dec_hat;
    a.acc = acc;
    a.tau = tau;
    a.P = P;
    for (int k = 0; k < P; ++k) {
        a.lam[k] = lambda[k];
        a.mu[k] = tau ? 0.0f : mu[k];
    }
    a.assign = assign_out;
    a.util = util_out;
    a.ttft_chosen = ttft_chosen_out ? ttft_chosen_out : (frontier_out ? c->scratch_tch : nullptr);
    a.ttft = kv_matrix ? nullptr : ttft_matrix_out;
    if (kv_matrix) {
        a.src = lr::kSrcMatrix;
        a.ttft_in = kv_matrix;
    }
    a.Gp = c->rt.Gp;
    a.QS = c->rt.QS;
    a.QT = c->rt.QT;
    a.vec_ok = (c->cfg.I % 4 == 0) && ((uintptr_t)a.ttft % 16 == 0);
    dim3 grid(std::min(c->sms * c->rt.occ, (Q + a.QS - 1) / a.QS), 1);
    set_row_split(a, c, (int)grid.x, 1, c->rt.occ, stream);
    cudaError_t e = lr::launch_cand(a, lr::cand_out_flags(a.ttft != nullptr, false, true, tau != nullptr, P), grid,
                                    c->rt.block, c->rt.smem, (cudaStream_t)stream);
    if (e != cudaSuccess) return cuda_fail(c, e, "route launch");
    if (frontier_out) {
        e = lr::launch_frontier(a, frontier_out, (cudaStream_t)stream);
        if (e != cudaSuccess) return cuda_fail(c, e, "frontier launch");
    }
    return LR_OK;
}

int lr_route_baseline(lr_ctx *c, int32_t policy, int32_t Q, const int32_t *prompt_len, const int32_t *dec_hat,
                      const float *acc, float lambda, int64_t rr_start, int32_t *assign_out, float *util_out,
                      float *ttft_chosen_out, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (policy < LR_POLICY_ROUND_ROBIN || policy > LR_POLICY_LATENCY_AGNOSTIC) return fail(c, LR_EINVAL, "policy");
    if (Q < 0) return fail(c, LR_EINVAL, "Q < 0");
    if (Q > c->max_queries) return fail(c, LR_ECAPACITY, "Q exceeds max_queries");
    if (!finite_nonneg(lambda)) return fail(c, LR_EINVAL, "lambda must be finite and >= 0");
    if (rr_start < 0) return fail(c, LR_EINVAL, "rr_start < 0");
    if (!c->bl_ok) return fail(c, LR_ECAPACITY, "num_instances too large for the baseline policies");
    if (Q == 0) return LR_OK;
    if (!prompt_len || !dec_hat || !acc || !assign_out || !util_out) return fail(c, LR_EINVAL, "null array");
    if (c->kv_on && ttft_chosen_out) {
        // the chosen instance's time is read from the KV-limited estimate matrix
        const int rc = estimate_common(c, Q, prompt_len, c->kv_mat, nullptr, nullptr, stream);
        if (rc != LR_OK) return rc;
    }
    lr::K2Launch a = k2_base(c);
    a.Q = Q;
    a.prompt = prompt_len;
    a.dec_hat = dec_hat;
    a.acc = acc;
    a.assign = assign_out;
    a.util = util_out;
    if (c->kv_on) a.ttft_in = c->kv_mat;
    a.ttft_chosen = ttft_chosen_out;
    const cudaError_t e = lr::launch_baseline(a, policy, (long long)rr_start, lambda, c->sms, (cudaStream_t)stream);
    return e == cudaSuccess ? LR_OK : cuda_fail(c, e, "baseline launch");
}

int lr_on_time_utility(lr_ctx *c, int32_t Q, const float *util, const float *ttft, const float *tau,
                       const float *delay, double *out, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (Q < 1) return fail(c, LR_EINVAL, "Q < 1");
    if (!util || !ttft || !tau || !out) return fail(c, LR_EINVAL, "null array");
    const cudaError_t e = lr::launch_on_time(Q, util, ttft, tau, delay, c->ontime_part, lr::kOnTimeParts, out,
                                             (cudaStream_t)stream);
    return e == cudaSuccess ? LR_OK : cuda_fail(c, e, "on-time utility launch");
}

int lr_route_frontier_static(lr_ctx *c, int32_t Q, const int32_t *prompt_len, const int32_t *dec_hat,
                             const float *acc, const float *tau, int32_t P, const float *lambda, const float *mu,
                             int32_t *assign_out, float *util_out, double *frontier_out, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (!frontier_out) return fail(c, LR_EINVAL, "null frontier_out");
    if (Q > 0 && P > 0 && (int64_t)P * Q > LR_STATIC_ROUTE_CAP)
        return fail(c, LR_ECAPACITY, "P * Q exceeds LR_STATIC_ROUTE_CAP (the static chosen-TTFT array)");
    float *tch = c->static_tch;
    if (!tch) return fail(c, LR_ECUDA, "no device address of the static chosen-TTFT array");
    // the same kernels as lr_route with a frontier and no chosen-TTFT output; only
    // the intermediate's storage differs
    return lr_route(c, Q, prompt_len, dec_hat, acc, tau, P, lambda, mu, assign_out, util_out, tch, frontier_out,
                    nullptr, stream);
}

int lr_set_queue_params(lr_ctx *c, const lr_queue_params *qp, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (!qp || !qp->prefill_tput || !qp->decode_batch_time) return fail(c, LR_EINVAL, "null queue parameters");
    const bool lps = qp->arrival_rate != nullptr;
    if (lps && (!qp->service_rate || !qp->parallelism))
        return fail(c, LR_EINVAL, "arrival_rate needs service_rate and parallelism");
    const int I = c->cfg.I;
    std::vector<lr::QueueRaw> raw(I);
    for (int j = 0; j < I; ++j) {
        lr::QueueRaw r;
        std::memset(&r, 0, sizeof(r));
        r.theta = qp->prefill_tput[j];
        r.tdec = qp->decode_batch_time[j];
        if (!(std::isfinite(r.theta) && r.theta > 0.0)) return fail(c, LR_EINVAL, "prefill_tput must be finite and > 0");
        if (!(std::isfinite(r.tdec) && r.tdec >= 0.0))
            return fail(c, LR_EINVAL, "decode_batch_time must be finite and >= 0");
        if (lps) {
            r.alpha = qp->arrival_rate[j];
            r.mu = qp->service_rate[j];
            r.k = qp->parallelism[j];
            r.ca2 = qp->arrival_scv ? qp->arrival_scv[j] : 1.0;
            r.cs2 = qp->service_scv ? qp->service_scv[j] : 1.0;
            r.has_lps = 1;
            if (!(std::isfinite(r.alpha) && r.alpha >= 0.0 && std::isfinite(r.mu) && r.alpha < r.mu))
                return fail(c, LR_EINVAL, "rates must satisfy 0 <= arrival_rate < service_rate (finite)");
            if (r.k < 1 || r.k > (1 << 20)) return fail(c, LR_EINVAL, "parallelism must be in [1, 2^20]");
            if (!(std::isfinite(r.ca2) && r.ca2 >= 0.0 && std::isfinite(r.cs2) && r.cs2 >= 0.0))
                return fail(c, LR_EINVAL, "squared coefficients of variation must be finite and >= 0");
        }
        raw[j] = r;
    }
    cudaStream_t st = (cudaStream_t)stream;
    // pageable source: the copy has read the vector when the call returns
    cudaError_t e = cudaMemcpyAsync(c->qraw, raw.data(), sizeof(lr::QueueRaw) * I, cudaMemcpyHostToDevice, st);
    if (e == cudaSuccess) e = lr::launch_queue_params(I, c->qraw, c->qd, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "queue parameters");
    c->have_qp = true;
    c->have_lps = lps;
    if (c->source == lr::kSrcLps && !lps) c->source = lr::kSrcSfs;
    return LR_OK;
}

int lr_set_ttft_source(lr_ctx *c, int32_t source) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (source != LR_TTFT_SFS && source != LR_TTFT_THROUGHPUT && source != LR_TTFT_LPS)
        return fail(c, LR_EINVAL, "unknown TTFT source");
    if (source != LR_TTFT_SFS && c->kv_on) return fail(c, LR_EINVAL, "KV-cache limits apply to the SFS source only");
    if (source != LR_TTFT_SFS && !c->have_qp) return fail(c, LR_EINVAL, "set the queue parameters first");
    if (source == LR_TTFT_LPS && !c->have_lps) return fail(c, LR_EINVAL, "the LPS source needs arrival and service rates");
    c->source = source;
    return LR_OK;
}

int lr_set_kv_limits(lr_ctx *c, const int32_t *block_size, const int64_t *num_blocks, const int64_t *max_ctx,
                     int32_t horizon) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    const bool on = block_size || num_blocks || max_ctx;
    if (on && !(block_size && num_blocks && max_ctx)) return fail(c, LR_EINVAL, "pass all three arrays or none");
    const int I = c->cfg.I;
    if (on) {
        if (horizon < 1 || horizon > (1 << 16)) return fail(c, LR_EINVAL, "horizon must be in [1, 2^16]");
        if (c->source != lr::kSrcSfs) return fail(c, LR_EINVAL, "KV-cache limits apply to the SFS source only");
        for (int j = 0; j < I; ++j) {
            if (block_size[j] < 1 || block_size[j] > lr::kKvMaxBlock) return fail(c, LR_EINVAL, "block_size out of range");
            if (num_blocks[j] < 1 || num_blocks[j] > (1LL << 40)) return fail(c, LR_EINVAL, "num_blocks out of range");
            if (max_ctx[j] < 2 || max_ctx[j] > (1LL << 40)) return fail(c, LR_EINVAL, "max_ctx out of range");
        }
    }
    int hist = 1;
    for (int j = 0; on && j < I; ++j) hist = std::max(hist, (int)block_size[j]);
    const size_t per_warp = lr::kv_smem_per_warp(c->cfg, hist);
    if (on && per_warp > 200 * 1024) return fail(c, LR_ECAPACITY, "snapshot capacities too large for one KV-load warp");
    cudaError_t e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(c, e, "synchronize");
    free_kv(c);
    // the live snapshot was summarized for the previous rule
    e = set_live_host(c, -1);
    if (e != cudaSuccess) return cuda_fail(c, e, "snapshot reset");
    if (!on) return LR_OK;
    int warps = lr::kKvWarps;
    while (warps > 1 && warps * per_warp > 200 * 1024) --warps;
    e = lr::set_kv_smem(warps * per_warp);
    if (e != cudaSuccess) return cuda_fail(c, e, "KV load shared memory");
    auto alloc = [&](size_t bytes, void **p) {
        cudaError_t ee = cudaMalloc(p, bytes > 0 ? bytes : 16);
        if (ee == cudaSuccess) c->kv_allocs.push_back(*p);
        return ee;
    };
    void *bs = nullptr, *nb = nullptr, *mc = nullptr, *kvi[2] = {nullptr, nullptr}, *kvr[2] = {nullptr, nullptr},
         *kvp[2] = {nullptr, nullptr}, *ord = nullptr, *lead = nullptr, *srt = nullptr, *mat = nullptr;
    e = alloc(sizeof(int32_t) * I, &bs);
    if (e == cudaSuccess) e = alloc(sizeof(int32_t) * (size_t)c->max_queries, &ord);
    if (e == cudaSuccess) e = alloc(sizeof(int32_t) * (size_t)c->max_queries, &lead);
    if (e == cudaSuccess) e = alloc(sizeof(float) * (size_t)c->max_queries * I, &mat);
    const size_t srt_words = 4 * (size_t)lr::kKvBuckets + 4 + 2 * (size_t)lr::kKvScanTiles + (size_t)(I + 7) / 8;
    if (e == cudaSuccess) e = alloc(sizeof(int32_t) * srt_words, &srt);
    if (e == cudaSuccess) e = cudaMemset(srt, 0, sizeof(int32_t) * srt_words);
    if (e == cudaSuccess) e = alloc(sizeof(long long) * I, &nb);
    if (e == cudaSuccess) e = alloc(sizeof(long long) * I, &mc);
    for (int b = 0; b < 2 && e == cudaSuccess; ++b) {
        e = alloc(sizeof(lr::KvInst) * I, &kvi[b]);
        if (e == cudaSuccess) e = alloc(sizeof(lr::KvRec) * (size_t)I * horizon, &kvr[b]);
        if (e == cudaSuccess) e = alloc(sizeof(int32_t) * (size_t)I * horizon, &kvp[b]);
    }
    if (e != cudaSuccess) {
        free_kv(c);
        return fail(c, LR_ENOMEM, cudaGetErrorString(e));
    }
    e = cudaMemcpy(bs, block_size, sizeof(int32_t) * I, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(nb, num_blocks, sizeof(long long) * I, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = cudaMemcpy(mc, max_ctx, sizeof(long long) * I, cudaMemcpyHostToDevice);
    if (e != cudaSuccess) {
        free_kv(c);
        return cuda_fail(c, e, "KV limits upload");
    }
    c->kv.bs = static_cast<const int32_t *>(bs);
    c->kv.nb = static_cast<const long long *>(nb);
    c->kv.mctx = static_cast<const long long *>(mc);
    c->kv.horizon = horizon;
    c->kv.hist = hist;
    c->kv_order = static_cast<int32_t *>(ord);
    c->kv_leaders = static_cast<int32_t *>(lead);
    c->kv_sort = static_cast<int32_t *>(srt);
    c->kv_mat = static_cast<float *>(mat);
    for (int b = 0; b < 2; ++b) {
        c->buf[b].kvi = static_cast<lr::KvInst *>(kvi[b]);
        c->buf[b].kvr = static_cast<lr::KvRec *>(kvr[b]);
        c->buf[b].kvp = static_cast<int32_t *>(kvp[b]);
    }
    c->kv_warps = warps;
    c->kv_smem = warps * per_warp;
    c->k3_kv_smem = lr::kK3Warps * lr::advance_kv_smem_per_warp(c->cfg);
    if (c->k3_kv_smem <= 200 * 1024) {
        e = lr::set_k3_kv_smem(c->k3_kv_smem);
        if (e != cudaSuccess) {
            free_kv(c);
            return cuda_fail(c, e, "KV advance shared memory");
        }
    }
    c->kv_on = true;
    return LR_OK;
}

int lr_calibrate(lr_ctx *c, int64_t N, const int64_t *features, const int32_t *model, const double *time,
                 int32_t shared_beta1, double *coef_out, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (N < 0) return fail(c, LR_EINVAL, "N < 0");
    if (!coef_out || (N > 0 && (!features || !model || !time))) return fail(c, LR_EINVAL, "null array");
    if (c->cfg.M > lr::kCalMaxModels) return fail(c, LR_ECAPACITY, "calibration supports at most 128 models");
    cudaError_t e = lr::launch_calibrate(N, reinterpret_cast<const long long *>(features), model, time, c->cfg.M,
                                         shared_beta1 ? 1 : 0, c->cal_acc, coef_out, c->ctl, c->sms,
                                         (cudaStream_t)stream);
    return e == cudaSuccess ? LR_OK : cuda_fail(c, e, "calibration launch");
}

int lr_advance(lr_ctx *c, int32_t Q, const int32_t *assign, const int32_t *prompt_len, const int32_t *dec,
               int32_t dec_cols, double t_now, void *stream) {
    return lr_advance_tracked(c, Q, assign, prompt_len, dec, dec_cols, -1, t_now, stream);
}

int lr_track_first_tokens(lr_ctx *c, double *first_token_time, int64_t capacity) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (!first_token_time) {
        c->ftt = nullptr;
        c->ftt_cap = 0;
        return LR_OK;
    }
    if (capacity < 1 || capacity > (1LL << 31) - 1) return fail(c, LR_EINVAL, "capacity must be in [1, 2^31 - 1]");
    cudaError_t e = cudaDeviceSynchronize();
    e = e == cudaSuccess ? reset_ids(c, nullptr) : e;
    if (e == cudaSuccess) e = cudaDeviceSynchronize();
    if (e != cudaSuccess) return cuda_fail(c, e, "tracking reset");
    c->ftt = first_token_time;
    c->ftt_cap = capacity;
    return LR_OK;
}

int lr_advance_tracked(lr_ctx *c, int32_t Q, const int32_t *assign, const int32_t *prompt_len, const int32_t *dec,
                       int32_t dec_cols, int64_t id_base, double t_now, void *stream) {
    if (!c) return LR_EINVAL;
    c->err.clear();
    if (id_base >= 0 && !c->ftt) return fail(c, LR_EINVAL, "first-token tracking is off (lr_track_first_tokens)");
    if (id_base >= 0 && (Q > c->ftt_cap || id_base > c->ftt_cap - Q))
        return fail(c, LR_ECAPACITY, "ids id_base .. id_base + Q - 1 exceed the tracking capacity");
    if (Q < 0) return fail(c, LR_EINVAL, "Q < 0");
    if (Q > 0 && (!assign || !prompt_len || !dec)) return fail(c, LR_EINVAL, "null array");
    if (dec_cols != 1 && dec_cols != c->cfg.M) return fail(c, LR_EINVAL, "dec_cols must be 1 or num_models");
    if (!std::isfinite(t_now)) return fail(c, LR_EINVAL, "t_now must be finite");
    if (c->cfg.capR < c->max_seqs) return fail(c, LR_ECAPACITY, "advancing needs cap_running >= every max_seqs");
    if ((c->kv_on ? c->k3_kv_smem : c->k3_smem) > 200 * 1024)
        return fail(c, LR_ECAPACITY, "queue capacities too large for one advance warp");
    lr::K3Launch k;
    std::memset(&k, 0, sizeof(k));
    k.cfg = c->cfg;
    k.buf0 = c->buf[0];
    k.buf1 = c->buf[1];
    k.scratch = c->scratch;
    k.ctl = c->ctl;
    k.Q = Q;
    k.assign = assign;
    k.prompt = prompt_len;
    k.dec = dec;
    k.dec_cols = dec_cols;
    k.t_now = t_now;
    k.track = c->ftt != nullptr;
    k.id_base = id_base;
    k.ftt = c->ftt;
    cudaStream_t st = (cudaStream_t)stream;
    const int k3_grid = (c->cfg.I + lr::kK3Warps - 1) / lr::kK3Warps;
    if (c->kv_on) {
        // the KV step rule, then the KV load summarizes and publishes the snapshot
        k.kv = c->kv;
        cudaError_t e = lr::launch_advance_kv(k, k3_grid, c->k3_kv_smem, st);
        if (e != cudaSuccess) return cuda_fail(c, e, "KV advance launch");
        lr::KvLoad kl;
        std::memset(&kl, 0, sizeof(kl));
        kl.cfg = c->cfg;
        kl.kv = c->kv;
        kl.buf0 = c->buf[0];
        kl.buf1 = c->buf[1];
        kl.ctl = c->ctl;
        const lr::StateBuf &sc = c->scratch;
        kl.in = lr::StateIn{sc.n_run, sc.run_ctx, sc.run_pre, sc.run_dec, sc.n_wait, sc.wait_pre, sc.wait_dec, sc.clock};
        e = lr::launch_kv_load(kl, (c->cfg.I + c->kv_warps - 1) / c->kv_warps, c->kv_warps, c->kv_smem, st);
        if (e != cudaSuccess) return cuda_fail(c, e, "KV load launch");
        c->load_stream = stream;
        c->loaded_any = true;
        return LR_OK;
    }
    cudaError_t e = lr::launch_advance(k, k3_grid, c->k3_smem, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "advance launch");
    // summarize and publish the advanced snapshot exactly as a loaded one
    lr::K1Launch a;
    std::memset(&a, 0, sizeof(a));
    a.cfg = c->cfg;
    a.buf0 = c->buf[0];
    a.buf1 = c->buf[1];
    a.ctl = c->ctl;
    const lr::StateBuf &sc = c->scratch;
    a.in = lr::StateIn{sc.n_run, sc.run_ctx, sc.run_pre, sc.run_dec, sc.n_wait, sc.wait_pre, sc.wait_dec, sc.clock};
    const int grid = (c->cfg.I + lr::kK1Warps - 1) / lr::kK1Warps;
    e = lr::launch_trajectory(a, grid, lr::kK1Warps * 32, c->k1_smem, st);
    if (e != cudaSuccess) return cuda_fail(c, e, "trajectory launch");
    c->load_stream = stream;
    c->loaded_any = true;
    return LR_OK;
}

int lr_read_state(const lr_ctx *c, int32_t *n_run, int32_t *run_ctx, int32_t *run_pre, int32_t *run_dec,
                  int32_t *n_wait, int32_t *wait_pre, int32_t *wait_dec, double *clock, void *stream) {
    if (!c) return LR_EINVAL;
    lr::StateOut o{n_run, run_ctx, run_pre, run_dec, n_wait, wait_pre, wait_dec, clock};
    cudaError_t e = lr::launch_read_state(c->cfg, c->buf[0], c->buf[1], c->ctl, o, (cudaStream_t)stream);
    return e == cudaSuccess ? LR_OK : LR_ECUDA;
}

int lr_status(lr_ctx *c, void *stream) {
    if (!c) return LR_EINVAL;
    int32_t h = 0;
    cudaStream_t st = (cudaStream_t)stream;
    cudaError_t e = cudaMemcpyAsync(&h, &c->ctl->status, sizeof(int32_t), cudaMemcpyDeviceToHost, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e == cudaSuccess) e = cudaMemsetAsync(&c->ctl->status, 0, sizeof(int32_t), st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(c, e, "status");
    return h;
}

const char *lr_strerror(int code) {
    switch (code) {
        case LR_OK: return "ok";
        case LR_EINVAL: return "invalid argument or input value";
        case LR_ENOMEM: return "out of memory";
        case LR_ECUDA: return "CUDA runtime error";
        case LR_ECAPACITY: return "size exceeds the context's capacity";
        case LR_ETRAJ: return "simulated trajectory exceeded max_iters";
        case LR_ESTATE: return "snapshot violates the state preconditions";
        case LR_ENOSTATE: return "no snapshot loaded";
        default: return "unknown error";
    }
}

const char *lr_last_error(const lr_ctx *c) { return c ? c->err.c_str() : ""; }

}  // extern "C"
