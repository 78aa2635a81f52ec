// C-ABI host code of the route-scoring library (declarations in include/hwr.h).
//
// Owns the context: device copies of the deployment table, the predictor
// (fp32 copies for the SIMT kernels, bf16 shared-memory images for the
// tcgen05 kernels), the model embeddings and the hardware snapshot; grow-only
// scratch and I/O staging; and the dispatch of each call onto the kernels of
// k_simt.cu and k_tc.cu on the context stream.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <chrono>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "hwr_internal.cuh"

using namespace hwr;

namespace {

thread_local std::string g_create_error;

// An NVTX range over one API call: a profiler that records NVTX (Nsight
// Systems, for one) shows each call on the calling thread's timeline; with
// none attached a push / pop costs a few nanoseconds.
struct ApiRange {
    explicit ApiRange(const char *name) { nvtxRangePushA(name); }
    ~ApiRange() { nvtxRangePop(); }
    ApiRange(const ApiRange &) = delete;
    ApiRange &operator=(const ApiRange &) = delete;
};

// Host-side fault hooks for tests, read at hwr_create: HWR_TEST_FAIL_ALLOC=n
// makes the n-th allocation of the context (counting from 1) report failure;
// HWR_TEST_STALL=1 makes the tensor-path producers never signal their tiles,
// so the predictor kernel's bounded waits run out (HWR_ERR_TIMEOUT).
struct AllocHook {
    long fail_at = 0, count = 0;
};

// Path thresholds, from sweeps of batch sizes on GB300 (defaults;
// HWR_TC_MIN_PAIRS and HWR_PAIRS_MAX_PAIRS override them at hwr_create):
// batches of at most pairs_max pairs (Q * D) take the small-batch SIMT
// kernel; larger bf16 batches of at least tc_min_pairs pairs take the
// tensor-core kernels; the rest the fused SIMT kernel.  pairs_max is
// SMALL_MAX_PAIRS where the tensor-core path exists; otherwise FP32_MAX_PAIRS
// for hidden layers wider than 64 x 64 and 0 for narrower ones.
// (Device pointers, isolated calls.  bf16, H = 256: the tensor path costs
// 32-33.5 us at D = 32 for 16-64 queries and 36-37 us at D = 64 for 8-32; the
// small-batch kernel 29.7 / 30.5 / 34.3 / 44 us at D = 32 for 1 / 16 / 32 /
// 64 queries and 29.5 / 31.1 / 34.8 / 44.6 us at D = 64 for 1 / 8 / 16 / 32:
// ahead up to about 768 pairs.  fp32: the fused kernel
// costs ~21 us at H = 32 and ~33 us at H = 128 from 1 to 512 queries; the
// small-batch kernel costs ~24 us at H = 32 whatever the size, and 25.5-29 us
// at H = 128, D = 12 from 1 to 170 queries (2,040 pairs).)
constexpr int TC_MIN_PAIRS = 257;
constexpr int PIPE_CHUNK_MIN = 8192;   // smallest chunk of a pipelined host batch
constexpr int SMALL_MAX_PAIRS = 768;
constexpr int FP32_MAX_PAIRS = PAIRS_MAX_PAIRS;

}  // namespace

struct hwr_ctx {
    int M = 0, G = 0, D = 0, F = 0, H1 = 0, H2 = 0, E = 0, P = 0, NH = 2;
    int Mpad = 0, Epad = 0;
    hwr_dtype dtype = HWR_F32;
    bool tc_ok = false;
    cudaStream_t stream = nullptr;
    bool own_stream = false;
    bool broken = false;
    bool have_snapshot = false;
    int test_stall = 0;          // HWR_TEST_STALL: tensor-path producers never signal
    int tc_min_pairs = TC_MIN_PAIRS, pairs_max = -1;   // -1: by the context's paths
    int device = -1;             // the CUDA device current at hwr_create
    long poll_us = 1000000;      // small-batch output poll limit (HWR_TEST_POLL_US)
    bool async_pending = false;  // an HWR_ASYNC call may still have work queued
    // the GPU reads and writes pageable host memory coherently (address
    // translation services over the CPU-GPU link, as on Grace + GB300):
    // small synchronous calls then use the caller's arrays directly
    bool ats = false;
    std::vector<uint8_t> xform_h;   // feature transforms (host copy, snapshot checks)
    std::string err;
    AllocHook hook;
    std::vector<void *> allocs;  // device buffers (cudaMalloc)

    // device state
    int32_t *dep_model = nullptr, *dep_gpu = nullptr;
    float *log10p = nullptr;
    float *W1 = nullptr, *b1 = nullptr, *W2 = nullptr, *b2 = nullptr;
    float *W3 = nullptr, *b3 = nullptr, *mu = nullptr, *sd = nullptr;
    uint8_t *xform = nullptr;
    float *memb = nullptr;
    float *W1q = nullptr;            // [2][H1]
    float *W2T = nullptr;            // [H1][H2p] fp32 (rows zero-padded), for the SIMT tiles
    float *W1T = nullptr;            // [F][H1] fp32, W1 slot-major
    uint16_t *W2img = nullptr, *membimg = nullptr;
    std::vector<char> head_consts;   // output-layer constants for the tensor path
    int32_t *running = nullptr, *waiting = nullptr;
    float *kv = nullptr, *gpu_util = nullptr, *ttft = nullptr, *tpot = nullptr;
    float *X = nullptr, *Spre = nullptr, *A = nullptr;
    uint16_t *Abf = nullptr;
    // host feature constants for the tensor path
    float mu_in = 0, sd_in = 1, mu_out = 0, sd_out = 1;
    uint8_t xf_in = 0, xf_out = 0;

    // mapped pinned status word written by kernels with bounded waits
    int32_t *status_h = nullptr, *status_d = nullptr;

    // snapshot staging (pinned) and its copy-done event
    void *snap_h = nullptr;
    const uint32_t *snap_hd = nullptr;   // device address of the mapped snap_h
    void *snap_d = nullptr;
    cudaEvent_t snap_ev = nullptr;
    // completion counter of the tensor-core predictor kernels (device): every
    // CTA adds one as it finishes; host side, the CTAs launched in all and by
    // the most recent predictor launch
    uint32_t *done_d = nullptr;
    uint32_t pred_ctas = 0, pred_ctas_last = 0;
    // outputs of the last tensor-core route (its predictor may still run
    // while the next route's kernels start)
    struct Range {
        const void *p = nullptr;
        size_t n = 0;
    } prev_out[4];                   // chosen, latency, utility, per-pair costs
    // a snapshot kernel may still read the staging: set at its launch, cleared
    // once the host has seen later work on the stream complete
    bool snap_busy = false;

    // grow-only scratch
    float *qual = nullptr;   size_t qual_cap = 0;     // 2 x [Q][Mpad], alternating per call
    float *qual_last = nullptr;                       // the buffer the last quality kernel wrote
    int qual_flip = 0;
    char *part = nullptr;    size_t part_cap = 0;     // split-deployment partials
    int32_t *count = nullptr; size_t count_cap = 0;   // per-row arrivals (self-resetting)
    float *pairC = nullptr;  float *pairQ = nullptr;  int32_t *pairN = nullptr;  // small batches
    float *pairH = nullptr;
    float *mC = nullptr;     size_t mC_cap = 0;       // multi-lambda: pair costs [Q][D]
    float *mQ = nullptr;     size_t mQ_cap = 0;       // multi-lambda: quality [Q][M]
    float *ctab = nullptr;   size_t ctab_cap = 0;
    float *qseq = nullptr;   size_t qseq_cap = 0;
    int seq_qs = 0;
    // sequential mode with the table on the tensor cores: bf16 prefixes
    // [D (Qs+1)][H1], model of each (deployment, count) group
    uint16_t *prebf = nullptr; size_t prebf_cap = 0;
    int32_t *dmv = nullptr;  size_t dmv_cap = 0;
    int seq_slots = 0;       // sequential-table blocks resident at once
    int nsm = 1;             // SMs of the context's device

    // I/O staging for host pointers: device [emb | in | out] and [chosen | lat | util]
    char *io_d = nullptr;    size_t io_cap = 0;
    char *out_d = nullptr;   size_t out_cap = 0;
    char *pin_h = nullptr;   size_t pin_cap = 0;       // pinned, mapped host staging
    char *pin_d = nullptr;                            // its device address
    cudaEvent_t pin_ev = nullptr;
    // large host-pointer batches: chunked copies on a second stream overlap
    // the kernels of the previous chunk
    cudaStream_t copy_stream = nullptr;
    cudaEvent_t chunk_ev[8] = {};
    cudaEvent_t io_free_ev = nullptr;   // earlier work on the context stream is done

    // profiling
    struct Pending { int k; cudaEvent_t a, b; };
    std::vector<Pending> pending;
    std::vector<cudaEvent_t> ev_pool;
    hwr_stats stats;
};

// ---------------------------------------------------------------------------
// helpers

static hwr_status fail(hwr_ctx *c, hwr_status s, const char *fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (c) {
        c->err = buf;
        if (s == HWR_ERR_CUDA || s == HWR_ERR_TIMEOUT) c->broken = true;
    } else {
        g_create_error = buf;
    }
    return s;
}

static hwr_status cuda_fail(hwr_ctx *c, cudaError_t e, const char *what) {
    return fail(c, e == cudaErrorMemoryAllocation ? HWR_ERR_OOM : HWR_ERR_CUDA,
                "%s: %s", what, cudaGetErrorString(e));
}

#define CK(ctx, call, what)                                   \
    do {                                                      \
        cudaError_t e_ = (call);                              \
        if (e_ != cudaSuccess) return cuda_fail(ctx, e_, what); \
    } while (0)

static bool hook_fires(hwr_ctx *c) {
    return c->hook.fail_at > 0 && ++c->hook.count == c->hook.fail_at;
}

template <class T>
static hwr_status dev_alloc(hwr_ctx *c, T **p, size_t n) {
    *p = nullptr;
    if (n == 0) n = 1;
    if (hook_fires(c)) return fail(c, HWR_ERR_OOM, "allocation %ld failed (test hook)", c->hook.count);
    void *q = nullptr;
    cudaError_t e = cudaMalloc(&q, n * sizeof(T));
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(c, HWR_ERR_OOM, "cudaMalloc(%zu): %s", n * sizeof(T), cudaGetErrorString(e));
    }
    c->allocs.push_back(q);
    *p = (T *)q;
    return HWR_OK;
}

static void dev_free(hwr_ctx *c, void *p) {
    if (!p) return;
    for (size_t i = 0; i < c->allocs.size(); ++i)
        if (c->allocs[i] == p) {
            c->allocs.erase(c->allocs.begin() + i);
            break;
        }
    cudaFree(p);
}

// Grow a scratch buffer to hold n elements (contents not preserved).
template <class T>
static hwr_status grow(hwr_ctx *c, T **p, size_t *cap, size_t n) {
    if (n <= *cap && *p) return HWR_OK;
    size_t want = n + n / 4 + 64;
    if (*p) {
        cudaError_t e = cudaStreamSynchronize(c->stream);
        if (e != cudaSuccess) return cuda_fail(c, e, "synchronize before regrow");
        dev_free(c, *p);
        *p = nullptr;
        *cap = 0;
    }
    hwr_status s = dev_alloc(c, p, want);
    if (s == HWR_OK) *cap = want;
    return s;
}

static hwr_status pin_grow(hwr_ctx *c, size_t bytes) {
    if (bytes <= c->pin_cap && c->pin_h) return HWR_OK;
    if (c->pin_h) {
        cudaStreamSynchronize(c->stream);
        cudaFreeHost(c->pin_h);
        c->pin_h = nullptr;
        c->pin_cap = 0;
    }
    size_t want = bytes + bytes / 4 + 4096;
    if (hook_fires(c)) return fail(c, HWR_ERR_OOM, "allocation %ld failed (test hook)", c->hook.count);
    cudaError_t e = cudaHostAlloc((void **)&c->pin_h, want, cudaHostAllocMapped);
    if (e == cudaSuccess) e = cudaHostGetDevicePointer((void **)&c->pin_d, c->pin_h, 0);
    if (e != cudaSuccess) {
        cudaGetLastError();
        if (c->pin_h) cudaFreeHost(c->pin_h);
        c->pin_h = nullptr;
        c->pin_d = nullptr;
        return fail(c, HWR_ERR_OOM, "cudaHostAlloc(%zu): %s", want, cudaGetErrorString(e));
    }
    c->pin_cap = want;
    return HWR_OK;
}

static float bf16_bits_to_f32(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
}

static Model model_view(const hwr_ctx *c) {
    Model m;
    m.M = c->M; m.G = c->G; m.D = c->D; m.F = c->F; m.H1 = c->H1; m.H2 = c->H2;
    m.E = c->E; m.P = c->P; m.NH = c->NH;
    m.dep_model = c->dep_model; m.dep_gpu = c->dep_gpu; m.log10p = c->log10p;
    m.W1 = c->W1; m.b1 = c->b1; m.W2 = c->W2; m.b2 = c->b2; m.W3 = c->W3; m.b3 = c->b3;
    m.W2T = c->W2T; m.H2p = (c->H2 + 3) & ~3; m.W1T = c->W1T;
    m.mu = c->mu; m.sd = c->sd; m.xform = c->xform; m.memb = c->memb;
    m.running = c->running; m.waiting = c->waiting; m.kv = c->kv;
    m.gpu_util = c->gpu_util; m.ttft = c->ttft; m.tpot = c->tpot;
    m.X = c->X; m.Spre = c->Spre; m.A = c->A; m.Abf = c->Abf;
    return m;
}

static TcModel tc_view(const hwr_ctx *c) {
    TcModel t;
    t.M = c->M; t.Mpad = c->Mpad; t.D = c->D; t.H1 = c->H1; t.H2 = c->H2;
    t.E = c->E; t.Epad = c->Epad; t.NH = c->NH;
    t.W2img = c->W2img; t.membimg = c->membimg; t.Abf = c->Abf; t.W1q = c->W1q;
    t.b2 = c->b2; t.W3 = c->W3; t.b3 = c->b3; t.dep_model = c->dep_model;
    t.mu_in = c->mu_in; t.sd_in = c->sd_in; t.mu_out = c->mu_out; t.sd_out = c->sd_out;
    t.xf_in = c->xf_in; t.xf_out = c->xf_out;
    t.head = (const HeadConsts *)c->head_consts.data();
    t.test_stall = c->test_stall;
    return t;
}

// Profiling: bracket a launch with events when asked.
static cudaEvent_t take_event(hwr_ctx *c) {
    if (!c->ev_pool.empty()) {
        cudaEvent_t e = c->ev_pool.back();
        c->ev_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    return e;
}

struct LaunchScope {
    hwr_ctx *c;
    int k;
    bool prof;
    cudaEvent_t a = nullptr;
    LaunchScope(hwr_ctx *c_, int k_, bool prof_) : c(c_), k(k_), prof(prof_) {
        if (prof && (a = take_event(c))) cudaEventRecord(a, c->stream);
    }
    void done() {
        c->stats.kernel_launches++;
        c->stats.launches[k]++;
        if (prof && a) {
            cudaEvent_t b = take_event(c);
            if (b) {
                cudaEventRecord(b, c->stream);
                c->pending.push_back({k, a, b});
            } else {
                c->ev_pool.push_back(a);
            }
        }
    }
};

static hwr_status collect_profile(hwr_ctx *c) {
    if (c->pending.empty()) return HWR_OK;
    CK(c, cudaStreamSynchronize(c->stream), "synchronize for profile");
    for (auto &p : c->pending) {
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) {
            c->stats.profiled_ms[p.k] += ms;
            c->stats.profiled_launches[p.k]++;
        } else {
            cudaGetLastError();
        }
        c->ev_pool.push_back(p.a);
        c->ev_pool.push_back(p.b);
    }
    c->pending.clear();
    return HWR_OK;
}

static hwr_status check_status_word(hwr_ctx *c) {
    int32_t st = *(volatile int32_t *)c->status_h;
    if (st == ST_TIMEOUT)
        return fail(c, HWR_ERR_TIMEOUT, "a device-side wait exceeded its bound (kernel gave up)");
    if (st != ST_OK) return fail(c, HWR_ERR_CUDA, "kernel reported status %d", st);
    return HWR_OK;
}

// ---------------------------------------------------------------------------
// create / destroy

static hwr_status validate_create(const hwr_deployment_table *t, const hwr_predictor *p,
                                  const void *memb, int32_t E, hwr_dtype edt) {
    if (!t || !p || !memb) return fail(nullptr, HWR_ERR_INVALID_ARG, "NULL table, predictor or model_emb");
    if (!t->dep_model || !t->dep_gpu || !t->model_log10_params)
        return fail(nullptr, HWR_ERR_INVALID_ARG, "NULL array in deployment table");
    if (!p->W1 || !p->W2 || !p->W3 || !p->b1 || !p->b2 || !p->b3 || !p->feat_mean ||
        !p->feat_std || !p->feat_xform)
        return fail(nullptr, HWR_ERR_INVALID_ARG, "NULL array in predictor");
    const int M = t->n_models, G = t->n_gpu_types, D = t->n_deployments;
    if (M < 1 || G < 1 || D < 1) return fail(nullptr, HWR_ERR_INVALID_ARG, "M, G and D must be >= 1");
    if (p->dtype != HWR_F32 && p->dtype != HWR_BF16)
        return fail(nullptr, HWR_ERR_INVALID_ARG, "unknown predictor dtype %d", (int)p->dtype);
    if (edt != p->dtype)
        return fail(nullptr, HWR_ERR_DTYPE, "embedding dtype %d differs from predictor dtype %d",
                    (int)edt, (int)p->dtype);
    if (p->F < M + G + 9) return fail(nullptr, HWR_ERR_INVALID_ARG, "F=%d < M+G+9=%d", p->F, M + G + 9);
    if (E < 8 || E % 8) return fail(nullptr, HWR_ERR_INVALID_ARG, "E=%d must be a multiple of 8, >= 8", E);
    if (p->H1 < 1 || p->H2 < 1) return fail(nullptr, HWR_ERR_INVALID_ARG, "H1, H2 must be >= 1");
    if (D > MAX_D) return fail(nullptr, HWR_ERR_UNSUPPORTED, "D=%d > %d", D, MAX_D);
    if (p->H1 > MAX_H || p->H2 > MAX_H) return fail(nullptr, HWR_ERR_UNSUPPORTED, "H1/H2 > %d", MAX_H);
    if (p->F > 256) return fail(nullptr, HWR_ERR_UNSUPPORTED, "F=%d > 256", p->F);
    if (E > 8192) return fail(nullptr, HWR_ERR_UNSUPPORTED, "E=%d > 8192", E);
    if (M > 64) return fail(nullptr, HWR_ERR_UNSUPPORTED, "M=%d > 64", M);
    for (int d = 0; d < D; ++d) {
        if (t->dep_model[d] < 0 || t->dep_model[d] >= M || t->dep_gpu[d] < 0 || t->dep_gpu[d] >= G)
            return fail(nullptr, HWR_ERR_INVALID_ARG, "deployment %d: model/gpu id out of range", d);
    }
    for (int k = 0; k < p->F; ++k) {
        if (!(p->feat_std[k] != 0.f) || !isfinite(p->feat_std[k]) || !isfinite(p->feat_mean[k]))
            return fail(nullptr, HWR_ERR_INVALID_ARG, "feature %d: std must be finite and non-zero", k);
        if (p->feat_xform[k] > 2) return fail(nullptr, HWR_ERR_INVALID_ARG, "feature %d: xform > 2", k);
    }
    if (p->n_heads != 0 && p->n_heads != 2 && p->n_heads != 3)
        return fail(nullptr, HWR_ERR_INVALID_ARG, "n_heads=%d (2 or 3)", p->n_heads);
    return HWR_OK;
}

static hwr_status upload(hwr_ctx *c, void *dst, const void *src, size_t bytes, const char *what) {
    CK(c, cudaMemcpy(dst, src, bytes, cudaMemcpyHostToDevice), what);
    return HWR_OK;
}

#define TRY(x)                          \
    do {                                \
        hwr_status s_ = (x);            \
        if (s_ != HWR_OK) return s_;    \
    } while (0)

static hwr_status build_ctx(hwr_ctx *c, const hwr_deployment_table *t, const hwr_predictor *p,
                            const void *memb_in, void *stream) {
    const int M = c->M, D = c->D, F = c->F, H1 = c->H1, H2 = c->H2, E = c->E;
    const bool bf = c->dtype == HWR_BF16;
    if (stream) {
        c->stream = (cudaStream_t)stream;
    } else {
        CK(c, cudaStreamCreateWithFlags(&c->stream, cudaStreamNonBlocking), "create stream");
        c->own_stream = true;
    }
    CK(c, simt_prepare(), "configure SIMT kernels");

    // fp32 copies of every weight (bf16 widened exactly)
    auto widen = [&](const void *src, size_t n) {
        std::vector<float> v(n);
        if (bf) {
            const uint16_t *s = (const uint16_t *)src;
            for (size_t i = 0; i < n; ++i) v[i] = bf16_bits_to_f32(s[i]);
        } else {
            memcpy(v.data(), src, n * sizeof(float));
        }
        return v;
    };
    const int NH = c->NH;
    std::vector<float> w1 = widen(p->W1, (size_t)H1 * F), w2 = widen(p->W2, (size_t)H2 * H1),
                       w3 = widen(p->W3, (size_t)NH * H2), me = widen(memb_in, (size_t)E * M);

    TRY(dev_alloc(c, &c->dep_model, D));
    TRY(dev_alloc(c, &c->dep_gpu, D));
    TRY(dev_alloc(c, &c->log10p, M));
    TRY(dev_alloc(c, &c->W1, w1.size()));
    TRY(dev_alloc(c, &c->b1, H1));
    TRY(dev_alloc(c, &c->W2, w2.size()));
    TRY(dev_alloc(c, &c->b2, H2));
    TRY(dev_alloc(c, &c->W3, w3.size()));
    TRY(dev_alloc(c, &c->b3, 3));
    TRY(dev_alloc(c, &c->mu, F));
    TRY(dev_alloc(c, &c->sd, F));
    TRY(dev_alloc(c, &c->xform, F));
    TRY(dev_alloc(c, &c->memb, me.size()));
    TRY(dev_alloc(c, &c->W1q, 2 * (size_t)H1));
    const int H2p = (H2 + 3) & ~3;
    TRY(dev_alloc(c, &c->W2T, (size_t)H1 * H2p));
    TRY(dev_alloc(c, &c->W1T, (size_t)F * H1));
    TRY(dev_alloc(c, &c->pairC, (size_t)PAIRS_MAX_PAIRS));
    TRY(dev_alloc(c, &c->pairQ, (size_t)PAIRS_MAX_PAIRS * M));
    TRY(dev_alloc(c, &c->pairN, 2 * (size_t)PAIRS_MAX_PAIRS));
    TRY(dev_alloc(c, &c->pairH, (size_t)PAIRS_MAX_PAIRS * H2));
    // the six snapshot arrays, contiguous: an upload lands in them directly
    TRY(dev_alloc(c, (char **)&c->snap_d, 6 * (size_t)D * 4));
    c->running = (int32_t *)c->snap_d;
    c->waiting = c->running + D;
    c->kv = (float *)(c->waiting + D);
    c->gpu_util = c->kv + D;
    c->ttft = c->gpu_util + D;
    c->tpot = c->ttft + D;
    TRY(dev_alloc(c, &c->X, (size_t)D * F));
    TRY(dev_alloc(c, &c->Spre, (size_t)D * H1));
    TRY(dev_alloc(c, &c->A, (size_t)D * H1));
    TRY(dev_alloc(c, &c->Abf, (size_t)D * H1));

    TRY(upload(c, c->dep_model, t->dep_model, D * 4, "upload table"));
    TRY(upload(c, c->dep_gpu, t->dep_gpu, D * 4, "upload table"));
    TRY(upload(c, c->log10p, t->model_log10_params, M * 4, "upload table"));
    TRY(upload(c, c->W1, w1.data(), w1.size() * 4, "upload W1"));
    TRY(upload(c, c->b1, p->b1, H1 * 4, "upload b1"));
    TRY(upload(c, c->W2, w2.data(), w2.size() * 4, "upload W2"));
    TRY(upload(c, c->b2, p->b2, H2 * 4, "upload b2"));
    TRY(upload(c, c->W3, w3.data(), w3.size() * 4, "upload W3"));
    TRY(upload(c, c->b3, p->b3, (size_t)NH * 4, "upload b3"));
    TRY(upload(c, c->mu, p->feat_mean, F * 4, "upload mean"));
    TRY(upload(c, c->sd, p->feat_std, F * 4, "upload std"));
    TRY(upload(c, c->xform, p->feat_xform, F, "upload xform"));
    TRY(upload(c, c->memb, me.data(), me.size() * 4, "upload model embeddings"));
    std::vector<float> w1q(2 * (size_t)H1);
    for (int j = 0; j < H1; ++j) {
        w1q[j] = w1[(size_t)j * F + F - 2];
        w1q[H1 + j] = w1[(size_t)j * F + F - 1];
    }
    TRY(upload(c, c->W1q, w1q.data(), w1q.size() * 4, "upload W1 query columns"));
    std::vector<float> w2t((size_t)H1 * H2p, 0.0f);
    for (int n = 0; n < H2; ++n)
        for (int k = 0; k < H1; ++k) w2t[(size_t)k * H2p + n] = w2[(size_t)n * H1 + k];
    TRY(upload(c, c->W2T, w2t.data(), w2t.size() * 4, "upload W2 transposed"));
    std::vector<float> w1t((size_t)F * H1);
    for (int j = 0; j < H1; ++j)
        for (int k = 0; k < F; ++k) w1t[(size_t)k * H1 + j] = w1[(size_t)j * F + k];
    TRY(upload(c, c->W1T, w1t.data(), w1t.size() * 4, "upload W1 transposed"));
    CK(c, cudaMemset(c->pairN, 0, 2 * PAIRS_MAX_PAIRS * sizeof(int32_t)), "zero counters");
    c->xform_h.assign(p->feat_xform, p->feat_xform + F);
    c->mu_in = p->feat_mean[F - 2]; c->sd_in = p->feat_std[F - 2]; c->xf_in = p->feat_xform[F - 2];
    c->mu_out = p->feat_mean[F - 1]; c->sd_out = p->feat_std[F - 1]; c->xf_out = p->feat_xform[F - 1];

    CK(c, cudaMemset(c->running, 0, D * 4), "zero snapshot");
    CK(c, cudaMemset(c->waiting, 0, D * 4), "zero snapshot");
    CK(c, cudaMemset(c->kv, 0, D * 4), "zero snapshot");
    CK(c, cudaMemset(c->gpu_util, 0, D * 4), "zero snapshot");
    CK(c, cudaMemset(c->ttft, 0, D * 4), "zero snapshot");
    CK(c, cudaMemset(c->tpot, 0, D * 4), "zero snapshot");

    // tensor-core images (bf16 only)
    c->Mpad = M <= 16 ? 16 : 32;
    c->Epad = (E + 63) / 64 * 64;
    c->tc_ok = bf && tc_supported(M, H1, H2, E);
    if (c->tc_ok) {
        CK(c, tc_prepare(), "configure tensor-core kernels");
        std::vector<uint16_t> img(tc_w2img_elems(H1, H2));
        tc_build_w2img((const uint16_t *)p->W2, H1, H2, img.data());
        TRY(dev_alloc(c, &c->W2img, img.size()));
        TRY(dev_alloc(c, &c->done_d, 1));
        CK(c, cudaMemset(c->done_d, 0, sizeof(uint32_t)), "zero completion counter");
        TRY(upload(c, c->W2img, img.data(), img.size() * 2, "upload W2 image"));
        std::vector<uint16_t> mimg(tc_membimg_elems(c->Mpad, c->Epad));
        tc_build_membimg((const uint16_t *)memb_in, E, M, c->Mpad, c->Epad, mimg.data());
        TRY(dev_alloc(c, &c->membimg, mimg.size()));
        TRY(upload(c, c->membimg, mimg.data(), mimg.size() * 2, "upload memb image"));
        c->head_consts.resize(tc_head_consts_bytes());
        tc_fill_head_consts(c->head_consts.data(), p->b2, w3.data(), p->b3, H2, NH);
    }

    // status word: mapped pinned host memory the kernels write directly
    if (hook_fires(c)) return fail(c, HWR_ERR_OOM, "allocation %ld failed (test hook)", c->hook.count);
    CK(c, cudaHostAlloc((void **)&c->status_h, 64, cudaHostAllocMapped), "alloc status word");
    memset(c->status_h, 0, 64);
    CK(c, cudaHostGetDevicePointer((void **)&c->status_d, c->status_h, 0), "map status word");

    // snapshot staging: 6 arrays of D 4-byte values
    if (hook_fires(c)) return fail(c, HWR_ERR_OOM, "allocation %ld failed (test hook)", c->hook.count);
    CK(c, cudaHostAlloc(&c->snap_h, 6 * (size_t)D * 4, cudaHostAllocMapped), "alloc snapshot staging");
    CK(c, cudaHostGetDevicePointer((void **)&c->snap_hd, c->snap_h, 0), "map snapshot staging");
    CK(c, cudaEventCreateWithFlags(&c->snap_ev, cudaEventDisableTiming), "create event");
    CK(c, cudaEventCreateWithFlags(&c->pin_ev, cudaEventDisableTiming), "create event");
    CK(c, cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking), "create copy stream");
    for (auto &e : c->chunk_ev)
        CK(c, cudaEventCreateWithFlags(&e, cudaEventDisableTiming), "create event");
    CK(c, cudaEventCreateWithFlags(&c->io_free_ev, cudaEventDisableTiming), "create event");

    c->seq_qs = seq_chunk(model_view(c));
    c->seq_slots = seq_table_slots(model_view(c));
    CK(c, cudaDeviceGetAttribute(&c->nsm, cudaDevAttrMultiProcessorCount, c->device), "SM count");
    CK(c, cudaDeviceSynchronize(), "create");
    return HWR_OK;
}

static void free_ctx(hwr_ctx *c) {
    if (c->stream) cudaStreamSynchronize(c->stream);
    for (auto &p : c->pending) {
        cudaEventDestroy(p.a);
        cudaEventDestroy(p.b);
    }
    for (auto e : c->ev_pool) cudaEventDestroy(e);
    for (void *p : c->allocs) cudaFree(p);
    c->allocs.clear();
    if (c->status_h) cudaFreeHost(c->status_h);
    if (c->snap_h) cudaFreeHost(c->snap_h);
    if (c->pin_h) cudaFreeHost(c->pin_h);
    if (c->snap_ev) cudaEventDestroy(c->snap_ev);
    if (c->pin_ev) cudaEventDestroy(c->pin_ev);
    for (auto e : c->chunk_ev)
        if (e) cudaEventDestroy(e);
    if (c->io_free_ev) cudaEventDestroy(c->io_free_ev);
    if (c->copy_stream) {
        cudaStreamSynchronize(c->copy_stream);
        cudaStreamDestroy(c->copy_stream);
    }
    if (c->own_stream && c->stream) cudaStreamDestroy(c->stream);
    cudaGetLastError();
    delete c;
}

extern "C" hwr_status hwr_create(const hwr_deployment_table *table, const hwr_predictor *pred,
                                 const void *model_emb, int32_t E, hwr_dtype emb_dtype,
                                 void *cuda_stream, hwr_ctx **out) {
    ApiRange range_("hwr_create");
    if (!out) return fail(nullptr, HWR_ERR_INVALID_ARG, "out is NULL");
    *out = nullptr;
    g_create_error.clear();
    hwr_status s = validate_create(table, pred, model_emb, E, emb_dtype);
    if (s != HWR_OK) return s;
    hwr_ctx *c = new (std::nothrow) hwr_ctx();
    if (!c) return fail(nullptr, HWR_ERR_OOM, "host allocation failed");
    memset(&c->stats, 0, sizeof c->stats);
    c->M = table->n_models; c->G = table->n_gpu_types; c->D = table->n_deployments;
    c->F = pred->F; c->H1 = pred->H1; c->H2 = pred->H2; c->E = E; c->P = c->M + c->G;
    c->dtype = pred->dtype;
    c->NH = pred->n_heads == 3 ? 3 : 2;
    if (cudaGetDevice(&c->device) != cudaSuccess) {
        cudaGetLastError();
        delete c;
        return fail(nullptr, HWR_ERR_CUDA, "no current CUDA device");
    }
    if (const char *h = getenv("HWR_TEST_FAIL_ALLOC")) c->hook.fail_at = atol(h);
    if (const char *h = getenv("HWR_TEST_POLL_US")) c->poll_us = atol(h) < 0 ? 0 : atol(h);
    {
        int pageable = 0;
        if (cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, c->device) !=
            cudaSuccess) {
            cudaGetLastError();
            pageable = 0;
        }
        const char *h = getenv("HWR_TEST_NO_ATS");   // test hook: force the staging copies
        c->ats = pageable == 1 && !(h && atoi(h) != 0);
    }
    if (const char *h = getenv("HWR_TEST_STALL")) c->test_stall = atoi(h) != 0;
    if (const char *h = getenv("HWR_TC_MIN_PAIRS")) c->tc_min_pairs = atoi(h) > 1 ? atoi(h) : 1;
    if (const char *h = getenv("HWR_PAIRS_MAX_PAIRS"))
        c->pairs_max = atoi(h) < 0 ? 0 : (atoi(h) > PAIRS_MAX_PAIRS ? PAIRS_MAX_PAIRS : atoi(h));
    s = build_ctx(c, table, pred, model_emb, cuda_stream);
    if (s != HWR_OK) {
        g_create_error = c->err;
        free_ctx(c);
        return s;
    }
    if (c->pairs_max < 0)
        c->pairs_max = c->tc_ok ? SMALL_MAX_PAIRS : c->H1 * c->H2 > 64 * 64 ? FP32_MAX_PAIRS : 0;
    *out = c;
    return HWR_OK;
}

extern "C" hwr_status hwr_destroy(hwr_ctx *c) {
    ApiRange range_("hwr_destroy");
    if (c) free_ctx(c);
    return HWR_OK;
}

// ---------------------------------------------------------------------------
// snapshot

extern "C" hwr_status hwr_update_snapshot(hwr_ctx *c, const hwr_snapshot *s) {
    ApiRange range_("hwr_update_snapshot");
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (c->broken) return HWR_ERR_STATE;
    if (!s || !s->running || !s->waiting || !s->kv_util || !s->gpu_util || !s->ttft_avg ||
        !s->tpot_avg)
        return fail(c, HWR_ERR_INVALID_ARG, "NULL snapshot array");
    // every signal must be a value its feature transform accepts: counts
    // >= 0, finite values, > 0 under log, > -1 under log1p
    const float *fs[4] = {s->kv_util, s->gpu_util, s->ttft_avg, s->tpot_avg};
    static const char *names[6] = {"running", "waiting", "kv_util", "gpu_util", "ttft_avg",
                                   "tpot_avg"};
    for (int k = 0; k < 6; ++k) {
        const uint8_t xf = c->xform_h[c->P + 1 + k];
        for (int d = 0; d < c->D; ++d) {
            const double v = k < 2 ? (double)(k == 0 ? s->running : s->waiting)[d] : (double)fs[k - 2][d];
            const bool bad = !isfinite(v) || (k < 2 && v < 0) || (xf == 2 && !(v > 0)) ||
                             (xf == 1 && !(v > -1));
            if (bad)
                return fail(c, HWR_ERR_INVALID_ARG,
                            "snapshot %s[%d] = %g is outside the domain of its feature%s", names[k],
                            d, v, xf == 2 ? " (log)" : xf == 1 ? " (log1p)" : "");
        }
    }
    const size_t n = (size_t)c->D * 4;
    // the previous snapshot copy must have left the staging buffer
    if (c->snap_busy) CK(c, cudaEventSynchronize(c->snap_ev), "wait for snapshot staging");
    char *h = (char *)c->snap_h;
    memcpy(h + 0 * n, s->running, n);
    memcpy(h + 1 * n, s->waiting, n);
    memcpy(h + 2 * n, s->kv_util, n);
    memcpy(h + 3 * n, s->gpu_util, n);
    memcpy(h + 4 * n, s->ttft_avg, n);
    memcpy(h + 5 * n, s->tpot_avg, n);
    // the snapshot kernel reads the staging (mapped) into the six device arrays
    // itself: no separate copy; the staging is free again once it has run
    LaunchScope ls(c, HWR_K_SNAPSHOT, false);
    CK(c, launch_snapshot(model_view(c), c->snap_hd, c->stream), "snapshot kernel");
    ls.done();
    CK(c, cudaEventRecord(c->snap_ev, c->stream), "record");
    c->snap_busy = true;
    c->have_snapshot = true;
    return HWR_OK;
}

extern "C" hwr_status hwr_get_snapshot(hwr_ctx *c, int32_t *running_out) {
    ApiRange range_("hwr_get_snapshot");
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (c->broken) return HWR_ERR_STATE;
    if (!running_out) return fail(c, HWR_ERR_INVALID_ARG, "running_out is NULL");
    CK(c, cudaMemcpyAsync(running_out, c->running, (size_t)c->D * 4, cudaMemcpyDeviceToHost,
                          c->stream), "read running counts");
    CK(c, cudaStreamSynchronize(c->stream), "synchronize");
    c->snap_busy = false;
    return HWR_OK;
}

// ---------------------------------------------------------------------------
// routing

// Whether byte ranges [a, a + na) and [b, b + nb) share a byte.
static bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
    const uintptr_t x = (uintptr_t)a, y = (uintptr_t)b;
    return a && b && na && nb && x < y + nb && y < x + na;
}

static hwr_status run_kernels(hwr_ctx *c, const Queries &q, uint32_t flags, bool tensor) {
    const bool prof = flags & HWR_PROFILE;
    const Model m = model_view(c);
    if (flags & HWR_SEQUENTIAL) {
        // HWR_PATH_TENSOR: the table on the tensor cores (bf16 contexts)
        const bool tcs = (flags & HWR_PATH_TENSOR) && c->tc_ok;
        // Chunks of equal size, at most the limit: the SIMT table grows with
        // the square of a chunk, so 64 queries under a 55-query limit run as
        // 32 + 32, not 55 + 9 (the walk, and so every result, is the same
        // either way).  The tensor-core table is cheap per entry and a chunk
        // costs four dependent kernels: its chunks go up to SEQ_MAX_CHUNK,
        // the chain reading the rows that do not fit its shared memory from L2.
        const int limit = tcs ? SEQ_MAX_CHUNK : c->seq_qs;
        const int nchunks = (q.Q + limit - 1) / limit;
        const int Qs = (q.Q + nchunks - 1) / nchunks;
        if (tcs) {
            const size_t Dv = (size_t)c->D * (Qs + 1);
            TRY(grow(c, &c->prebf, &c->prebf_cap, Dv * c->H1));
            TRY(grow(c, &c->dmv, &c->dmv_cap, Dv));
            TRY(grow(c, &c->qual, &c->qual_cap, 2 * (size_t)Qs * c->Mpad));
        }
        TRY(grow(c, &c->ctab, &c->ctab_cap, seq_table_floats(c->D, Qs)));
        TRY(grow(c, &c->qseq, &c->qseq_cap, seq_aux_floats(c->D, c->M, c->H1, Qs)));
        const size_t es = c->dtype == HWR_BF16 ? 2 : 4;
        for (int lo = 0; lo < q.Q; lo += Qs) {
            Queries k = q;
            const int n = q.Q - lo < Qs ? q.Q - lo : Qs;
            k.Q = n;
            k.in_len = q.in_len + lo;
            k.out_len = q.out_len + lo;
            k.emb = (const char *)q.emb + (size_t)lo * c->E * es;
            k.chosen = q.chosen + lo;
            k.lat = q.lat + lo;
            k.util = q.util + lo;
            if (q.slo_q) k.slo_q = q.slo_q + lo;
            if (tcs) {
                // preparation (features, prefixes, their bf16 copies), then the
                // chunk's quality and the cost of every (query, deployment,
                // count) on the tensor cores, then the chain.  The predictor
                // kernel runs as a dependent of the quality kernel: only its
                // epilogue waits, and the prefixes it reads early come from the
                // preparation kernel, which finished before the quality kernel
                // began.
                const TcModel t = tc_view(c);
                TcModel tv = t;
                tv.D = c->D * (n + 1);
                tv.Abf = c->prebf;
                tv.dep_model = c->dmv;
                Queries kt = k;
                kt.pair_C = c->ctab;
                kt.seq_n = n;
                kt.no_select = 1;
                kt.slo_mode = 0;      // budgets are the chain's business
                kt.slo_q = nullptr;
                LaunchScope a(c, HWR_K_SEQ_TABLE, prof);
                CK(c, launch_seq_prep_tc(m, k, n, c->qseq, c->prebf, c->dmv, c->stream),
                   "sequential preparation");
                // fixed halves of the buffer (calls of different sizes must not
                // overlap the half the previous call's kernels still read)
                float *qb = c->qual + (c->qual_flip ? c->qual_cap / 2 : 0);
                c->qual_flip ^= 1;
                // the preparation kernel lets its dependents start early, and
                // the cost table reads its prefixes before its dependency wait:
                // the table starts only once this grid has waited for it
                CK(c, launch_qual_tc(t, k, qb, c->status_d, c->stream, true, false, 0, c->done_d,
                                     c->pred_ctas - c->pred_ctas_last),
                   "quality kernel");
                int ctas = 0;
                CK(c, launch_mlp_tc_scores(tv, kt, qb, c->status_d, c->stream, c->done_d, &ctas),
                   "sequential table (tensor cores)");
                c->pred_ctas += (uint32_t)ctas;
                c->pred_ctas_last = (uint32_t)ctas;
                a.done();
                CK(c, launch_seq_chain_tc(m, k, n, c->ctab, c->qseq, qb, c->Mpad, c->stream),
                   "sequential chain");
                // preparation, quality and chain beside the scope's table kernel
                c->stats.kernel_launches += 3;
                c->stats.launches[HWR_K_SEQ_TABLE] += 3;
                continue;
            }
            LaunchScope a(c, HWR_K_SEQ_TABLE, prof);
            CK(c, launch_seq_table(m, k, n, c->seq_slots, c->ctab, c->qseq, c->stream),
               "sequential table");
            a.done();
            CK(c, launch_seq_chain(m, k, n, c->ctab, c->qseq, c->stream), "sequential chain");
            // the preparation kernel (inside launch_seq_table) and the chain
            c->stats.kernel_launches += 2;
            c->stats.launches[HWR_K_SEQ_TABLE] += 2;
        }
        return HWR_OK;
    }
    if (tensor) {
        const TcModel t = tc_view(c);
        TRY(grow(c, &c->qual, &c->qual_cap, 2 * (size_t)q.Q * c->Mpad));
        // the two halves alternate, so this call's quality kernel may run
        // alongside the previous call's predictor, which reads the other
        float *qb = c->qual + (c->qual_flip ? c->qual_cap / 2 : 0);
        c->qual_flip ^= 1;
        c->qual_last = qb;
        const MlpSplit sp = tc_mlp_split(t, q.Q);
        if (sp.nsplit > 1) {
            TRY(grow(c, &c->part, &c->part_cap, (size_t)sp.nsplit * q.Q * 16));
            if (c->count_cap < (size_t)q.Q) {
                TRY(grow(c, &c->count, &c->count_cap, (size_t)q.Q));
                CK(c, cudaMemsetAsync(c->count, 0, c->count_cap * 4, c->stream), "zero counters");
            }
        }
        // The predictor may start as soon as the quality kernel has: before
        // its dependency wait it reads only weights, the snapshot's prefixes
        // and this call's inputs -- unless those inputs are outputs of the
        // previous tensor-core route, whose predictor may still be running.
        const size_t qb4 = (size_t)q.Q * 4;
        bool early = true;
        for (const auto &o : c->prev_out)
            if (overlaps(q.in_len, qb4, o.p, o.n) || overlaps(q.out_len, qb4, o.p, o.n) ||
                overlaps(q.emb, (size_t)q.Q * c->E * 2, o.p, o.n) ||
                (q.slo_q && overlaps(q.slo_q, qb4, o.p, o.n)))
                early = false;
        const int free_sms = tc_mlp_free_sms(q.Q, sp);
        LaunchScope a(c, HWR_K_QUAL_TC, prof);
        CK(c, launch_qual_tc(t, q, qb, c->status_d, c->stream, true, early, free_sms, c->done_d,
                             c->pred_ctas - c->pred_ctas_last),
           "quality kernel");
        a.done();
        c->prev_out[0] = {q.chosen, qb4};
        c->prev_out[1] = {q.lat, qb4};
        c->prev_out[2] = {q.util, qb4};
        c->prev_out[3] = {q.pair_C, q.pair_C ? qb4 * c->D : 0};
        LaunchScope b(c, HWR_K_MLP_TC, prof);
        int ctas = 0;
        CK(c, launch_mlp_tc(t, q, qb, sp, c->part, c->count, c->status_d, c->stream, c->done_d,
                            &ctas),
           "predictor kernel");
        c->pred_ctas += (uint32_t)ctas;
        c->pred_ctas_last = (uint32_t)ctas;
        b.done();
        return HWR_OK;
    }
    LaunchScope a(c, HWR_K_ROUTE_SIMT, prof);
    if ((long)q.Q * c->D <= c->pairs_max)
        CK(c, launch_route_pairs(m, q, c->pairC, c->pairQ, c->pairH, c->pairN, c->nsm, c->stream),
           "route kernel");
    else
        CK(c, launch_route_simt(m, q, c->stream), "route kernel");
    a.done();
    return HWR_OK;
}

static size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Outputs of a small synchronous call on the small-batch kernel: the kernel
// stores each query's chosen index last, after a system-scope fence, into
// mapped host memory that held a value it never writes; wait for all Q of
// them (acquire loads).  False after a second: the caller then synchronises
// the stream, which reports a failed launch.
constexpr int32_t OUT_PENDING = INT32_MIN;
static bool wait_chosen(const int32_t *ch, int Q, long limit_us) {
    const auto t0 = std::chrono::steady_clock::now();
    const auto limit = std::chrono::microseconds(limit_us);
    for (int i = 0; i < Q; ++i) {
        unsigned n = 0;
        while (__atomic_load_n(ch + i, __ATOMIC_ACQUIRE) == OUT_PENDING)
            if ((++n & 1023u) == 0 && std::chrono::steady_clock::now() - t0 > limit) return false;
    }
    return true;
}

// Shared body of hwr_route_batch and hwr_route_batch_slo.  `spec` (may be
// NULL) replaces the scalar SLO by per-query budgets or the Eq. 4-5 model.
// Score outputs of hwr_score_batch: cost [Q][D] and quality [Q][M] (either may be NULL).
struct ScoreOut {
    float *cost;
    float *quality;
};

static hwr_status route_impl(hwr_ctx *c, int32_t Q, const float *in_len, const float *out_len,
                             const void *q_emb, float slo, const hwr_slo_spec *spec,
                             float lambda, uint32_t flags, int32_t *chosen,
                             float *pred_latency, float *utility, const Lambdas *ml = nullptr,
                             const ScoreOut *so = nullptr) {
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (c->broken) return HWR_ERR_STATE;
    const uint32_t known = HWR_SEQUENTIAL | HWR_DEVICE_PTRS | HWR_ASYNC | HWR_SCORE_CONVEX |
                           HWR_PATH_SIMT | HWR_PATH_TENSOR | HWR_PROFILE;
    if (flags & ~known) return fail(c, HWR_ERR_INVALID_ARG, "unknown flag bits 0x%x", flags & ~known);
    if (Q < 0) return fail(c, HWR_ERR_INVALID_ARG, "Q=%d < 0", Q);
    if (Q == 0) return HWR_OK;
    if (!in_len || !out_len || !q_emb || (!so && (!chosen || !pred_latency || !utility)))
        return fail(c, HWR_ERR_INVALID_ARG, "NULL input or output array");
    if (!spec && slo != slo) return fail(c, HWR_ERR_INVALID_ARG, "SLO is NaN");
    if (spec && !spec->budget &&
        !(isfinite(spec->ttft_a) && isfinite(spec->ttft_b) && isfinite(spec->slack) &&
          isfinite(spec->tpot)))
        return fail(c, HWR_ERR_INVALID_ARG, "SLO model parameters must be finite");
    if (!isfinite(lambda)) return fail(c, HWR_ERR_INVALID_ARG, "lambda is not finite");
    if ((flags & HWR_PATH_SIMT) && (flags & HWR_PATH_TENSOR))
        return fail(c, HWR_ERR_INVALID_ARG, "HWR_PATH_SIMT and HWR_PATH_TENSOR together");
    if (!c->have_snapshot)
        return fail(c, HWR_ERR_INVALID_ARG, "route before the first hwr_update_snapshot");
    const bool seq = flags & HWR_SEQUENTIAL;
    if ((flags & HWR_PATH_TENSOR) && !c->tc_ok)
        return fail(c, HWR_ERR_UNSUPPORTED,
                    "tensor-core path unavailable for this context (fp32 or unsupported shape)");
    const bool tensor = !seq && c->tc_ok &&
                        ((flags & HWR_PATH_TENSOR) ||
                         (!(flags & HWR_PATH_SIMT) && (long)Q * c->D >= c->tc_min_pairs &&
                          (long)Q * c->D > c->pairs_max));
    const bool dev = flags & HWR_DEVICE_PTRS;
    const size_t es = c->dtype == HWR_BF16 ? 2 : 4;
    const int K = ml ? ml->K : 1;
    if ((ml || so) && seq)
        return fail(c, HWR_ERR_UNSUPPORTED, "HWR_SEQUENTIAL with several lambdas or scoring");
    if (dev && (tensor || (seq && (flags & HWR_PATH_TENSOR))) && ((uintptr_t)q_emb & 15))
        return fail(c, HWR_ERR_INVALID_ARG, "device q_emb must be 16-byte aligned");

    Queries q;
    q.Q = Q;
    q.emb_bf16 = c->dtype == HWR_BF16;
    q.slo = slo;
    q.lam = lambda;
    q.wq = (flags & HWR_SCORE_CONVEX) ? 1.0f - lambda : 1.0f;
    const bool budgets = spec && spec->budget;
    if (spec) {
        q.slo_mode = budgets ? 1 : 2;
        q.slo_a = spec->ttft_a;
        q.slo_b = spec->ttft_b;
        q.slo_slack = spec->slack;
        q.slo_tpot = spec->tpot;
    }

    const size_t emb_b = (size_t)Q * c->E * es, len_b = (size_t)Q * 4;
    const size_t off_in = align_up(emb_b, 256), off_out = off_in + align_up(len_b, 256);
    const size_t off_slo = off_out + align_up(len_b, 256);
    const size_t in_total = (budgets ? off_slo : off_out) + len_b;
    const size_t outs_b = (size_t)K * len_b;   // each output holds K rows of Q
    const size_t o_lat = align_up(outs_b, 256), o_util = o_lat + align_up(outs_b, 256);
    const size_t out_total = o_util + outs_b;
    const bool packed = !dev && !(flags & HWR_ASYNC) && in_total <= ((size_t)1 << 20);
    // Large host batches: copy in chunks on the copy stream while the kernels
    // of the previous chunk run (the link, not the GPU, bounds this path).  At
    // most eight chunks: on GB300, 4, 6, 12 and 16 chunks of a 65,536-query
    // batch were all slower end to end than 8 (fewer leave a longer compute
    // tail after the last copy, more add per-chunk launch and copy overhead).
    const int nchunk = (!dev && !packed && !seq && Q >= 2 * PIPE_CHUNK_MIN)
                           ? (Q / PIPE_CHUNK_MIN < 8 ? Q / PIPE_CHUNK_MIN : 8) : 1;
    const bool pipelined = nchunk > 1;
    // a small synchronous call for the small-batch kernel or the SIMT
    // sequential kernels: they read the inputs from the mapped staging itself
    // with plain loads (no host-to-device copy)
    const bool zero_copy = packed && !tensor && !ml && !so && (c->pin_d || c->ats) &&
                           (seq ? !(flags & HWR_PATH_TENSOR) : (long)Q * c->D <= c->pairs_max);
    // ... and on these kernels (the small-batch kernel, the sequential chain)
    // the host waits for the outputs themselves instead of synchronising the
    // stream
    // ... unless work queued earlier on the stream (an HWR_ASYNC call, or the
    // caller's own work on a stream it passed in) is still running: then
    // the kernel starts late and the host synchronises instead of spinning
    // ... and where the GPU reaches pageable host memory, from the caller's
    // own arrays: the kernels read the inputs and write the outputs there
    // (plain element loads and stores), with no staging copy either way
    const bool direct = zero_copy && c->ats;
    bool poll = zero_copy && c->poll_us > 0;
    if (poll && (c->async_pending || !c->own_stream)) {
        const cudaError_t e = cudaStreamQuery(c->stream);
        if (e == cudaSuccess) {
            c->async_pending = false;
        } else {
            if (e != cudaErrorNotReady) return cuda_fail(c, e, "query stream");
            poll = false;
        }
    }

    if (dev) {
        q.in_len = in_len; q.out_len = out_len; q.emb = q_emb;
        q.chosen = chosen; q.lat = pred_latency; q.util = utility;
        if (budgets) q.slo_q = spec->budget;
        if (so) {   // the kernels' own decisions go to scratch
            TRY(grow(c, &c->out_d, &c->out_cap, out_total));
            q.chosen = (int32_t *)c->out_d;
            q.lat = (float *)(c->out_d + o_lat);
            q.util = (float *)(c->out_d + o_util);
        }
    } else if (direct) {
        q.inputs_host = 1;
        q.emb = q_emb;
        q.in_len = in_len;
        q.out_len = out_len;
        if (budgets) q.slo_q = spec->budget;
        q.chosen = chosen;
        q.lat = pred_latency;
        q.util = utility;
        if (poll)
            for (int i = 0; i < Q; ++i) chosen[i] = OUT_PENDING;
    } else {
        TRY(grow(c, &c->io_d, &c->io_cap, in_total));
        TRY(grow(c, &c->out_d, &c->out_cap, out_total));
        if (packed) {
            TRY(pin_grow(c, align_up(in_total, 256) + out_total));
            CK(c, cudaEventSynchronize(c->pin_ev), "wait for staging");
            memcpy(c->pin_h, q_emb, emb_b);
            memcpy(c->pin_h + off_in, in_len, len_b);
            memcpy(c->pin_h + off_out, out_len, len_b);
            if (budgets) memcpy(c->pin_h + off_slo, spec->budget, len_b);
            if (poll) {
                int32_t *ch = (int32_t *)(c->pin_h + align_up(in_total, 256));
                for (int i = 0; i < Q; ++i) ch[i] = OUT_PENDING;
            }
            if (!zero_copy)
                CK(c, cudaMemcpyAsync(c->io_d, c->pin_h, in_total, cudaMemcpyHostToDevice,
                                      c->stream), "copy inputs");
        } else if (!pipelined) {
            CK(c, cudaMemcpyAsync(c->io_d, q_emb, emb_b, cudaMemcpyHostToDevice, c->stream), "copy emb");
            CK(c, cudaMemcpyAsync(c->io_d + off_in, in_len, len_b, cudaMemcpyHostToDevice, c->stream),
               "copy in_len");
            CK(c, cudaMemcpyAsync(c->io_d + off_out, out_len, len_b, cudaMemcpyHostToDevice, c->stream),
               "copy out_len");
            if (budgets)
                CK(c, cudaMemcpyAsync(c->io_d + off_slo, spec->budget, len_b, cudaMemcpyHostToDevice,
                                      c->stream), "copy budgets");
        }
        const char *ib = zero_copy ? c->pin_d : c->io_d;
        q.inputs_host = zero_copy;
        q.emb = ib;
        if (budgets) q.slo_q = (const float *)(ib + off_slo);
        q.in_len = (const float *)(ib + off_in);
        q.out_len = (const float *)(ib + off_out);
        // small synchronous calls: the kernels write the outputs straight into
        // the mapped staging (plain stores), so no device-to-host copy follows
        char *ob = packed && !so ? c->pin_d + align_up(in_total, 256) : c->out_d;
        q.chosen = (int32_t *)ob;
        q.lat = (float *)(ob + o_lat);
        q.util = (float *)(ob + o_util);
    }

    const Model mv = model_view(c);
    // Stored scores: cost [Q][D] and quality [Q][M], for the selection over
    // several lambdas or as the output of hwr_score_batch.
    float *SC = nullptr, *SQ = nullptr;
    if (ml || so) {
        if (so && dev) {
            SC = so->cost;
            SQ = so->quality;
        } else {
            TRY(grow(c, &c->mC, &c->mC_cap, (size_t)Q * c->D));
            TRY(grow(c, &c->mQ, &c->mQ_cap, (size_t)Q * c->M));
            SC = c->mC;
            SQ = c->mQ;
        }
    }
    const size_t rowC = (size_t)c->D * 4, rowQ = (size_t)c->M * 4;
    // One chunk [lo, lo + n): its kernels, then (several lambdas) the selection
    // for every lambda from the scores the kernels stored.
    auto run_chunk = [&](Queries qc, int lo) -> hwr_status {
        const int n = qc.Q;
        const bool small = !tensor && (long)n * c->D <= c->pairs_max;
        if (SC) qc.pair_C = SC + (size_t)lo * c->D;
        if (SQ) qc.qual_out = SQ + (size_t)lo * c->M;
        TRY(run_kernels(c, qc, flags, tensor));
        if (!SC && !SQ) return HWR_OK;
        // paths that keep their scores in their own scratch: copy them over
        if (small && SC)
            CK(c, cudaMemcpyAsync(SC + (size_t)lo * c->D, c->pairC, n * rowC,
                                  cudaMemcpyDeviceToDevice, c->stream), "copy costs");
        if (small && SQ)
            CK(c, cudaMemcpyAsync(SQ + (size_t)lo * c->M, c->pairQ, n * rowQ,
                                  cudaMemcpyDeviceToDevice, c->stream), "copy quality");
        // the selection over several lambdas reads the tensor path's quality
        // buffer itself (rows of Mpad); only scoring copies it out
        const float *selQ = SQ ? SQ + (size_t)lo * c->M : nullptr;
        int qstride = c->M;
        if (tensor && SQ && so)
            CK(c, cudaMemcpy2DAsync(SQ + (size_t)lo * c->M, rowQ, c->qual_last, (size_t)c->Mpad * 4,
                                    rowQ, n, cudaMemcpyDeviceToDevice, c->stream),
               "copy quality");
        if (tensor && SQ && !so) {
            selQ = c->qual_last;
            qstride = c->Mpad;
        }
        if (!ml) return HWR_OK;
        Queries qs = qc;
        qs.chosen = q.chosen + lo;
        qs.lat = q.lat + lo;
        qs.util = q.util + lo;
        LaunchScope ls(c, HWR_K_ROUTE_SIMT, flags & HWR_PROFILE);
        CK(c, launch_select_multi(mv, qs, SC + (size_t)lo * c->D, selQ, qstride, *ml, Q,
                                  c->stream), "select kernel");
        ls.done();
        return HWR_OK;
    };

    if (pipelined) {
        // everything already queued on the context stream (earlier calls'
        // kernels read io_d) must finish before io_d is rewritten
        CK(c, cudaEventRecord(c->io_free_ev, c->stream), "record");
        CK(c, cudaStreamWaitEvent(c->copy_stream, c->io_free_ev, 0), "order copies");
        const int per = ((Q + nchunk - 1) / nchunk + 127) / 128 * 128;
        // the lengths (and budgets) of the whole batch in one copy each, ahead
        // of the embedding chunks: small copies per chunk cost more than they move
        CK(c, cudaMemcpyAsync(c->io_d + off_in, in_len, len_b, cudaMemcpyHostToDevice,
                              c->copy_stream), "copy in_len");
        CK(c, cudaMemcpyAsync(c->io_d + off_out, out_len, len_b, cudaMemcpyHostToDevice,
                              c->copy_stream), "copy out_len");
        if (budgets)
            CK(c, cudaMemcpyAsync(c->io_d + off_slo, spec->budget, len_b, cudaMemcpyHostToDevice,
                                  c->copy_stream), "copy budgets");
        int k = 0;
        for (int lo = 0; lo < Q; lo += per, ++k) {
            const int n = Q - lo < per ? Q - lo : per;
            const size_t eo = (size_t)lo * c->E * es, eb = (size_t)n * c->E * es;
            CK(c, cudaMemcpyAsync(c->io_d + eo, (const char *)q_emb + eo, eb, cudaMemcpyHostToDevice,
                                  c->copy_stream), "copy emb");
            CK(c, cudaEventRecord(c->chunk_ev[k], c->copy_stream), "record");
            CK(c, cudaStreamWaitEvent(c->stream, c->chunk_ev[k], 0), "order kernels");
            Queries qc = q;
            qc.Q = n;
            qc.emb = c->io_d + eo;
            qc.in_len = q.in_len + lo;
            qc.out_len = q.out_len + lo;
            qc.chosen = q.chosen + lo;
            qc.lat = q.lat + lo;
            qc.util = q.util + lo;
            if (q.slo_q) qc.slo_q = q.slo_q + lo;
            TRY(run_chunk(qc, lo));
        }
    } else {
        TRY(run_chunk(q, 0));
    }

    bool synced = false;
    if (so && !dev) {
        if (so->cost)
            CK(c, cudaMemcpyAsync(so->cost, SC, (size_t)Q * rowC, cudaMemcpyDeviceToHost, c->stream),
               "copy costs");
        if (so->quality)
            CK(c, cudaMemcpyAsync(so->quality, SQ, (size_t)Q * rowQ, cudaMemcpyDeviceToHost,
                                  c->stream), "copy quality");
    } else if (!dev) {
        if (direct) {
            // outputs are already in the caller's arrays once the kernel wrote them
            if (!(poll && wait_chosen(chosen, Q, c->poll_us)))
                CK(c, cudaStreamSynchronize(c->stream), "synchronize");
            synced = true;
        } else if (packed) {
            const char *ob = c->pin_h + align_up(in_total, 256);
            CK(c, cudaEventRecord(c->pin_ev, c->stream), "record");
            if (!(poll && wait_chosen((const int32_t *)ob, Q, c->poll_us)))
                CK(c, cudaStreamSynchronize(c->stream), "synchronize");
            synced = true;
            memcpy(chosen, ob, outs_b);
            memcpy(pred_latency, ob + o_lat, outs_b);
            memcpy(utility, ob + o_util, outs_b);
        } else {
            CK(c, cudaMemcpyAsync(chosen, c->out_d, outs_b, cudaMemcpyDeviceToHost, c->stream),
               "copy chosen");
            CK(c, cudaMemcpyAsync(pred_latency, c->out_d + o_lat, outs_b, cudaMemcpyDeviceToHost,
                                  c->stream), "copy latency");
            CK(c, cudaMemcpyAsync(utility, c->out_d + o_util, outs_b, cudaMemcpyDeviceToHost,
                                  c->stream), "copy utility");
        }
    }
    c->stats.queries_routed += Q;
    if ((flags & HWR_ASYNC) && !synced) {
        c->async_pending = true;
        return HWR_OK;
    }
    if (!synced) CK(c, cudaStreamSynchronize(c->stream), "synchronize");
    // this call's work is complete, and with it every earlier kernel
    c->async_pending = false;
    c->snap_busy = false;
    CK(c, cudaGetLastError(), "kernel");
    if (tensor || (seq && (flags & HWR_PATH_TENSOR))) TRY(check_status_word(c));
    return HWR_OK;
}

extern "C" hwr_status hwr_route_batch(hwr_ctx *c, int32_t Q, const float *in_len,
                                      const float *out_len, const void *q_emb, float slo,
                                      float lambda, uint32_t flags, int32_t *chosen,
                                      float *pred_latency, float *utility) {
    ApiRange range_("hwr_route_batch");
    return route_impl(c, Q, in_len, out_len, q_emb, slo, nullptr, lambda, flags, chosen,
                      pred_latency, utility);
}

extern "C" hwr_status hwr_score_batch(hwr_ctx *c, int32_t Q, const float *in_len,
                                      const float *out_len, const void *q_emb, uint32_t flags,
                                      float *cost, float *quality) {
    ApiRange range_("hwr_score_batch");
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (!cost && !quality) return fail(c, HWR_ERR_INVALID_ARG, "cost and quality both NULL");
    ScoreOut so{cost, quality};
    return route_impl(c, Q, in_len, out_len, q_emb, INFINITY, nullptr, 0.0f,
                      flags & ~HWR_SCORE_CONVEX, nullptr, nullptr, nullptr, nullptr, &so);
}

extern "C" hwr_status hwr_route_batch_multi(hwr_ctx *c, int32_t Q, const float *in_len,
                                            const float *out_len, const void *q_emb, float slo,
                                            const float *lambdas, int32_t K, uint32_t flags,
                                            int32_t *chosen, float *pred_latency,
                                            float *utility) {
    ApiRange range_("hwr_route_batch_multi");
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (!lambdas) return fail(c, HWR_ERR_INVALID_ARG, "lambdas is NULL");
    if (K < 1 || K > MAX_LAMBDAS)
        return fail(c, HWR_ERR_INVALID_ARG, "K=%d outside [1, %d]", K, MAX_LAMBDAS);
    Lambdas L;
    L.K = K;
    for (int k = 0; k < K; ++k) {
        if (!isfinite(lambdas[k])) return fail(c, HWR_ERR_INVALID_ARG, "lambda %d not finite", k);
        L.lam[k] = lambdas[k];
        L.wq[k] = (flags & HWR_SCORE_CONVEX) ? 1.0f - lambdas[k] : 1.0f;
    }
    return route_impl(c, Q, in_len, out_len, q_emb, slo, nullptr, lambdas[0], flags, chosen,
                      pred_latency, utility, &L);
}

extern "C" hwr_status hwr_route_batch_slo(hwr_ctx *c, int32_t Q, const float *in_len,
                                          const float *out_len, const void *q_emb,
                                          const hwr_slo_spec *slo, float lambda, uint32_t flags,
                                          int32_t *chosen, float *pred_latency, float *utility) {
    ApiRange range_("hwr_route_batch_slo");
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (!slo) return fail(c, HWR_ERR_INVALID_ARG, "slo specification is NULL");
    return route_impl(c, Q, in_len, out_len, q_emb, 0.0f, slo, lambda, flags, chosen,
                      pred_latency, utility);
}

extern "C" hwr_status hwr_synchronize(hwr_ctx *c) {
    ApiRange range_("hwr_synchronize");
    if (!c) return fail(nullptr, HWR_ERR_INVALID_ARG, "ctx is NULL");
    if (c->broken) return HWR_ERR_STATE;
    CK(c, cudaStreamSynchronize(c->stream), "synchronize");
    c->async_pending = false;
    c->snap_busy = false;
    return check_status_word(c);
}

extern "C" hwr_status hwr_get_stats(hwr_ctx *c, hwr_stats *out, int reset) {
    if (!c || !out) return fail(c, HWR_ERR_INVALID_ARG, "NULL argument");
    if (!c->broken) TRY(collect_profile(c));
    *out = c->stats;
    if (reset) {
        for (int k = 0; k < HWR_K_COUNT; ++k) {
            c->stats.profiled_ms[k] = 0;
            c->stats.profiled_launches[k] = 0;
        }
    }
    return HWR_OK;
}

extern "C" const char *hwr_status_string(hwr_status s) {
    switch (s) {
        case HWR_OK: return "ok";
        case HWR_ERR_INVALID_ARG: return "invalid argument";
        case HWR_ERR_DTYPE: return "embedding dtype does not match the predictor";
        case HWR_ERR_OOM: return "out of memory";
        case HWR_ERR_CUDA: return "CUDA error";
        case HWR_ERR_TIMEOUT: return "device-side wait timed out";
        case HWR_ERR_STATE: return "context unusable after an earlier failure";
        case HWR_ERR_UNSUPPORTED: return "unsupported by this build";
    }
    return "unknown status";
}

extern "C" const char *hwr_last_error(const hwr_ctx *c) {
    return c ? c->err.c_str() : g_create_error.c_str();
}

// ---------------------------------------------------------------------------
// Internal helpers for hwr_route_batch_noalloc (hwr_noalloc.cu): the tensor
// path with caller-provided scratch, and error reporting on a context.

hwr_status hwr_internal_fail(hwr_ctx *c, hwr_status s, const char *msg) {
    return fail(c, s, "%s", msg);
}

int hwr_internal_device(const hwr_ctx *c) { return c->device; }

hwr_status hwr_internal_route_tensor_scratch(hwr_ctx *c, int32_t Q, const float *in_len,
                                             const float *out_len, const void *q_emb, float slo,
                                             float lambda, uint32_t flags, int32_t *chosen,
                                             float *pred_latency, float *utility, float *qual,
                                             void *part, int32_t *count, int max_split) {
    if (c->broken) return HWR_ERR_STATE;
    if (!c->have_snapshot)
        return fail(c, HWR_ERR_INVALID_ARG, "route before the first hwr_update_snapshot");
    if (!c->tc_ok)
        return fail(c, HWR_ERR_UNSUPPORTED, "no tensor-core path for this context (fp32 or shape)");
    if (!in_len || !out_len || !q_emb || !chosen || !pred_latency || !utility)
        return fail(c, HWR_ERR_INVALID_ARG, "NULL input or output array");
    if (slo != slo) return fail(c, HWR_ERR_INVALID_ARG, "SLO is NaN");
    if (!isfinite(lambda)) return fail(c, HWR_ERR_INVALID_ARG, "lambda is not finite");
    if ((uintptr_t)q_emb & 15) return fail(c, HWR_ERR_INVALID_ARG, "q_emb must be 16-byte aligned");
    if (Q == 0) return HWR_OK;
    Queries q;
    q.Q = Q;
    q.emb_bf16 = 1;
    q.slo = slo;
    q.lam = lambda;
    q.wq = (flags & HWR_SCORE_CONVEX) ? 1.0f - lambda : 1.0f;
    q.in_len = in_len;
    q.out_len = out_len;
    q.emb = q_emb;
    q.chosen = chosen;
    q.lat = pred_latency;
    q.util = utility;
    const TcModel t = tc_view(c);
    const MlpSplit sp = tc_mlp_split(t, Q, max_split);
    if (sp.nsplit > 1)
        CK(c, cudaMemsetAsync(count, 0, (size_t)Q * sizeof(int32_t), c->stream), "clear counters");
    // one static quality buffer: a plain launch, ordered after the kernel before
    CK(c, launch_qual_tc(t, q, qual, c->status_d, c->stream, false, false, 0, nullptr, 0),
       "quality kernel");
    c->stats.kernel_launches++;
    c->stats.launches[HWR_K_QUAL_TC]++;
    int ctas = 0;
    CK(c, launch_mlp_tc(t, q, qual, sp, part, count, c->status_d, c->stream, nullptr, &ctas),
       "predictor kernel");
    // this predictor may still run when the next tensor-core route starts
    // early: that route checks its inputs against these outputs
    const size_t qb4 = (size_t)Q * 4;
    c->prev_out[0] = {chosen, qb4};
    c->prev_out[1] = {pred_latency, qb4};
    c->prev_out[2] = {utility, qb4};
    c->prev_out[3] = {};
    c->stats.kernel_launches++;
    c->stats.launches[HWR_K_MLP_TC]++;
    c->stats.queries_routed += Q;
    if (flags & HWR_ASYNC) {
        c->async_pending = true;
        return HWR_OK;
    }
    CK(c, cudaStreamSynchronize(c->stream), "synchronize");
    c->async_pending = false;
    CK(c, cudaGetLastError(), "kernel");
    return check_status_word(c);
}
