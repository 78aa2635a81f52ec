/*
 * hwr.h -- C ABI of the GB300 (sm_103a) route-scoring library for HW-Router
 * (hardware-aware routing for multi-LLM serving).
 *
 * The router's decision problem (HW-Router Sec. 3.1): a set of deployments
 * (M_i, g_i) -- one LLM on one GPU type -- and a stream of queries x; pick for
 * each query the deployment that maximises a quality/cost trade-off.  Per
 * (query, deployment) pair the library
 *   1. assembles feat(x, M_i, S_i): one-hot model and GPU ids, model size,
 *      the runtime signals S_i of Table 2 (running and waiting queue lengths,
 *      KV-cache usage, recent TTFT and TPOT) plus GPU utilisation, and the
 *      query's input length and expected output length (Sec. 3.2, Eq. 1);
 *   2. runs the latency predictor f_cost -- two fully connected hidden layers
 *      with ReLU and two softplus heads, TTFT and TPOT (Eq. 1);
 *   3. forms the cost C = TTFT + N_out * TPOT with N_out the query's expected
 *      output length (Eq. 2);
 *   4. scores quality Q = sigmoid(query embedding . model embedding), which
 *      depends on the model only (Sec. 3.2, "Quality Predictor");
 *   5. masks deployments with C > SLO and takes the argmax of
 *      U = Q - lambda * C (or the paper's (1 - lambda) Q - lambda C with
 *      HWR_SCORE_CONVEX) per query (Sec. 3.1; Eq. 3).
 *
 * Selection rule (Eq. 3 plus the readings where the paper is silent): feasible
 * means C <= SLO; among feasible deployments the largest U wins, lowest index
 * on ties; if none is feasible, the smallest C wins, lowest index on ties.
 * chosen = -1 only if every cost of the query is NaN.
 *
 * Feature slot layout (F slots, P = M + G):
 *   [0, M) one-hot model | [M, P) one-hot GPU type | P log10(params) |
 *   P+1 running | P+2 waiting | P+3 KV util | P+4 GPU util | P+5 recent TTFT |
 *   P+6 recent TPOT | P+7 .. F-3 zero padding | F-2 input length |
 *   F-1 expected output length.
 * Each slot k is transformed by feat_xform[k] (0 identity, 1 log1p, 2 log)
 * and standardised as (t - feat_mean[k]) / feat_std[k].  Requires F >= P + 9.
 *
 * Conventions for every call
 *   - Status codes are returned, never signalled; nothing aborts the process.
 *   - The context is bound to one CUDA stream (given at create; NULL means the
 *     library creates its own non-blocking stream) and every device operation
 *     of the context is ordered on it.  A context is not thread-safe.
 *   - create / update_snapshot copy what they are given: the caller keeps
 *     ownership of every pointer passed in.  Outputs belong to the caller.
 *   - After HWR_ERR_CUDA or HWR_ERR_TIMEOUT the context is broken: every later
 *     call except hwr_destroy returns HWR_ERR_STATE.  After HWR_ERR_INVALID_ARG,
 *     HWR_ERR_DTYPE or HWR_ERR_UNSUPPORTED the context is unchanged and usable.
 *   - hwr_last_error() gives a one-line description of the last failure.
 */
#ifndef HWR_H
#define HWR_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    HWR_OK = 0,
    HWR_ERR_INVALID_ARG = 1, /* NULL pointer, bad size or value */
    HWR_ERR_DTYPE = 2,       /* embedding dtype does not match the predictor */
    HWR_ERR_OOM = 3,         /* a device or pinned-host allocation failed */
    HWR_ERR_CUDA = 4,        /* a CUDA call or kernel failed */
    HWR_ERR_TIMEOUT = 5,     /* a device-side wait gave up (bounded spin) */
    HWR_ERR_STATE = 6,       /* context unusable after an earlier failure */
    HWR_ERR_UNSUPPORTED = 7  /* valid request outside this build's limits */
} hwr_status;

typedef enum { HWR_F32 = 0, HWR_BF16 = 1 } hwr_dtype;

/* Flags of hwr_route_batch. */
#define HWR_SEQUENTIAL   (1u << 0) /* in-batch queue update, see route_batch */
#define HWR_DEVICE_PTRS  (1u << 1) /* inputs and outputs are device pointers */
#define HWR_ASYNC        (1u << 2) /* return without synchronising the stream */
#define HWR_SCORE_CONVEX (1u << 3) /* U = (1 - lambda) Q - lambda C (Sec. 3.1) */
#define HWR_PATH_SIMT    (1u << 4) /* force the fp32 SIMT kernels */
#define HWR_PATH_TENSOR  (1u << 5) /* force the tcgen05 kernels (bf16 only) */
#define HWR_PROFILE      (1u << 6) /* time each kernel with CUDA events */

typedef struct hwr_ctx hwr_ctx;

/* Static deployment table (Sec. 3.1: the set of model-GPU pairs).
 * Deployment d runs model dep_model[d] in [0, n_models) on GPU type
 * dep_gpu[d] in [0, n_gpu_types).  model_log10_params[m] is the model size
 * feature.  All arrays are host memory. */
typedef struct {
    int32_t n_models, n_gpu_types, n_deployments;
    const int32_t *dep_model;          /* [D] */
    const int32_t *dep_gpu;            /* [D] */
    const float *model_log10_params;   /* [M] */
} hwr_deployment_table;

/* Latency predictor f_cost (Eq. 1): F -> H1 -> H2 -> NH with ReLU after
 * both hidden layers and softplus on the outputs: TTFT, TPOT and, with three
 * heads, the predicted output length N_out.  The cost of Eq. 2 uses N_out from
 * the third head when there is one, else the query's given expected output
 * length.  Weights are row-major [out][in] in `dtype` (fp32, or bf16 bit
 * patterns as uint16): W1 [H1][F], W2 [H2][H1], W3 [NH][H2].  Biases and
 * standardisation are fp32.  All arrays are host memory. */
typedef struct {
    int32_t F, H1, H2;
    hwr_dtype dtype;
    const void *W1, *W2, *W3;
    const float *b1, *b2, *b3;         /* [H1], [H2], [NH] */
    const float *feat_mean, *feat_std; /* [F]; feat_std must be non-zero */
    const uint8_t *feat_xform;         /* [F]: 0 identity, 1 log1p, 2 log */
    int32_t n_heads;                   /* NH: 2 (or 0, meaning 2) or 3 */
} hwr_predictor;

/* Runtime signals S_i of one snapshot (Table 2, plus GPU utilisation), one
 * entry per deployment, host memory.  Times in seconds, utilisations in
 * [0, 1]. */
typedef struct {
    const int32_t *running, *waiting;  /* [D] */
    const float *kv_util, *gpu_util;   /* [D] */
    const float *ttft_avg, *tpot_avg;  /* [D] */
} hwr_snapshot;

/*
 * Create a routing context: the router's static problem of Sec. 3.1 -- the
 * deployment set (M_i, g_i) -- with the cost predictor f_cost of Sec. 3.2 (2)
 * (Eq. 1) and the model embeddings of the quality predictor, Sec. 3.2 (3).
 *   table, pred   host structs as above (copied).
 *   model_emb     host [E][n_models] model embedding matrix (copied), in
 *                 emb_dtype.  Quality of model m for query q is
 *                 sigmoid(sum_k q_emb[q][k] * model_emb[k][m]).
 *   E             embedding width; E % 8 == 0, 8 <= E <= 8192.
 *   emb_dtype     must equal pred->dtype (else HWR_ERR_DTYPE): fp32 contexts
 *                 take fp32 query embeddings, bf16 contexts bf16.
 *   cuda_stream   cudaStream_t to order all work on, or NULL.
 *   out           receives the context; set to NULL on failure.
 * Limits (HWR_ERR_UNSUPPORTED beyond them): 1 <= D <= 64; M <= 32 (bf16) or
 * M <= 64 (fp32); H1, H2 in [1, 256]; F <= 256.  The bf16 tensor-core path
 * further needs H1 % 64 == 0 and H2 % 16 == 0 (else the SIMT kernels run).
 * The context holds no snapshot until hwr_update_snapshot is called.  The
 * CUDA device current at this call is the context's device: every later call
 * on the context must be made with it current.
 * Errors: INVALID_ARG, DTYPE, UNSUPPORTED, OOM, CUDA (also: no CUDA device).
 */
hwr_status hwr_create(const hwr_deployment_table *table,
                      const hwr_predictor *pred, const void *model_emb,
                      int32_t E, hwr_dtype emb_dtype, void *cuda_stream,
                      hwr_ctx **out);

/*
 * Replace the hardware snapshot (the hardware monitor's cache, Sec. 3.2 (1)).
 * Copies D entries of every array host -> device and recomputes the
 * deployment part of the predictor's first layer on the device.  Ordered on
 * the context stream; returns once the host arrays may be reused.
 * Every value must lie in the domain of its feature's transform: running and
 * waiting >= 0; every float finite; > 0 where the slot's feat_xform is log,
 * > -1 where it is log1p.  A snapshot with any other value is rejected
 * (INVALID_ARG, the context keeps its previous snapshot): such a value would
 * turn the deployment's features, and so its cost, into NaN.
 * Errors: INVALID_ARG (NULL array or a value outside its domain), STATE, CUDA.
 */
hwr_status hwr_update_snapshot(hwr_ctx *ctx, const hwr_snapshot *snap);

/*
 * Copy the context's current running counts (D int32, host memory): the
 * running-queue signal of the cached monitor view (Sec. 3.2 (1), Table 2),
 * including the increments made by HWR_SEQUENTIAL routing.  Synchronises the
 * context stream.  Errors: INVALID_ARG, STATE, CUDA.
 */
hwr_status hwr_get_snapshot(hwr_ctx *ctx, int32_t *running_out);

/*
 * Route Q queries (Q >= 0; Q = 0 is a no-op).
 *   in_len[Q], out_len[Q]  fp32 input length and expected output length
 *                          (N_out of Eq. 2) in tokens.
 *   q_emb                  [Q][E] query embeddings, dtype of the context.
 *   slo                    latency budget B in seconds (Eq. 3); +inf allowed,
 *                          NaN rejected.
 *   lambda                 cost weight; finite.
 *   flags                  HWR_* flags above.
 *   chosen[Q]              chosen deployment index (int32).
 *   pred_latency[Q]        predicted cost C of the chosen deployment (s).
 *   utility[Q]             utility U of the chosen deployment.
 * Without HWR_DEVICE_PTRS all six arrays are host memory; the call copies the
 * inputs host -> device and the outputs back, and (without HWR_ASYNC)
 * returns after the results are in place (small batches on the small-batch
 * kernel, and small HWR_SEQUENTIAL batches on the SIMT kernels, return as
 * soon as every output is written, possibly before the kernel's last blocks
 * retire -- the sequential chain then still persists the picks, which later
 * work on the context is ordered after; a failure after that point is
 * reported by the next call on the context or by hwr_synchronize.  When earlier work is still
 * queued on the stream -- after an HWR_ASYNC call, or the caller's own work on
 * a stream it passed to hwr_create -- the call synchronises the stream
 * instead of waiting on the outputs).  Where the GPU can read and write
 * pageable host memory (cudaDevAttrPageableMemoryAccess, e.g. Grace + GB300
 * over the coherent CPU-GPU link), such small synchronous calls use the
 * caller's arrays directly: the kernels read the inputs and write the outputs
 * there, so the arrays must stay untouched until the call returns.  Pinned
 * host memory gives the full
 * link bandwidth.  With HWR_DEVICE_PTRS they are device pointers read and
 * written in stream order.  With HWR_ASYNC the call returns after enqueueing;
 * host arrays must then stay valid until hwr_synchronize().
 * HWR_SEQUENTIAL: queries are routed in index order and each decision
 * increments its deployment's running count before the next query is scored;
 * the increments persist in the context until the next update_snapshot.  By
 * default the scores follow the canonical fp32 order (SIMT kernels, also in
 * bf16 contexts); with HWR_PATH_TENSOR as well (bf16 contexts) the score
 * table is computed on the tensor cores (bf16 operands, fp32 accumulation:
 * the tensor path's tolerance, and a near tie may then be decided the other
 * way, which changes the later counts).
 * Routing before the first hwr_update_snapshot is rejected (INVALID_ARG).
 * Errors: INVALID_ARG, UNSUPPORTED (e.g. HWR_PATH_TENSOR on an fp32 context),
 * STATE, OOM, CUDA, TIMEOUT.
 */
hwr_status hwr_route_batch(hwr_ctx *ctx, int32_t Q, const float *in_len,
                           const float *out_len, const void *q_emb, float slo,
                           float lambda, uint32_t flags, int32_t *chosen,
                           float *pred_latency, float *utility);

/*
 * Per-query latency budgets (HW-Router Sec. 4.4, Eq. 4-5).  The paper's SLO
 * for a request with p input tokens and d output tokens is
 * TTFT_SLO(p) + d * TPOT_SLO with TTFT_SLO(p) = slack * (a + b p); routing
 * uses the query's expected output length for d.
 *   budget   [Q] budget per query in seconds (host or device memory, as the
 *            other arrays of the call), or NULL to use the model below;
 *   ttft_a, ttft_b, slack, tpot   the model (finite) when budget is NULL;
 *            evaluated per query on the device in fp32 as
 *            t = fma(b, p, a); s = slack * t; B = fma(tpot, d, s).
 * A NaN budget makes every deployment of that query infeasible.
 */
typedef struct {
    const float *budget;
    float ttft_a, ttft_b, slack, tpot;
} hwr_slo_spec;

/*
 * As hwr_route_batch, with the SLO budget B of Eq. 3 given per query by
 * `slo` instead of one scalar for the batch (all flags and paths apply).
 * Errors: as hwr_route_batch; INVALID_ARG also for a NULL spec or
 * non-finite model parameters.
 */
hwr_status hwr_route_batch_slo(hwr_ctx *ctx, int32_t Q, const float *in_len,
                               const float *out_len, const void *q_emb,
                               const hwr_slo_spec *slo, float lambda,
                               uint32_t flags, int32_t *chosen,
                               float *pred_latency, float *utility);

/*
 * Score one batch without deciding: the cost predictor's C = TTFT + N_out *
 * TPOT (Eq. 1-2) for every (query, deployment) pair and the quality score of
 * every (query, model) pair (Sec. 3.2 (3)), under the current snapshot.
 *   cost     [Q][D] row-major, or NULL;
 *   quality  [Q][M] row-major, or NULL (not both NULL).
 * Host or device memory per HWR_DEVICE_PTRS.  Values are those the routing
 * calls compare: bit-identical to what a route of the same batch on the same
 * path computes for each pair.  HWR_SCORE_CONVEX is ignored; HWR_SEQUENTIAL
 * is UNSUPPORTED.  Errors: as hwr_route_batch.
 */
hwr_status hwr_score_batch(hwr_ctx *ctx, int32_t Q, const float *in_len,
                           const float *out_len, const void *q_emb,
                           uint32_t flags, float *cost, float *quality);

/*
 * Route one batch for K values of lambda at once (1 <= K <= 16): the
 * predictor and the quality scores are evaluated once and the decision maker
 * of Eq. 3 is applied for every lambda -- the routing half of the paper's
 * quality-latency Pareto sweep over lambda (Sec. 5, RQ1).
 *   lambdas     [K] host array of finite values;
 *   chosen, pred_latency, utility   [K][Q]: row k holds the results for
 *               lambdas[k] (host or device memory per HWR_DEVICE_PTRS).
 * Each row equals what hwr_route_batch returns for that lambda.  Flags as for
 * hwr_route_batch except HWR_SEQUENTIAL (UNSUPPORTED).
 * Errors: as hwr_route_batch; INVALID_ARG for K out of range or a
 * non-finite lambda.
 */
hwr_status hwr_route_batch_multi(hwr_ctx *ctx, int32_t Q, const float *in_len,
                                 const float *out_len, const void *q_emb,
                                 float slo, const float *lambdas, int32_t K,
                                 uint32_t flags, int32_t *chosen,
                                 float *pred_latency, float *utility);

/*
 * Route a batch without allocating anything at call time.
 *
 * The paper has no counterpart to this call; it exists for callers that
 * cannot allocate GPU memory while they route -- for example a router that
 * lives inside an LLM serving process whose engine reserved nearly all of the
 * GPU's memory up front for its KV cache, or a latency-critical serving loop
 * that must not take the device-wide synchronisation of cudaMalloc.
 * hwr_route_batch may grow its scratch with cudaMalloc; this call never does:
 * it calls no cudaMalloc, cudaFree or other allocating routine and uses one
 * fixed scratch array (about 6.1 MiB) that the library reserves in device
 * memory on every GPU where it is loaded, for as long as the process runs.
 *
 * Same arguments and outputs as hwr_route_batch, with these restrictions:
 *   - the context must be bf16 with tensor-core support (else UNSUPPORTED);
 *   - 0 <= Q <= HWR_NOALLOC_MAX_Q (larger Q: HWR_ERR_UNSUPPORTED);
 *   - all six arrays are device pointers (HWR_DEVICE_PTRS is implied);
 *     q_emb must be 16-byte aligned;
 *   - flags may hold only HWR_DEVICE_PTRS, HWR_ASYNC and HWR_SCORE_CONVEX.
 * The current device must be the context's device.  The first call on a
 * device looks up the scratch array's device address (once per device); make
 * that first call before any stream capture begins.  The scratch is shared by
 * all calls on a device and keeps the last call's contents (the parts that
 * must start at zero are cleared on every call): calls whose work overlaps on
 * the GPU -- different streams, contexts or threads -- race on it and must be
 * ordered by the caller.  Synchronises the context stream unless HWR_ASYNC.
 * Errors: INVALID_ARG, UNSUPPORTED, STATE, CUDA, TIMEOUT.
 */
#define HWR_NOALLOC_MAX_Q 32768
hwr_status hwr_route_batch_noalloc(hwr_ctx *ctx, int32_t Q, const float *in_len,
                                   const float *out_len, const void *q_emb,
                                   float slo, float lambda, uint32_t flags,
                                   int32_t *chosen, float *pred_latency,
                                   float *utility);

/* Wait for all work of the context; reports device-side timeouts
 * (HWR_ERR_TIMEOUT) and asynchronous kernel failures (HWR_ERR_CUDA). */
hwr_status hwr_synchronize(hwr_ctx *ctx);

/* Free every resource of the context (synchronises its stream first).
 * NULL is accepted.  Always valid, also on a broken context. */
hwr_status hwr_destroy(hwr_ctx *ctx);

/* Static description of a status code; never NULL. */
const char *hwr_status_string(hwr_status s);

/* One-line description of the last failure on this context (or of the last
 * failed hwr_create when ctx is NULL); empty string if none. */
const char *hwr_last_error(const hwr_ctx *ctx);

/* Counters since create: queries routed, kernels launched, and per-kernel
 * totals from HWR_PROFILE calls.  Kernel ids: */
enum {
    HWR_K_SNAPSHOT = 0, /* deployment features + first-layer prefix */
    HWR_K_ROUTE_SIMT,   /* fused fp32 gather -> MLP -> mask -> argmax */
    HWR_K_SEQ_TABLE,    /* sequential mode: feature prep + score table + serial chain */
    HWR_K_QUAL_TC,      /* bf16 quality contraction, TMA + tcgen05 */
    HWR_K_MLP_TC,       /* bf16 predictor + mask + argmax, tcgen05 */
    HWR_K_COUNT
};
typedef struct {
    int64_t queries_routed;
    int64_t kernel_launches;             /* all kernels, all calls */
    int64_t launches[HWR_K_COUNT];       /* per kernel, all calls */
    int64_t profiled_launches[HWR_K_COUNT];
    double profiled_ms[HWR_K_COUNT];     /* summed CUDA-event durations */
} hwr_stats;

/* Fill *out (synchronises the stream to read pending profile events).
 * reset != 0 zeroes the profile sums afterwards. */
hwr_status hwr_get_stats(hwr_ctx *ctx, hwr_stats *out, int reset);

#ifdef __cplusplus
}
#endif

#endif /* HWR_H */
