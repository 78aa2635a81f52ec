/*
 * CPU oracle for HW-Router route scoring.  TEST INFRASTRUCTURE ONLY: it is
 * used by tests/, by __graft_entry__.smoke() and by bench.py's CPU-baseline
 * leg, never by the library.  It shares no code with the CUDA path.
 *
 * What it computes (HW-Router, Sec. 3.1 and Sec. 3.2):
 *   for every query q and deployment d = (model M_i, GPU g_i):
 *     x      = feat(q, M_i, S_i): one-hot model id, one-hot GPU id, model size,
 *              the runtime signals of Table 2 (+ GPU utilisation), and the
 *              query features (input length, expected output length), each
 *              slot transformed (identity / log1p / log) and standardised
 *              (Sec. 3.2 "Cost Predictor", Eq. 1: concatenation of query
 *              features, one-hot ids and runtime metrics).
 *     h1     = relu(W1 x + b1), h2 = relu(W2 h1 + b2), z = W3 h2 + b3
 *              (two fully connected hidden layers with ReLU, Eq. 1)
 *     TTFT   = softplus(z0), TPOT = softplus(z1)
 *              (with three heads also N_out = softplus(z2), Eq. 1)
 *     C      = TTFT + N_out * TPOT                      (Eq. 2)
 *              N_out: the third head, or with two heads the query's given
 *              expected output length
 *     Qual   = sigmoid(emb_q . memb[:, model(d)])        (Sec. 3.2 "Quality
 *              Predictor": depends on the model only, not on the GPU)
 *     U      = w * Qual - lambda * C, w = 1 or (1 - lambda)   (Sec. 3.1, Eq. 3)
 *   chosen   = argmax_d U over deployments with C <= SLO (Eq. 3 constraint),
 *              lowest index on ties; if no deployment is feasible, the one with
 *              the smallest C (lowest index on ties).
 *   Sequential mode: queries are taken in order and each decision raises the
 *   chosen deployment's running count by one before the next query is scored.
 *
 * Readings where the paper is silent (all listed with reasons in the design
 * notes): two output heads with N_out = the query's expected output length;
 * softplus output activation; feasibility as C <= SLO; the fallback and tie
 * rules above; the feature slot layout and transforms.
 *
 * Two numeric modes:
 *   ORC_F64  all arithmetic in double; bf16/fp32 inputs widened exactly;
 *            sums taken left to right.  This is the reference value.
 *   ORC_F32  "canonical fp32": every dot product is acc = bias, then
 *            acc = fmaf(w[k], x[k], acc) for k ascending; the query features
 *            are the last two slots, so the deployment part of layer 1 is a
 *            plain prefix of the same chain.  Features, softplus and sigmoid
 *            are evaluated in double and rounded to float once.  C =
 *            fmaf(N_out, TPOT, TTFT); U = fmaf(-lambda, C, w * Qual).
 *            A GPU kernel that follows the same written order reproduces these
 *            values bit for bit, which is what makes chosen indices comparable
 *            exactly.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_F64 0
#define ORC_F32 1

typedef struct {
    int32_t M, G, D, F, H1, H2, E;
    int32_t n_heads;                    /* 2: TTFT, TPOT; 3: + N_out (Eq. 1) */
    const int32_t *dep_model, *dep_gpu; /* [D] */
    const float *log10p;                /* [M] */
    const float *W1, *b1;               /* [H1][F], [H1] */
    const float *W2, *b2;               /* [H2][H1], [H2] */
    const float *W3, *b3;               /* [n_heads][H2], [n_heads] */
    const float *mu, *sd;               /* [F] */
    const uint8_t *xform;               /* [F]: 0 identity, 1 log1p, 2 log */
    const float *memb;                  /* [E][M] */
} orc_model;

typedef struct {
    const int32_t *running, *waiting;   /* [D] */
    const float *kv, *gpu_util, *ttft, *tpot;
} orc_snapshot;

/* ---- scalar helpers ---------------------------------------------------- */

static float bf16_bits_to_float(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* softplus(z) = log(1 + e^z), written in the overflow-free form
 * max(z, 0) + log1p(e^{-|z|}) (an identity, not an approximation). */
double orc_softplus_f64(double z)
{
    return fmax(z, 0.0) + log1p(exp(-fabs(z)));
}

double orc_sigmoid_f64(double s)
{
    return 1.0 / (1.0 + exp(-s));
}

float orc_softplus_f32(float z) { return (float)orc_softplus_f64((double)z); }
float orc_sigmoid_f32(float s) { return (float)orc_sigmoid_f64((double)s); }

static double slot_transform(uint8_t code, double v)
{
    if (code == 1) return log1p(v);
    if (code == 2) return log(v);
    return v;
}

/* Raw (untransformed) value of feature slot k for query (in_len, out_len)
 * on deployment d.  Layout: [one-hot model | one-hot GPU | log10 params |
 * running | waiting | kv | gpu util | ttft | tpot | zero pad | in | out]. */
static double raw_feature(const orc_model *m, const orc_snapshot *s, int d,
                          int k, double in_len, double out_len)
{
    const int M = m->M, G = m->G, F = m->F, P = M + G;
    if (k < M) return m->dep_model[d] == k ? 1.0 : 0.0;
    if (k < P) return m->dep_gpu[d] == k - M ? 1.0 : 0.0;
    if (k == P) return (double)m->log10p[m->dep_model[d]];
    if (k == P + 1) return (double)s->running[d];
    if (k == P + 2) return (double)s->waiting[d];
    if (k == P + 3) return (double)s->kv[d];
    if (k == P + 4) return (double)s->gpu_util[d];
    if (k == P + 5) return (double)s->ttft[d];
    if (k == P + 6) return (double)s->tpot[d];
    if (k == F - 2) return in_len;
    if (k == F - 1) return out_len;
    return 0.0;
}

/* Standardised feature vector x[0..F) in double (both modes start here; the
 * fp32 mode rounds each slot to float once). */
void orc_features(const orc_model *m, const orc_snapshot *s, int d,
                  float in_len, float out_len, int mode, double *x)
{
    for (int k = 0; k < m->F; ++k) {
        double t = slot_transform(m->xform[k],
                                  raw_feature(m, s, d, k, in_len, out_len));
        double v = (t - (double)m->mu[k]) / (double)m->sd[k];
        x[k] = mode == ORC_F32 ? (double)(float)v : v;
    }
}

/* ---- predictor (Eq. 1) ------------------------------------------------- */

static void predict_f64(const orc_model *m, const double *x, double *ttft,
                        double *tpot, double *nout, double *h1, double *h2)
{
    for (int j = 0; j < m->H1; ++j) {
        double acc = m->b1[j];
        for (int k = 0; k < m->F; ++k)
            acc += (double)m->W1[(size_t)j * m->F + k] * x[k];
        h1[j] = acc > 0.0 ? acc : 0.0;
    }
    for (int i = 0; i < m->H2; ++i) {
        double acc = m->b2[i];
        for (int j = 0; j < m->H1; ++j)
            acc += (double)m->W2[(size_t)i * m->H1 + j] * h1[j];
        h2[i] = acc > 0.0 ? acc : 0.0;
    }
    double z[3] = {0.0, 0.0, 0.0};
    for (int o = 0; o < m->n_heads; ++o) {
        double acc = m->b3[o];
        for (int i = 0; i < m->H2; ++i)
            acc += (double)m->W3[(size_t)o * m->H2 + i] * h2[i];
        z[o] = acc;
    }
    *ttft = orc_softplus_f64(z[0]);
    *tpot = orc_softplus_f64(z[1]);
    *nout = m->n_heads == 3 ? orc_softplus_f64(z[2]) : 0.0;
}

static void predict_f32(const orc_model *m, const float *x, float *ttft,
                        float *tpot, float *nout, float *h1, float *h2)
{
    for (int j = 0; j < m->H1; ++j) {
        float acc = m->b1[j];
        for (int k = 0; k < m->F; ++k)
            acc = fmaf(m->W1[(size_t)j * m->F + k], x[k], acc);
        h1[j] = acc > 0.0f ? acc : 0.0f;
    }
    for (int i = 0; i < m->H2; ++i) {
        float acc = m->b2[i];
        for (int j = 0; j < m->H1; ++j)
            acc = fmaf(m->W2[(size_t)i * m->H1 + j], h1[j], acc);
        h2[i] = acc > 0.0f ? acc : 0.0f;
    }
    float z[3] = {0.0f, 0.0f, 0.0f};
    for (int o = 0; o < m->n_heads; ++o) {
        float acc = m->b3[o];
        for (int i = 0; i < m->H2; ++i)
            acc = fmaf(m->W3[(size_t)o * m->H2 + i], h2[i], acc);
        z[o] = acc;
    }
    *ttft = orc_softplus_f32(z[0]);
    *tpot = orc_softplus_f32(z[1]);
    *nout = m->n_heads == 3 ? orc_softplus_f32(z[2]) : 0.0f;
}

/* Single-evaluation entry point (used by the pins): x has F doubles (in fp32
 * mode they are taken as floats).  nout is the third head (0 with two). */
void orc_predict(const orc_model *m, const double *x, int mode, double *ttft,
                 double *tpot, double *nout)
{
    double *h = (double *)malloc(sizeof(double) * (size_t)(m->H1 + m->H2));
    if (mode == ORC_F64) {
        predict_f64(m, x, ttft, tpot, nout, h, h + m->H1);
    } else {
        float *xf = (float *)malloc(sizeof(float) * (size_t)(m->F + m->H1 + m->H2));
        float a, b, c;
        for (int k = 0; k < m->F; ++k) xf[k] = (float)x[k];
        predict_f32(m, xf, &a, &b, &c, xf + m->F, xf + m->F + m->H1);
        *ttft = a;
        *tpot = b;
        *nout = c;
        free(xf);
    }
    free(h);
}

/* ---- quality (Sec. 3.2 "Quality Predictor") ----------------------------- */

static double emb_at(const void *emb, int bf16, size_t i)
{
    return bf16 ? (double)bf16_bits_to_float(((const uint16_t *)emb)[i])
                : (double)((const float *)emb)[i];
}

/* qual[m] for one query row (E values starting at element offset `row`). */
void orc_quality(const orc_model *m, const void *emb, int emb_bf16,
                 size_t row, int mode, double *qual)
{
    for (int mi = 0; mi < m->M; ++mi) {
        if (mode == ORC_F64) {
            double s = 0.0;
            for (int k = 0; k < m->E; ++k)
                s += emb_at(emb, emb_bf16, row + k) *
                     (double)m->memb[(size_t)k * m->M + mi];
            qual[mi] = orc_sigmoid_f64(s);
        } else {
            float s = 0.0f;
            for (int k = 0; k < m->E; ++k)
                s = fmaf((float)emb_at(emb, emb_bf16, row + k),
                         m->memb[(size_t)k * m->M + mi], s);
            qual[mi] = orc_sigmoid_f32(s);
        }
    }
}

/* ---- decision maker (Eq. 3) -------------------------------------------- */

/* Feasible set: C <= slo with a defined utility.  Best feasible utility,
 * lowest index on ties; with no feasible deployment, smallest C, lowest index
 * on ties; -1 if every C is NaN.  Values are compared in the precision given
 * (fp32 mode passes float-valued doubles and compares them as floats). */
int orc_select(int D, const double *C, const double *U, double slo, int mode)
{
    int best = -1;
    for (int d = 0; d < D; ++d) {
        int feas = mode == ORC_F32 ? ((float)C[d] <= (float)slo) : (C[d] <= slo);
        if (!feas || U[d] != U[d]) continue;
        if (best < 0) { best = d; continue; }
        int better = mode == ORC_F32 ? ((float)U[d] > (float)U[best]) : (U[d] > U[best]);
        if (better) best = d;
    }
    if (best >= 0) return best;
    for (int d = 0; d < D; ++d) {
        if (C[d] != C[d]) continue;
        if (best < 0) { best = d; continue; }
        int better = mode == ORC_F32 ? ((float)C[d] < (float)C[best]) : (C[d] < C[best]);
        if (better) best = d;
    }
    return best;
}

/* ---- per-query latency budget (Sec. 4.4, Eq. 4-5) ---------------------- */

/* SLO budget of a query with p input tokens and d expected output tokens:
 * TTFT_SLO(p) = slack * (a + b p) and the request meets the SLO when its
 * latency is at most TTFT_SLO(p) + d * TPOT_SLO.  fp32 order:
 * t = fma(b, p, a); s = slack * t; B = fma(tpot_slo, d, s). */
double orc_slo_budget(float a, float b, float slack, float tpot_slo, float p, float d,
                      int mode)
{
    if (mode == ORC_F64)
        return (double)slack * ((double)a + (double)b * (double)p) +
               (double)d * (double)tpot_slo;
    float t = fmaf(b, p, a);
    float s = slack * t;
    return (double)fmaf(tpot_slo, d, s);
}

/* ---- one query against every deployment ------------------------------- */

typedef struct {
    double *x, *h, *C, *U, *qual;
    float *xf, *hf;
} orc_work;

static int work_alloc(const orc_model *m, orc_work *w)
{
    w->x = (double *)malloc(sizeof(double) * (size_t)m->F);
    w->h = (double *)malloc(sizeof(double) * (size_t)(m->H1 + m->H2));
    w->C = (double *)malloc(sizeof(double) * (size_t)m->D);
    w->U = (double *)malloc(sizeof(double) * (size_t)m->D);
    w->qual = (double *)malloc(sizeof(double) * (size_t)m->M);
    w->xf = (float *)malloc(sizeof(float) * (size_t)m->F);
    w->hf = (float *)malloc(sizeof(float) * (size_t)(m->H1 + m->H2));
    return w->x && w->h && w->C && w->U && w->qual && w->xf && w->hf;
}

static void work_free(orc_work *w)
{
    free(w->x); free(w->h); free(w->C); free(w->U); free(w->qual);
    free(w->xf); free(w->hf);
}

/* Scores of deployment d for query q into w->C[d], w->U[d]; w->qual must
 * already hold the query's quality per model. */
static void score_pair(const orc_model *m, const orc_snapshot *s, float in_len,
                       float out_len, int d, float slo_unused, float lam,
                       int convex, int mode, orc_work *w)
{
    (void)slo_unused;
    orc_features(m, s, d, in_len, out_len, mode, w->x);
    double qual = w->qual[m->dep_model[d]];
    if (mode == ORC_F64) {
        double ttft, tpot, nout;
        predict_f64(m, w->x, &ttft, &tpot, &nout, w->h, w->h + m->H1);
        /* N_out of Eq. 2: the third head's prediction, else the given length */
        double n = m->n_heads == 3 ? nout : (double)out_len;
        double C = ttft + n * tpot;
        double wq = convex ? 1.0 - (double)lam : 1.0;
        w->C[d] = C;
        w->U[d] = wq * qual - (double)lam * C;
    } else {
        float ttft, tpot, nout;
        for (int k = 0; k < m->F; ++k) w->xf[k] = (float)w->x[k];
        predict_f32(m, w->xf, &ttft, &tpot, &nout, w->hf, w->hf + m->H1);
        float n = m->n_heads == 3 ? nout : out_len;
        float C = fmaf(n, tpot, ttft);
        float wq = convex ? 1.0f - lam : 1.0f;
        w->C[d] = C;
        w->U[d] = fmaf(-lam, C, wq * (float)qual);
    }
}

static void finish_query(const orc_model *m, const orc_work *w, float slo,
                         int mode, int32_t *chosen, double *lat, double *util)
{
    int c = orc_select(m->D, w->C, w->U, (double)slo, mode);
    *chosen = c;
    *lat = c >= 0 ? w->C[c] : NAN;
    *util = c >= 0 ? w->U[c] : NAN;
}

/*
 * Route Q queries.  emb is [Q][E] (float32, or bf16 bits if emb_bf16).
 * Batch mode (sequential = 0): every query sees the snapshot as given;
 * queries are independent and split over `nthreads` OpenMP threads.
 * Sequential mode: queries in order; running_io holds the running counts
 * used for scoring and is incremented by each decision.  The snapshot's own
 * running array is not read in sequential mode.
 * Outputs: chosen[Q], lat[Q], util[Q] (double; float-valued in fp32 mode).
 * Returns 0, or -1 on allocation failure.
 */
int orc_route(const orc_model *m, const orc_snapshot *s, int32_t Q,
              const float *in_len, const float *out_len, const void *emb,
              int emb_bf16, float slo, float lam, int convex, int mode,
              int sequential, int32_t *running_io, int32_t *chosen,
              double *lat, double *util, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    if (!sequential) {
        int fail = 0;
#pragma omp parallel num_threads(nthreads) reduction(| : fail)
        {
            orc_work w;
            if (!work_alloc(m, &w)) {
                fail = 1;
            } else {
#pragma omp for schedule(dynamic, 8)
                for (int32_t q = 0; q < Q; ++q) {
                    orc_quality(m, emb, emb_bf16, (size_t)q * m->E, mode, w.qual);
                    for (int d = 0; d < m->D; ++d)
                        score_pair(m, s, in_len[q], out_len[q], d, slo, lam,
                                   convex, mode, &w);
                    finish_query(m, &w, slo, mode, &chosen[q], &lat[q], &util[q]);
                }
            }
            work_free(&w);
        }
        return fail ? -1 : 0;
    }

    /* Sequential: the deployments of one query are independent of each other,
     * so they may be scored on several threads; queries stay in order. */
    orc_snapshot cur = *s;
    cur.running = running_io;
    orc_work *ws = (orc_work *)calloc((size_t)nthreads, sizeof(orc_work));
    double *C = (double *)malloc(sizeof(double) * (size_t)m->D);
    double *U = (double *)malloc(sizeof(double) * (size_t)m->D);
    double *qual = (double *)malloc(sizeof(double) * (size_t)m->M);
    int fail = !ws || !C || !U || !qual;
    for (int t = 0; !fail && t < nthreads; ++t) fail = !work_alloc(m, &ws[t]);
    for (int32_t q = 0; !fail && q < Q; ++q) {
        orc_quality(m, emb, emb_bf16, (size_t)q * m->E, mode, qual);
#pragma omp parallel for num_threads(nthreads) schedule(static) if (nthreads > 1)
        for (int d = 0; d < m->D; ++d) {
            int t = 0;
#ifdef _OPENMP
            t = omp_get_thread_num();
#endif
            orc_work *w = &ws[t];
            memcpy(w->qual, qual, sizeof(double) * (size_t)m->M);
            score_pair(m, &cur, in_len[q], out_len[q], d, slo, lam, convex,
                       mode, w);
            C[d] = w->C[d];
            U[d] = w->U[d];
        }
        int c = orc_select(m->D, C, U, (double)slo, mode);
        chosen[q] = c;
        lat[q] = c >= 0 ? C[c] : NAN;
        util[q] = c >= 0 ? U[c] : NAN;
        if (c >= 0) running_io[c] += 1;
    }
    if (ws)
        for (int t = 0; t < nthreads; ++t) work_free(&ws[t]);
    free(ws); free(C); free(U); free(qual);
    return fail ? -1 : 0;
}

/* As orc_route in batch or sequential mode, with one SLO budget per query
 * (slo_q[Q], in the precision of the mode: float values). */
int orc_route_q(const orc_model *m, const orc_snapshot *s, int32_t Q, const float *in_len,
                const float *out_len, const void *emb, int emb_bf16, const float *slo_q,
                float lam, int convex, int mode, int sequential, int32_t *running_io,
                int32_t *chosen, double *lat, double *util, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    orc_snapshot cur = *s;
    if (sequential) cur.running = running_io;
    int fail = 0;
    orc_work w;
    if (!work_alloc(m, &w)) {
        work_free(&w);
        return -1;
    }
    for (int32_t q = 0; q < Q; ++q) {
        orc_quality(m, emb, emb_bf16, (size_t)q * m->E, mode, w.qual);
        for (int d = 0; d < m->D; ++d)
            score_pair(m, &cur, in_len[q], out_len[q], d, slo_q[q], lam, convex, mode, &w);
        finish_query(m, &w, slo_q[q], mode, &chosen[q], &lat[q], &util[q]);
        if (sequential && chosen[q] >= 0) running_io[chosen[q]] += 1;
    }
    (void)nthreads;
    work_free(&w);
    return fail ? -1 : 0;
}

/* Per-pair latency and utility for every (q, d) (used to compute top-2
 * margins in the parity tests).  C and U are [Q][D]. */
int orc_score_all(const orc_model *m, const orc_snapshot *s, int32_t Q,
                  const float *in_len, const float *out_len, const void *emb,
                  int emb_bf16, float lam, int convex, int mode, double *C,
                  double *U, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    int fail = 0;
#pragma omp parallel num_threads(nthreads) reduction(| : fail)
    {
        orc_work w;
        if (!work_alloc(m, &w)) {
            fail = 1;
        } else {
#pragma omp for schedule(dynamic, 8)
            for (int32_t q = 0; q < Q; ++q) {
                orc_quality(m, emb, emb_bf16, (size_t)q * m->E, mode, w.qual);
                for (int d = 0; d < m->D; ++d) {
                    score_pair(m, s, in_len[q], out_len[q], d, 0.0f, lam,
                               convex, mode, &w);
                    C[(size_t)q * m->D + d] = w.C[d];
                    U[(size_t)q * m->D + d] = w.U[d];
                }
            }
        }
        work_free(&w);
    }
    return fail ? -1 : 0;
}
