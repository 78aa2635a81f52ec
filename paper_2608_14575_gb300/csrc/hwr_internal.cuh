// Internal interface between the C-ABI host code (hwr_api.cu) and the CUDA
// kernels (k_simt.cu: fp32 SIMT kernels, k_tc.cu: bf16 tcgen05 kernels).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "hwr.h"

namespace hwr {

// Device status word, written by kernels whose waits are bounded.
enum : int32_t { ST_OK = 0, ST_TIMEOUT = 1, ST_BAD_LAUNCH = 2 };

constexpr int SIMT_THREADS = 256;
constexpr int SIMT_KC = 32;          // K chunk of the layer-2 tile (64 rows: 8 warps x 8)
constexpr int MAX_D = 64;
constexpr int MAX_H = 256;
constexpr int SEQ_MAX_CHUNK = 64;    // queries per sequential table
constexpr int SEQ_CHAIN_SMEM = 200 * 1024;

// Read-only device view of the predictor and deployment state.
struct Model {
    int M, G, D, F, H1, H2, E, P;
    int NH;                     // output heads: 2 (TTFT, TPOT) or 3 (+ N_out)
    const int32_t *dep_model;   // [D]
    const int32_t *dep_gpu;     // [D]
    const float *log10p;        // [M]
    const float *W1, *b1;       // [H1][F], [H1]   fp32 (bf16 widened)
    const float *W1T;           // [F][H1]: W1 transposed (slot-major, coalesced per slot)
    const float *W2, *b2;       // [H2][H1], [H2]
    const float *W2T;           // [H1][H2p]: W2 transposed, rows zero-padded to H2p
    int H2p;                    // H2 rounded up to a multiple of 4 (16-byte rows)
    const float *W3, *b3;       // [NH][H2], [NH]
    const float *mu, *sd;       // [F]
    const uint8_t *xform;       // [F]
    const float *memb;          // [E][M] fp32 (bf16 widened)
    // snapshot (SoA, [D]) and derived per-deployment state
    int32_t *running;
    const int32_t *waiting;
    const float *kv, *gpu_util, *ttft, *tpot;
    float *X;                   // [D][F] standardised deployment features
    float *Spre;                // [D][H1] layer-1 chain through slot P
    float *A;                   // [D][H1] layer-1 chain through slot F-3
    uint16_t *Abf;              // [D][H1] A rounded to bf16 (tensor-core path)
};

struct Queries {
    int Q;
    // the query inputs sit in host memory mapped into the device's address
    // space: kernels read them with plain loads only (no cp.async).  Kept in
    // the padding after Q: the struct stays 128 bytes (a larger parameter
    // block measured 2.6 % slower in the tensor-core predictor kernel)
    int inputs_host = 0;
    const float *in_len, *out_len;
    const void *emb;            // [Q][E], fp32 or bf16 bits
    int emb_bf16;
    float slo, lam, wq;         // wq = 1 or (1 - lambda)
    int32_t *chosen;
    float *lat, *util;
    // latency budget per query: 0 = the scalar slo, 1 = slo_q[q],
    // 2 = the SLO model of Eq. 4-5 from the query's lengths
    int slo_mode = 0;
    const float *slo_q = nullptr;
    float slo_a = 0.f, slo_b = 0.f, slo_slack = 1.f, slo_tpot = 0.f;
    // when set, kernels also store every pair's cost C [Q][D] and (SIMT fused
    // kernel) every query's quality [Q][M] for a later multi-lambda selection
    float *pair_C = nullptr;
    float *qual_out = nullptr;
    // when set, the tensor-core predictor kernel only stores pair_C (no
    // decision outputs, no partial results)
    int no_select = 0;
    // sequential table on the tensor cores: when > 0, deployment v of the
    // predictor is (deployment v / (seq_n + 1), count v % (seq_n + 1)) and
    // pair_C is the triangular sequential table of seq_n queries (tab_row)
    int seq_n = 0;
};
static_assert(sizeof(Queries) == 128, "Queries: a larger parameter block slows k_mlp_tc");

// The sequential score table of a chunk of Qs queries over D deployments:
// entry (picks so far c, deployment d, query i >= c) sits at
//   D * (c * Qs - c (c - 1) / 2) + d * (Qs - c) + (i - c);
// tri_off(c) is the offset of count c's block, tab_row(c, d) + i the entry.
__host__ __device__ inline size_t tri_off(int D, int Qs, int c) {
    return (size_t)D * ((size_t)c * Qs - (size_t)c * (c - 1) / 2);
}
__host__ __device__ __forceinline__ int tab_row(int D, int Qs, int c, int d) {
    return D * (c * Qs - (c * (c - 1)) / 2) + d * (Qs - c) - c;
}

// Several values of lambda applied to one set of scores.
constexpr int MAX_LAMBDAS = 16;
struct Lambdas {
    int K;
    float lam[MAX_LAMBDAS], wq[MAX_LAMBDAS];
};

#ifdef __CUDACC__
// Budget B of query `row` (Sec. 4.4, Eq. 4-5 for the model form):
// t = fma(b, p, a); s = slack * t; B = fma(tpot_slo, d, s).
__device__ __forceinline__ float query_budget(const Queries &q, int row) {
    if (q.slo_mode == 1) return q.slo_q[row];
    if (q.slo_mode == 2) {
        const float t = __fmaf_rn(q.slo_b, q.in_len[row], q.slo_a);
        return __fmaf_rn(q.slo_tpot, q.out_len[row], __fmul_rn(q.slo_slack, t));
    }
    return q.slo;
}
#endif

// ---- SIMT kernels (k_simt.cu) -------------------------------------------
// The snapshot signals are read from `stage` ([6][D] 4-byte values in host
// memory mapped into the device's address space, in the order running,
// waiting, kv, gpu_util, ttft, tpot) into the six device arrays, which m.running
// starts (they are contiguous, in that order).
cudaError_t launch_snapshot(const Model &m, const uint32_t *stage, cudaStream_t s);
// Fused gather -> MLP -> mask -> argmax for a batch.
cudaError_t launch_route_simt(const Model &m, const Queries &q, cudaStream_t s);
// Small-batch (latency) variant: groups of (query, deployment) pairs with
// layer 2 split by columns over several blocks, plus quality blocks; scratch
// pairC [Q][D], qualS [Q][M], h2 [Q D][H2], count [2 PAIRS_MAX_PAIRS] (query
// and group arrivals; zeroed once, self-resetting).  Q * D <= PAIRS_MAX_PAIRS.
// Reads W2 through m.W2T and layer 1's query columns through m.W1T.
constexpr int PAIRS_MAX_PAIRS = 2048;   // default upper bound on Q * D for this kernel
cudaError_t launch_route_pairs(const Model &m, const Queries &q, float *pairC, float *qualS,
                               float *h2, int32_t *count, int nsm, cudaStream_t s);
size_t route_pairs_smem(const Model &m);
// Sequential mode over one chunk of Qs <= seq_chunk(m) queries: the chunk's
// standardised features and layer-1 prefixes, and the score table (every
// (picks c, deployment d, query i >= c)) in launch_seq_table (two kernels),
// then the serial chain.
//   ctab: scratch of seq_table_floats(D, Qs) floats;
//   aux: scratch of seq_aux_floats(D, M, H1, Qs) floats;
//   slots: table blocks resident on the whole GPU at once (seq_table_slots).
cudaError_t launch_seq_table(const Model &m, const Queries &q, int Qs, int slots,
                             float *ctab, float *aux, cudaStream_t s);
cudaError_t launch_seq_chain(const Model &m, const Queries &q, int Qs,
                             const float *ctab, float *aux, cudaStream_t s);
size_t seq_aux_floats(int D, int M, int H1, int Qs);
// Sequential mode with the table on the tensor cores (bf16 contexts): the
// preparation kernel alone, also writing bf16 prefixes pre_bf [D (Qs + 1)][H1]
// and the model of each (deployment, count) group dmv [D (Qs + 1)] (group
// d (Qs + 1) + c); the chain over the triangular table ctab (written by the
// predictor kernel with q.seq_n = Qs) with quality rows qual [Qs][qstride].
cudaError_t launch_seq_prep_tc(const Model &m, const Queries &q, int Qs, float *aux,
                               uint16_t *pre_bf, int32_t *dmv, cudaStream_t s);
cudaError_t launch_seq_chain_tc(const Model &m, const Queries &q, int Qs, const float *ctab,
                                float *aux, const float *qual, int qstride, cudaStream_t s);
int seq_table_slots(const Model &m);
// Decision maker for K lambdas from stored scores: C [Q][D], quality
// qual[q * qstride + model]; outputs [K][ostride] starting at query 0.
cudaError_t launch_select_multi(const Model &m, const Queries &q, const float *C,
                                const float *qual, int qstride, const Lambdas &L, int ostride,
                                cudaStream_t s);
int seq_chunk(const Model &m);
size_t seq_table_floats(int D, int Qs);
size_t route_simt_smem(const Model &m);
size_t seq_table_smem(const Model &m);
cudaError_t simt_prepare();   // one-time smem opt-in

// ---- tcgen05 kernels (k_tc.cu) -------------------------------------------
struct HeadConsts;
struct TcModel {
    int M, Mpad, D, H1, H2, E, Epad, NH;
    const HeadConsts *head;     // host copy of b2, W3, b3 (kernel parameters)
    const uint16_t *W2img;      // bf16 W2 in the UMMA shared-memory image
    const uint16_t *membimg;    // bf16 memb^T in the UMMA shared-memory image
    const uint16_t *Abf;        // [D][H1] bf16 deployment prefix of layer 1
    const float *W1q;           // [2][H1]: W1 columns of the two query slots
    const float *b2, *W3, *b3;  // fp32
    const int32_t *dep_model;
    float mu_in, sd_in, mu_out, sd_out;
    uint8_t xf_in, xf_out;
    int test_stall;             // test hook: producers never signal (bounded waits expire)
};
bool tc_supported(int M, int H1, int H2, int E);
size_t tc_w2img_elems(int H1, int H2);
size_t tc_membimg_elems(int Mpad, int Epad);
// Host-side construction of the shared-memory images (bf16 bits in/out).
void tc_build_w2img(const uint16_t *W2, int H1, int H2, uint16_t *img);
void tc_build_membimg(const uint16_t *memb_EM, int E, int M, int Mpad, int Epad,
                      uint16_t *img);
// qual: scratch [Q][Mpad] fp32.  status: device int32 word.
// dependent: launched as a programmatic dependent of the kernel before it on
// the stream, running alongside it -- only when that kernel does not read
// `qual` (the context alternates two quality buffers between calls).
// early: its dependent may be scheduled as soon as the grid has started (only
// when the kernel before does not let its own dependents start early with
// results the predictor reads before its dependency wait, and this call's
// inputs are not the previous call's outputs); free_sms: SMs the predictor
// after it leaves free (a small batch is spread over those alone).
// done, done_target: the predictors' completion counter; before its first
// store the grid waits for it to reach done_target (nullptr: no wait).
cudaError_t launch_qual_tc(const TcModel &m, const Queries &q, float *qual,
                           int32_t *status, cudaStream_t s, bool dependent, bool early,
                           int free_sms, const uint32_t *done, uint32_t done_target);
// The first nwhole query tiles are processed whole; the deployments of each
// remaining tile are split over nsplit units.  With nsplit > 1, `part`
// (nsplit * Q records of 16 bytes) and `count` (Q int32, zero, self-resetting)
// are scratch.
struct MlpSplit {
    int nwhole, nsplit;
};
MlpSplit tc_mlp_split(const TcModel &m, int Q, int max_split = 8);
// SMs the predictor kernel for Q queries split as sp leaves free (0 if none).
int tc_mlp_free_sms(int Q, const MlpSplit &sp);
// done: completion counter every CTA increments (release) as it finishes
// (nullptr: none); *ctas: the CTAs launched (0 on failure).
cudaError_t launch_mlp_tc(const TcModel &m, const Queries &q, const float *qual,
                          const MlpSplit &sp, void *part, int32_t *count, int32_t *status,
                          cudaStream_t s, uint32_t *done, int *ctas);
cudaError_t tc_prepare();
// Costs of every (query, deployment) pair of at most 128 queries into
// q.pair_C [Q][m.D] (q.no_select set), the deployments spread over the SMs.
cudaError_t launch_mlp_tc_scores(const TcModel &m, const Queries &q, const float *qual,
                                 int32_t *status, cudaStream_t s, uint32_t *done, int *ctas);
size_t tc_head_consts_bytes();
void tc_fill_head_consts(void *dst, const float *b2, const float *W3, const float *b3, int H2,
                         int NH);

}  // namespace hwr
