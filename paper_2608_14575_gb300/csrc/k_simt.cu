// fp32 SIMT kernels of the route-scoring path, in "canonical order".
//
// Canonical order (the fp32 evaluation order this library guarantees, so
// that the same scores come out bit for bit on every run and agree with any
// other implementation that follows the same written order):
//   * feature slot k:  x = (float)((t(raw) - mu[k]) / sd[k]) with the slot
//     transform t (identity, log1p, log) and the arithmetic in double;
//   * every dot product starts from its bias (0 for the quality score) and
//     accumulates acc = fma(w[k], x[k], acc) for k ascending, one rounding per
//     step; the two query slots are the last two features, so the
//     deployment-only part of layer 1 is a prefix of the same chain and is
//     computed once per snapshot;
//   * ReLU is (acc > 0 ? acc : 0);
//   * softplus(z) = max(z, 0) + log1p(exp(-|z|)) and sigmoid(s) =
//     1 / (1 + exp(-s)) in double, rounded to float once;
//   * C = fma(N_out, TPOT, TTFT);  U = fma(-lambda, C, w * Qual).
// This file is compiled with --fmad=false so no other contraction happens.
//
// Method (HW-Router Sec. 3.2): feature assembly and the latency predictor
// (Eq. 1), cost (Eq. 2), hardware-independent quality, and the decision maker
// with its SLO constraint (Eq. 3).
#include <cuda_bf16.h>
#include <math.h>

#include "hwr_internal.cuh"
#include "select.cuh"

namespace hwr {

// ---------------------------------------------------------------------------
// scalar pieces

__device__ __forceinline__ float standardise(uint8_t code, double raw, float mu,
                                             float sd) {
    double t = raw;
    if (code == 1) t = log1p(raw);
    else if (code == 2) t = log(raw);
    return (float)((t - (double)mu) / (double)sd);
}

__device__ __forceinline__ float softplus_c(float z) {
    double zd = (double)z;
    return (float)(fmax(zd, 0.0) + log1p(exp(-fabs(zd))));
}

__device__ __forceinline__ float sigmoid_c(float s) {
    return (float)(1.0 / (1.0 + exp(-(double)s)));
}

// Raw value of deployment feature slot k < F - 2 (layout in hwr.h).
__device__ double deployment_raw(const Model &m, int d, int k, int32_t running) {
    const int M = m.M, P = m.P;
    if (k < M) return m.dep_model[d] == k ? 1.0 : 0.0;
    if (k < P) return m.dep_gpu[d] == k - M ? 1.0 : 0.0;
    if (k == P) return (double)m.log10p[m.dep_model[d]];
    if (k == P + 1) return (double)running;
    if (k == P + 2) return (double)m.waiting[d];
    if (k == P + 3) return (double)m.kv[d];
    if (k == P + 4) return (double)m.gpu_util[d];
    if (k == P + 5) return (double)m.ttft[d];
    if (k == P + 6) return (double)m.tpot[d];
    return 0.0;
}

__device__ __forceinline__ float emb_at(const void *emb, int bf16, size_t i) {
    if (bf16) {
        uint32_t u = (uint32_t)((const uint16_t *)emb)[i] << 16;
        return __uint_as_float(u);
    }
    return ((const float *)emb)[i];
}

// ---------------------------------------------------------------------------
// K_snap: standardised deployment features and the deployment prefix of
// layer 1 (the part of W1 x + b1 that does not depend on the query).

__global__ void __launch_bounds__(SIMT_THREADS) k_snapshot(Model m) {
    extern __shared__ float xs[];
    const int d = blockIdx.x;
    for (int k = threadIdx.x; k < m.F - 2; k += blockDim.x) {
        float x = standardise(m.xform[k], deployment_raw(m, d, k, m.running[d]),
                              m.mu[k], m.sd[k]);
        xs[k] = x;
        m.X[(size_t)d * m.F + k] = x;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < m.H1; j += blockDim.x) {
        const float *w = m.W1 + (size_t)j * m.F;
        float acc = m.b1[j];
        int k = 0;
        for (; k <= m.P; ++k) acc = __fmaf_rn(w[k], xs[k], acc);
        m.Spre[(size_t)d * m.H1 + j] = acc;
        for (; k < m.F - 2; ++k) acc = __fmaf_rn(w[k], xs[k], acc);
        m.A[(size_t)d * m.H1 + j] = acc;
        m.Abf[(size_t)d * m.H1 + j] = __bfloat16_as_ushort(__float2bfloat16_rn(acc));
    }
}

// ---------------------------------------------------------------------------
// The shared SIMT tile: rows are (query, deployment) pairs.  For every row it
// completes layer 1 from a deployment prefix and the two query features,
// runs layer 2 (register-tiled, K ascending in chunks of SIMT_KC), layer 3
// and the softplus heads.  Output: sp[NH r + 0] = TTFT, sp[NH r + 1] = TPOT
// and, with three heads, sp[NH r + 2] = N_out.
//
// Thread map: warp w owns rows w + 8 i (i < RPT); lane l owns columns
// l + 32 j (j < CPT).  Shared memory: h1 [8 RPT][KC + 1] and W2 chunk
// [KC][H2 + 1] during the K loop, then h2 [8 RPT][H2 + 1] in the same space.

template <int RPT>
__host__ __device__ constexpr size_t tile_floats_for(int H2) {
    return (size_t)8 * RPT * (SIMT_KC + 1) + (size_t)SIMT_KC * (H2 + 1) >
                   (size_t)8 * RPT * (H2 + 1)
               ? (size_t)8 * RPT * (SIMT_KC + 1) + (size_t)SIMT_KC * (H2 + 1)
               : (size_t)8 * RPT * (H2 + 1);
}

template <int RPT, int CPT, class Rows>
__device__ void pair_mlp(const Model &m, int R, const Rows &rows, const float *us,
                         const float *vs, float *tile, float *sp) {
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int H1 = m.H1, H2 = m.H2, F = m.F;
    float *h1s = tile;
    float *w2s = tile + 8 * RPT * (SIMT_KC + 1);
    const int w2ld = H2 + 1;

    float acc[RPT][CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        const int n = lane + 32 * j;
        const float b = n < H2 ? m.b2[n] : 0.f;
#pragma unroll
        for (int i = 0; i < RPT; ++i) acc[i][j] = b;
    }

    for (int k0 = 0; k0 < H1; k0 += SIMT_KC) {
        const int kc = min(SIMT_KC, H1 - k0);
        // layer 1, query suffix: h1 = relu(fma(w_out, v, fma(w_in, u, prefix)))
        for (int e = tid; e < R * SIMT_KC; e += SIMT_THREADS) {
            const int r = e / SIMT_KC, kk = e - r * SIMT_KC;
            if (kk < kc) {
                const int k = k0 + kk;
                const float *w = m.W1 + (size_t)k * F;
                float a = rows.prefix(r)[k];
                a = __fmaf_rn(w[F - 2], us[rows.query(r)], a);
                a = __fmaf_rn(w[F - 1], vs[rows.query(r)], a);
                h1s[r * (SIMT_KC + 1) + kk] = a > 0.f ? a : 0.f;
            }
        }
        for (int e = tid; e < H2 * SIMT_KC; e += SIMT_THREADS) {
            const int n = e / SIMT_KC, kk = e - n * SIMT_KC;
            if (kk < kc) w2s[kk * w2ld + n] = m.W2[(size_t)n * H1 + k0 + kk];
        }
        __syncthreads();
        for (int kk = 0; kk < kc; ++kk) {
            float b[CPT];
#pragma unroll
            for (int j = 0; j < CPT; ++j) {
                const int n = lane + 32 * j;
                b[j] = n < H2 ? w2s[kk * w2ld + n] : 0.f;
            }
#pragma unroll
            for (int i = 0; i < RPT; ++i) {
                const float a = h1s[(warp + 8 * i) * (SIMT_KC + 1) + kk];
#pragma unroll
                for (int j = 0; j < CPT; ++j) acc[i][j] = __fmaf_rn(b[j], a, acc[i][j]);
            }
        }
        __syncthreads();
    }

    float *h2s = tile;
#pragma unroll
    for (int i = 0; i < RPT; ++i) {
        const int r = warp + 8 * i;
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            const int n = lane + 32 * j;
            if (r < R && n < H2) {
                const float v = acc[i][j];
                h2s[r * w2ld + n] = v > 0.f ? v : 0.f;
            }
        }
    }
    __syncthreads();
    for (int e = tid; e < m.NH * R; e += SIMT_THREADS) {
        const int r = e / m.NH, o = e - r * m.NH;
        const float *w3 = m.W3 + (size_t)o * H2;
        float z = m.b3[o];
        for (int n = 0; n < H2; ++n) z = __fmaf_rn(w3[n], h2s[r * w2ld + n], z);
        sp[e] = softplus_c(z);
    }
    __syncthreads();
}

// ---------------------------------------------------------------------------
// K_route_simt: one block routes QB = 64 / D queries end to end.

struct RouteRows {
    const float *A;
    int D, H1;
    __device__ const float *prefix(int r) const { return A + (size_t)(r % D) * H1; }
    __device__ int query(int r) const { return r / D; }
};

__host__ __device__ inline int route_qb(int D) { return D >= 64 ? 1 : 64 / D; }

struct RouteLayout {
    int QB, R;
    size_t us, vs, ol, qual, sp, C, U, tile, total;  // float offsets
};

__host__ __device__ inline RouteLayout route_layout(int D, int M, int H2) {
    RouteLayout L;
    L.QB = route_qb(D);
    L.R = L.QB * D;
    size_t o = 0;
    L.us = o; o += 64;
    L.vs = o; o += 64;
    L.ol = o; o += 64;
    L.qual = o; o += (size_t)L.QB * M;
    L.sp = o; o += 3 * 64;
    L.C = o; o += 64;
    L.U = o; o += 64;
    o = (o + 3) & ~(size_t)3;
    L.tile = o;
    o += tile_floats_for<ROUTE_RPT>(H2);
    L.total = o;
    return L;
}

template <int CPT>
__global__ void __launch_bounds__(SIMT_THREADS) k_route_simt(Model m, Queries q) {
    extern __shared__ float sm[];
    const RouteLayout L = route_layout(m.D, m.M, m.H2);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int D = m.D, M = m.M, F = m.F, QB = L.QB, R = L.R;
    const int q0 = blockIdx.x * QB;
    float *us = sm + L.us, *vs = sm + L.vs, *ol = sm + L.ol, *qual = sm + L.qual;
    float *sp = sm + L.sp, *Cs = sm + L.C, *Us = sm + L.U;

    for (int qi = tid; qi < QB; qi += SIMT_THREADS) {
        const int qq = q0 + qi;
        float u = 0.f, v = 0.f, o = 0.f;
        if (qq < q.Q) {
            o = q.out_len[qq];
            u = standardise(m.xform[F - 2], (double)q.in_len[qq], m.mu[F - 2], m.sd[F - 2]);
            v = standardise(m.xform[F - 1], (double)o, m.mu[F - 1], m.sd[F - 1]);
        }
        us[qi] = u;
        vs[qi] = v;
        ol[qi] = o;
    }
    // quality: one serial chain per (query, model), from 0, k ascending
    for (int e = tid; e < QB * M; e += SIMT_THREADS) {
        const int qi = e / M, mi = e - qi * M, qq = q0 + qi;
        float s = 0.f;
        if (qq < q.Q) {
            const size_t row = (size_t)qq * m.E;
            for (int k = 0; k < m.E; ++k)
                s = __fmaf_rn(emb_at(q.emb, q.emb_bf16, row + k), m.memb[(size_t)k * M + mi], s);
        }
        qual[e] = sigmoid_c(s);
    }
    __syncthreads();

    RouteRows rows{m.A, D, m.H1};
    pair_mlp<ROUTE_RPT, CPT>(m, R, rows, us, vs, sm + L.tile, sp);

    for (int r = tid; r < R; r += SIMT_THREADS) {
        const int qi = r / D, d = r - qi * D;
        const float *h = sp + m.NH * r;   // TTFT, TPOT (, N_out)
        const float C = __fmaf_rn(m.NH == 3 ? h[2] : ol[qi], h[1], h[0]);
        const float Ql = qual[qi * M + m.dep_model[d]];
        Cs[r] = C;
        Us[r] = __fmaf_rn(-q.lam, C, __fmul_rn(q.wq, Ql));
        if (q.pair_C && q0 + qi < q.Q) q.pair_C[(size_t)(q0 + qi) * D + d] = C;
    }
    if (q.qual_out)
        for (int e = tid; e < QB * M; e += SIMT_THREADS)
            if (q0 + e / M < q.Q) q.qual_out[(size_t)q0 * M + e] = qual[e];
    __syncthreads();

    for (int qi = warp; qi < QB; qi += SIMT_THREADS / 32) {
        const int qq = q0 + qi;
        if (qq >= q.Q) continue;
        Cand best = no_cand();
        const float slo = query_budget(q, qq);
        for (int d = lane; d < D; d += 32) {
            Cand c = make_cand(Cs[qi * D + d], Us[qi * D + d], d, slo);
            if (better(c, best)) best = c;
        }
        best = warp_best(best);
        if (lane == 0) {
            const bool ok = best.cls > 0;
            q.chosen[qq] = ok ? best.d : -1;
            q.lat[qq] = ok ? best.C : __int_as_float(0x7fc00000);
            q.util[qq] = ok ? best.U : __int_as_float(0x7fc00000);
        }
    }
}

// ---------------------------------------------------------------------------
// Sequential mode.  Query i of a chunk is scored with running count r_d + c_d
// where c_d counts the chunk's earlier picks of d, c_d <= i.  K_seq_table
// scores every (c, d, i) with c <= i in parallel; K_seq_chain then walks the
// chunk in order reading the table entry of the current c_d.
//
// Table layout (triangular): for c in [0, Qs), d in [0, D), i in [c, Qs):
//   index = D * (c * Qs - c (c - 1) / 2) + d * (Qs - c) + (i - c).
// A table block takes deployment d and the two groups c1 and Qs - 1 - c1,
// whose row counts add up to Qs + 1.

__host__ __device__ inline size_t tri_off(int D, int Qs, int c) {
    return (size_t)D * ((size_t)c * Qs - (size_t)c * (c - 1) / 2);
}

size_t seq_table_floats(int D, int Qs) { return tri_off(D, Qs, Qs); }

struct SeqRows {
    const float *pre;  // [2][H1] in shared memory
    int H1, n1, c1, c2;
    __device__ const float *prefix(int r) const { return r < n1 ? pre : pre + H1; }
    __device__ int query(int r) const { return r < n1 ? c1 + r : c2 + (r - n1); }
};

struct SeqLayout {
    size_t us, vs, ol, pre, sp, tile, total;
};

__host__ __device__ inline SeqLayout seq_layout(int H1, int H2) {
    SeqLayout L;
    size_t o = 0;
    L.us = o; o += SEQ_MAX_CHUNK;
    L.vs = o; o += SEQ_MAX_CHUNK;
    L.ol = o; o += SEQ_MAX_CHUNK;
    L.pre = o; o += 2 * (size_t)H1;
    L.sp = o; o += 3 * 8 * SEQ_RPT;
    o = (o + 3) & ~(size_t)3;
    L.tile = o;
    o += tile_floats_for<SEQ_RPT>(H2);
    L.total = o;
    return L;
}

template <int CPT>
__global__ void __launch_bounds__(SIMT_THREADS)
k_seq_table(Model m, Queries q, int Qs, int nb_table, float *ctab, float *qualS) {
    extern __shared__ float sm[];
    const int tid = threadIdx.x;
    const int D = m.D, F = m.F, H1 = m.H1, M = m.M, P = m.P;
    if ((int)blockIdx.x >= nb_table) {
        // quality of the chunk's queries: one serial chain per (query, model)
        const int e = ((int)blockIdx.x - nb_table) * SIMT_THREADS + tid;
        if (e < Qs * M) {
            const int i = e / M, mi = e - i * M;
            const size_t row = (size_t)i * m.E;
            float s = 0.f;
            for (int k = 0; k < m.E; ++k)
                s = __fmaf_rn(emb_at(q.emb, q.emb_bf16, row + k), m.memb[(size_t)k * M + mi], s);
            qualS[e] = sigmoid_c(s);
        }
        return;
    }
    const SeqLayout L = seq_layout(H1, m.H2);
    float *us = sm + L.us, *vs = sm + L.vs, *ol = sm + L.ol, *pre = sm + L.pre;
    float *sp = sm + L.sp;
    const int d = blockIdx.x % D, c1 = blockIdx.x / D, c2 = Qs - 1 - c1;
    const bool two = c2 != c1;
    const int n1 = Qs - c1, R = n1 + (two ? c1 + 1 : 0);

    for (int i = tid; i < Qs; i += SIMT_THREADS) {
        const float o = q.out_len[i];
        us[i] = standardise(m.xform[F - 2], (double)q.in_len[i], m.mu[F - 2], m.sd[F - 2]);
        vs[i] = standardise(m.xform[F - 1], (double)o, m.mu[F - 1], m.sd[F - 1]);
        ol[i] = o;
    }
    // layer-1 prefixes for running counts r_d + c1 and r_d + c2: continue the
    // chain from slot P + 1 (running) with the deployment's other features
    const int32_t run = m.running[d];
    for (int e = tid; e < 2 * H1; e += SIMT_THREADS) {
        const int g = e / H1, j = e - g * H1;
        if (g == 1 && !two) continue;
        const int c = g ? c2 : c1;
        const float xr = standardise(m.xform[P + 1], (double)(run + c), m.mu[P + 1], m.sd[P + 1]);
        const float *w = m.W1 + (size_t)j * F;
        const float *x = m.X + (size_t)d * F;
        float acc = m.Spre[(size_t)d * H1 + j];
        acc = __fmaf_rn(w[P + 1], xr, acc);
        for (int k = P + 2; k < F - 2; ++k) acc = __fmaf_rn(w[k], x[k], acc);
        pre[e] = acc;
    }
    __syncthreads();

    SeqRows rows{pre, H1, n1, c1, c2};
    pair_mlp<SEQ_RPT, CPT>(m, R, rows, us, vs, sm + L.tile, sp);

    for (int r = tid; r < R; r += SIMT_THREADS) {
        const int c = r < n1 ? c1 : c2, i = rows.query(r);
        const float *h = sp + m.NH * r;
        const float C = __fmaf_rn(m.NH == 3 ? h[2] : ol[i], h[1], h[0]);
        ctab[tri_off(D, Qs, c) + (size_t)d * (Qs - c) + (i - c)] = C;
    }
}

__global__ void __launch_bounds__(SIMT_THREADS)
k_seq_chain(Model m, Queries q, int Qs, const float *ctab, const float *qualS) {
    extern __shared__ float sm[];
    const int tid = threadIdx.x, lane = tid & 31;
    const int D = m.D, M = m.M, F = m.F, H1 = m.H1, P = m.P;
    const size_t T = tri_off(D, Qs, Qs);
    float *tab = sm;
    float *qs = sm + T;
    int *dm = (int *)(qs + (size_t)Qs * M);
    int *cnt = dm + MAX_D;
    for (size_t e = tid; e < T; e += SIMT_THREADS) tab[e] = ctab[e];
    for (int e = tid; e < Qs * M; e += SIMT_THREADS) qs[e] = qualS[e];
    for (int e = tid; e < D; e += SIMT_THREADS) dm[e] = m.dep_model[e];
    __syncthreads();

    if (tid < 32) {
        int cA = 0, cB = 0;  // picks so far of deployments lane and lane + 32
        for (int i = 0; i < Qs; ++i) {
            Cand best = no_cand();
            const float slo = query_budget(q, i);
#pragma unroll
            for (int t = 0; t < 2; ++t) {
                const int d = lane + 32 * t;
                if (d < D) {
                    const int c = t ? cB : cA;
                    const float C = tab[tri_off(D, Qs, c) + (size_t)d * (Qs - c) + (i - c)];
                    const float U = __fmaf_rn(-q.lam, C, __fmul_rn(q.wq, qs[i * M + dm[d]]));
                    Cand cd = make_cand(C, U, d, slo);
                    if (better(cd, best)) best = cd;
                }
            }
            best = warp_best(best);
            const bool ok = best.cls > 0;
            if (lane == 0) {
                q.chosen[i] = ok ? best.d : -1;
                q.lat[i] = ok ? best.C : __int_as_float(0x7fc00000);
                q.util[i] = ok ? best.U : __int_as_float(0x7fc00000);
            }
            if (ok) {
                if (best.d == lane) ++cA;
                else if (best.d == lane + 32) ++cB;
            }
        }
        if (lane < D) cnt[lane] = cA;
        if (lane + 32 < D) cnt[lane + 32] = cB;
    }
    __syncthreads();
    // persist the increments and refresh the deployment state they touch
    for (int d = tid; d < D; d += SIMT_THREADS) m.running[d] += cnt[d];
    __syncthreads();
    for (int e = tid; e < D * H1; e += SIMT_THREADS) {
        const int d = e / H1, j = e - d * H1;
        const float xr = standardise(m.xform[P + 1], (double)m.running[d], m.mu[P + 1], m.sd[P + 1]);
        const float *w = m.W1 + (size_t)j * F;
        const float *x = m.X + (size_t)d * F;
        float acc = m.Spre[(size_t)d * H1 + j];
        acc = __fmaf_rn(w[P + 1], xr, acc);
        for (int k = P + 2; k < F - 2; ++k) acc = __fmaf_rn(w[k], x[k], acc);
        m.A[(size_t)d * H1 + j] = acc;
        m.Abf[(size_t)d * H1 + j] = __bfloat16_as_ushort(__float2bfloat16_rn(acc));
        if (j == 0) m.X[(size_t)d * F + P + 1] = xr;
    }
}

// ---------------------------------------------------------------------------
// K_route_pairs: the small-batch (latency) variant.  One block per (query,
// deployment) pair computes that pair's predictor with one thread per hidden
// unit (W2 read transposed so a warp's loads are contiguous); quality blocks
// run the per-(query, model) chains from shared memory; the last block to
// finish a query (per-query arrival counter, self-resetting) applies the
// decision maker.  Same canonical order as the kernels above.

struct PairArgs {
    const float *W2T;   // [H1][H2]: W2 transposed
    float *pairC;       // [Q][D] scratch
    float *qualS;       // [Q][M] scratch
    int32_t *count;     // [Q] arrivals, zero between calls
    int qblocks;        // quality blocks per query
};

constexpr int PAIR_MPB = 8;  // models per quality block

__device__ void pair_select(const Model &m, const Queries &q, const PairArgs &a, int qq) {
    // warp 0 of the last block of query qq: utility, SLO mask, argmax
    const int lane = threadIdx.x & 31;
    Cand best = no_cand();
    const float slo = query_budget(q, qq);
    for (int d = lane; d < m.D; d += 32) {
        const float C = __ldcg(&a.pairC[(size_t)qq * m.D + d]);
        const float Ql = __ldcg(&a.qualS[(size_t)qq * m.M + m.dep_model[d]]);
        const float U = __fmaf_rn(-q.lam, C, __fmul_rn(q.wq, Ql));
        Cand c = make_cand(C, U, d, slo);
        if (better(c, best)) best = c;
    }
    best = warp_best(best);
    if (lane == 0) {
        const bool ok = best.cls > 0;
        q.chosen[qq] = ok ? best.d : -1;
        q.lat[qq] = ok ? best.C : __int_as_float(0x7fc00000);
        q.util[qq] = ok ? best.U : __int_as_float(0x7fc00000);
        a.count[qq] = 0;
    }
}

__global__ void __launch_bounds__(SIMT_THREADS) k_route_pairs(Model m, Queries q, PairArgs a) {
    extern __shared__ float sm[];
    __shared__ int s_last;
    const int tid = threadIdx.x, F = m.F, H1 = m.H1, H2 = m.H2, D = m.D, M = m.M;
    const int npair = q.Q * D;
    int qq;
    if ((int)blockIdx.x < npair) {
        qq = blockIdx.x / D;
        const int d = blockIdx.x - qq * D;
        float *h1 = sm, *h2 = sm + MAX_H;
        __shared__ float uv[3];
        if (tid == 0) {
            const float o = q.out_len[qq];
            uv[0] = standardise(m.xform[F - 2], (double)q.in_len[qq], m.mu[F - 2], m.sd[F - 2]);
            uv[1] = standardise(m.xform[F - 1], (double)o, m.mu[F - 1], m.sd[F - 1]);
            uv[2] = o;
        }
        __syncthreads();
        for (int k = tid; k < H1; k += SIMT_THREADS) {
            const float *w = m.W1 + (size_t)k * F;
            float x = m.A[(size_t)d * H1 + k];
            x = __fmaf_rn(w[F - 2], uv[0], x);
            x = __fmaf_rn(w[F - 1], uv[1], x);
            h1[k] = x > 0.f ? x : 0.f;
        }
        __syncthreads();
        float *w3s = sm + 2 * MAX_H;   // W3 [NH][H2], staged for the head chains
        for (int i = tid; i < m.NH * H2; i += SIMT_THREADS) w3s[i] = m.W3[i];
        for (int n = tid; n < H2; n += SIMT_THREADS) {
            // serial chain over k (canonical order); W2 values fetched 32 at a
            // time, the next block in flight while this one is accumulated
            float acc = m.b2[n];
            float w[32], wn[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) w[j] = j < H1 ? a.W2T[(size_t)j * H2 + n] : 0.f;
            for (int k0 = 0; k0 < H1; k0 += 32) {
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    wn[j] = k0 + 32 + j < H1 ? a.W2T[(size_t)(k0 + 32 + j) * H2 + n] : 0.f;
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (k0 + j < H1) acc = __fmaf_rn(w[j], h1[k0 + j], acc);
#pragma unroll
                for (int j = 0; j < 32; ++j) w[j] = wn[j];
            }
            h2[n] = acc > 0.f ? acc : 0.f;
        }
        __syncthreads();
        __shared__ float heads[3];
        if (tid < 32 * m.NH) {
            // the output heads, one warp each
            const int o = tid >> 5;
            if ((tid & 31) == 0) {
                const float *w3 = w3s + (size_t)o * H2;
                float z = m.b3[o];
                for (int n = 0; n < H2; ++n) z = __fmaf_rn(w3[n], h2[n], z);
                heads[o] = softplus_c(z);
            }
        }
        __syncthreads();
        if (tid == 0)
            a.pairC[(size_t)qq * D + d] =
                __fmaf_rn(m.NH == 3 ? heads[2] : uv[2], heads[1], heads[0]);
    } else {
        // quality of models [m0, m0 + PAIR_MPB) for one query
        const int b = blockIdx.x - npair;
        qq = b / a.qblocks;
        const int m0 = (b - qq * a.qblocks) * PAIR_MPB, mn = min(PAIR_MPB, M - m0), E = m.E;
        float *er = sm, *mb = sm + E;   // emb row [E], model columns [mn][E]
        const size_t row = (size_t)qq * E;
        for (int k = tid; k < E; k += SIMT_THREADS) {
            er[k] = emb_at(q.emb, q.emb_bf16, row + k);
            for (int j = 0; j < mn; ++j) mb[(size_t)j * E + k] = m.memb[(size_t)k * M + m0 + j];
        }
        __syncthreads();
        if (tid < mn) {
            const float *c = mb + (size_t)tid * E;
            float s = 0.f;
#pragma unroll 8
            for (int k = 0; k < E; ++k) s = __fmaf_rn(er[k], c[k], s);
            a.qualS[(size_t)qq * M + m0 + tid] = sigmoid_c(s);
        }
    }
    // the last of the query's D + qblocks blocks applies the decision maker
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        s_last = atomicAdd(&a.count[qq], 1) == D + a.qblocks - 1;
    }
    __syncthreads();
    if (s_last && tid < 32) {
        __threadfence();
        pair_select(m, q, a, qq);
    }
}

// ---------------------------------------------------------------------------
// K_select_multi: the decision maker for several lambdas over stored scores
// (one warp per (query, lambda)); same candidate order as everywhere else.

__global__ void __launch_bounds__(SIMT_THREADS)
k_select_multi(Model m, Queries q, const float *C, const float *qual, int qstride, Lambdas L,
               int ostride) {
    const int wid = (blockIdx.x * SIMT_THREADS + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (wid >= q.Q * L.K) return;
    const int k = wid / q.Q, qq = wid - k * q.Q;
    const float slo = query_budget(q, qq), lam = L.lam[k], wq = L.wq[k];
    Cand best = no_cand();
    for (int d = lane; d < m.D; d += 32) {
        const float c = C[(size_t)qq * m.D + d];
        const float Ql = qual[(size_t)qq * qstride + m.dep_model[d]];
        Cand cd = make_cand(c, __fmaf_rn(-lam, c, __fmul_rn(wq, Ql)), d, slo);
        if (better(cd, best)) best = cd;
    }
    best = warp_best(best);
    if (lane == 0) {
        const bool ok = best.cls > 0;
        const size_t o = (size_t)k * ostride + qq;
        q.chosen[o] = ok ? best.d : -1;
        q.lat[o] = ok ? best.C : __int_as_float(0x7fc00000);
        q.util[o] = ok ? best.U : __int_as_float(0x7fc00000);
    }
}

// ---------------------------------------------------------------------------
// host launchers

static int cpt_for(int H2) { return H2 <= 32 ? 1 : H2 <= 64 ? 2 : H2 <= 128 ? 4 : 8; }

size_t route_simt_smem(const Model &m) {
    return route_layout(m.D, m.M, m.H2).total * sizeof(float);
}

size_t seq_table_smem(const Model &m) {
    return seq_layout(m.H1, m.H2).total * sizeof(float);
}

static size_t chain_smem(int D, int M, int Qs) {
    return (tri_off(D, Qs, Qs) + (size_t)Qs * M) * sizeof(float) + 2 * MAX_D * sizeof(int);
}

int seq_chunk(const Model &m) {
    int Qs = SEQ_MAX_CHUNK;
    while (Qs > 1 && chain_smem(m.D, m.M, Qs) > (size_t)SEQ_CHAIN_SMEM) --Qs;
    return Qs;
}

template <class K>
static cudaError_t opt_in(K kernel, int bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t simt_prepare() {
    const int big = 200 * 1024;
    cudaError_t e = cudaSuccess;
    if (e == cudaSuccess) e = opt_in(k_route_simt<1>, big);
    if (e == cudaSuccess) e = opt_in(k_route_simt<2>, big);
    if (e == cudaSuccess) e = opt_in(k_route_simt<4>, big);
    if (e == cudaSuccess) e = opt_in(k_route_simt<8>, big);
    if (e == cudaSuccess) e = opt_in(k_seq_table<1>, big);
    if (e == cudaSuccess) e = opt_in(k_seq_table<2>, big);
    if (e == cudaSuccess) e = opt_in(k_seq_table<4>, big);
    if (e == cudaSuccess) e = opt_in(k_seq_table<8>, big);
    if (e == cudaSuccess) e = opt_in(k_seq_chain, SEQ_CHAIN_SMEM + 1024);
    if (e == cudaSuccess) e = opt_in(k_route_pairs, big);
    return e;
}

cudaError_t launch_snapshot(const Model &m, cudaStream_t s) {
    k_snapshot<<<m.D, SIMT_THREADS, (size_t)m.F * sizeof(float), s>>>(m);
    return cudaGetLastError();
}

cudaError_t launch_route_simt(const Model &m, const Queries &q, cudaStream_t s) {
    if (q.Q <= 0) return cudaSuccess;
    const RouteLayout L = route_layout(m.D, m.M, m.H2);
    const int blocks = (q.Q + L.QB - 1) / L.QB;
    const size_t smem = L.total * sizeof(float);
    switch (cpt_for(m.H2)) {
        case 1: k_route_simt<1><<<blocks, SIMT_THREADS, smem, s>>>(m, q); break;
        case 2: k_route_simt<2><<<blocks, SIMT_THREADS, smem, s>>>(m, q); break;
        case 4: k_route_simt<4><<<blocks, SIMT_THREADS, smem, s>>>(m, q); break;
        default: k_route_simt<8><<<blocks, SIMT_THREADS, smem, s>>>(m, q); break;
    }
    return cudaGetLastError();
}

size_t route_pairs_smem(const Model &m) {
    const size_t pair = 5 * MAX_H * sizeof(float);
    const size_t qual = (size_t)m.E * (1 + PAIR_MPB) * sizeof(float);
    return pair > qual ? pair : qual;
}

cudaError_t launch_route_pairs(const Model &m, const Queries &q, const float *W2T, float *pairC,
                               float *qualS, int32_t *count, cudaStream_t s) {
    if (q.Q <= 0) return cudaSuccess;
    PairArgs a;
    a.W2T = W2T;
    a.pairC = pairC;
    a.qualS = qualS;
    a.count = count;
    a.qblocks = (m.M + PAIR_MPB - 1) / PAIR_MPB;
    const int blocks = q.Q * (m.D + a.qblocks);
    k_route_pairs<<<blocks, SIMT_THREADS, route_pairs_smem(m), s>>>(m, q, a);
    return cudaGetLastError();
}

cudaError_t launch_select_multi(const Model &m, const Queries &q, const float *C,
                                const float *qual, int qstride, const Lambdas &L, int ostride,
                                cudaStream_t s) {
    if (q.Q <= 0 || L.K <= 0) return cudaSuccess;
    const long warps = (long)q.Q * L.K;
    const int blocks = (int)((warps * 32 + SIMT_THREADS - 1) / SIMT_THREADS);
    k_select_multi<<<blocks, SIMT_THREADS, 0, s>>>(m, q, C, qual, qstride, L, ostride);
    return cudaGetLastError();
}

cudaError_t launch_seq_table(const Model &m, const Queries &q, int Qs, float *ctab,
                             float *qual, cudaStream_t s) {
    const int nb_table = m.D * ((Qs + 1) / 2);
    const int nb_qual = (Qs * m.M + SIMT_THREADS - 1) / SIMT_THREADS;
    const size_t smem = seq_layout(m.H1, m.H2).total * sizeof(float);
    const int blocks = nb_table + nb_qual;
    switch (cpt_for(m.H2)) {
        case 1: k_seq_table<1><<<blocks, SIMT_THREADS, smem, s>>>(m, q, Qs, nb_table, ctab, qual); break;
        case 2: k_seq_table<2><<<blocks, SIMT_THREADS, smem, s>>>(m, q, Qs, nb_table, ctab, qual); break;
        case 4: k_seq_table<4><<<blocks, SIMT_THREADS, smem, s>>>(m, q, Qs, nb_table, ctab, qual); break;
        default: k_seq_table<8><<<blocks, SIMT_THREADS, smem, s>>>(m, q, Qs, nb_table, ctab, qual); break;
    }
    return cudaGetLastError();
}

cudaError_t launch_seq_chain(const Model &m, const Queries &q, int Qs, const float *ctab,
                             const float *qual, cudaStream_t s) {
    k_seq_chain<<<1, SIMT_THREADS, chain_smem(m.D, m.M, Qs), s>>>(m, q, Qs, ctab, qual);
    return cudaGetLastError();
}

}  // namespace hwr
