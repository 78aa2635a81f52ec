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
#include "umma.cuh"

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

// Quality score (Sec. 3.2, hardware-independent term) of queries
// [q0, q0 + nq): one serial chain per (query, model) from 0 with k ascending,
// then the sigmoid.  The embedding rows (as stored, fp32 or bf16) and the
// model columns are staged through `stage` (at least (nq + M) * 8 + 64
// floats) in chunks of the embedding dimension by 16-byte asynchronous copies
// when the embeddings are 16-byte aligned (plain loads otherwise); the
// chains read shared memory only.  Every thread of the block calls this;
// thread t < nq * M returns the score of query t / M, model t % M (rows at or
// past q.Q give sigmoid(0)), the others return 0.  Ends with the stage free
// for reuse after a barrier.  NT threads take part: the whole block
// (NT = SIMT_THREADS, block barriers, thread index t = threadIdx.x) or one
// warp (NT = 32, warp barriers, t = lane), which then runs the chains
// t, t + 32 (CH = 2: at most 64 (query, model) pairs) and returns the score of
// chain t + 32 j in res[j].
template <int NT>
__device__ __forceinline__ void group_sync() {
    if constexpr (NT == 32) __syncwarp();
    else __syncthreads();
}

template <int NT, int CH>
__device__ void quality_group(const Model &m, const Queries &q, int q0, int nq, float *stage,
                              int stage_floats, int t, float (&res)[CH]) {
    const int tid = t, M = m.M, E = m.E;
    const int es = q.emb_bf16 ? 2 : 4;
    const bool async = !q.inputs_host && ((uintptr_t)q.emb & 15) == 0;
    // row stride ld (elements): 16-byte rows whose 4-byte word stride is 4
    // mod 32, so the chains of one warp (up to 8 rows) read distinct banks
    auto stride = [&](int ek) {
        return es == 4 ? ((ek - 4 + 31) / 32) * 32 + 4 : ((ek - 8 + 63) / 64) * 64 + 8;
    };
    int ek = E;
    while (ek > 8 && ((size_t)nq * stride(ek) * es + 16 + (size_t)ek * M * 4) > 4 * (size_t)stage_floats)
        ek -= 8;
    const int ld = stride(ek);
    char *er = reinterpret_cast<char *>(stage);
    float *mb = reinterpret_cast<float *>(er + (((size_t)nq * ld * es + 15) & ~(size_t)15));
    float s[CH];
#pragma unroll
    for (int j = 0; j < CH; ++j) s[j] = 0.f;
    for (int k0 = 0; k0 < E; k0 += ek) {
        const int kc = min(ek, E - k0);
        group_sync<NT>();
        if (async) {
            const int gpr = kc * es / 16;     // granules per row (kc is a multiple of 8)
            const uint32_t eb = (uint32_t)__cvta_generic_to_shared(er);
            for (int g = tid; g < nq * gpr; g += NT) {
                const int i = g / gpr, c = g - i * gpr, qq = q0 + i;
                const char *src = (const char *)q.emb + ((size_t)(qq < q.Q ? qq : 0) * E + k0) * es + 16 * c;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(
                                 eb + (uint32_t)(i * ld * es + 16 * c)),
                             "l"(__cvta_generic_to_global(src)), "r"(qq < q.Q ? 16 : 0)
                             : "memory");
            }
            const uint32_t mbs = (uint32_t)__cvta_generic_to_shared(mb);
            for (int g = tid; g < kc * M / 4; g += NT)
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(mbs + 16u * g),
                             "l"(__cvta_generic_to_global(m.memb + (size_t)k0 * M + 4 * g))
                             : "memory");
            asm volatile("cp.async.commit_group;" ::: "memory");
            asm volatile("cp.async.wait_group 0;" ::: "memory");
        } else {
            for (int t = tid; t < nq * kc; t += NT) {
                const int i = t / kc, k = t - i * kc, qq = q0 + i;
                const size_t src = (size_t)(qq < q.Q ? qq : 0) * E + k0 + k;
                if (es == 4) reinterpret_cast<float *>(er)[i * ld + k] = qq < q.Q ? ((const float *)q.emb)[src] : 0.f;
                else reinterpret_cast<uint16_t *>(er)[i * ld + k] = qq < q.Q ? ((const uint16_t *)q.emb)[src] : 0;
            }
            for (int t = tid; t < kc * M; t += NT) mb[t] = m.memb[(size_t)k0 * M + t];
        }
        group_sync<NT>();
#pragma unroll
        for (int j = 0; j < CH; ++j) {
            const int e = tid + NT * j, qi = e / M, mi = e - qi * M;
            if (e < nq * M) {
                const float *b = mb + mi;
                float acc = s[j];
                if (es == 4) {
                    const float *a = reinterpret_cast<const float *>(er) + qi * ld;
#pragma unroll 8
                    for (int k = 0; k < kc; ++k) acc = __fmaf_rn(a[k], b[k * M], acc);
                } else {
                    const uint16_t *a = reinterpret_cast<const uint16_t *>(er) + qi * ld;
#pragma unroll 8
                    for (int k = 0; k < kc; ++k)
                        acc = __fmaf_rn(__uint_as_float((uint32_t)a[k] << 16), b[k * M], acc);
                }
                s[j] = acc;
            }
        }
    }
#pragma unroll
    for (int j = 0; j < CH; ++j) res[j] = tid + NT * j < nq * M ? sigmoid_c(s[j]) : 0.f;
}

__device__ __forceinline__ float quality_staged(const Model &m, const Queries &q, int q0, int nq,
                                                float *stage, int stage_floats) {
    float r[1];
    quality_group<SIMT_THREADS, 1>(m, q, q0, nq, stage, stage_floats, threadIdx.x, r);
    return r[0];
}

// ---------------------------------------------------------------------------
// K_snap: standardised deployment features and the deployment prefix of
// layer 1 (the part of W1 x + b1 that does not depend on the query).

__global__ void __launch_bounds__(SIMT_THREADS) k_snapshot(Model m, const uint32_t *stage) {
    extern __shared__ float xs[];
    const int d = blockIdx.x;
    // this deployment's six signals, from the host's staging ([6][D], mapped)
    // into the context's device arrays (running, waiting, kv, gpu_util, ttft, tpot)
    if (threadIdx.x < 6)
        reinterpret_cast<uint32_t *>(m.running)[(size_t)threadIdx.x * m.D + d] =
            stage[(size_t)threadIdx.x * m.D + d];
    __syncthreads();
    for (int k = threadIdx.x; k < m.F - 2; k += blockDim.x) {
        float x = standardise(m.xform[k], deployment_raw(m, d, k, m.running[d]),
                              m.mu[k], m.sd[k]);
        xs[k] = x;
        m.X[(size_t)d * m.F + k] = x;
    }
    __syncthreads();
    for (int j = threadIdx.x; j < m.H1; j += blockDim.x) {
        const float *w = m.W1T + j;   // slot k at w[k * H1]
        float acc = m.b1[j];
        // slots k0 .. k1 - 1 in order, their weights loaded eight at a time
        // ahead of the FMAs (the loads would otherwise wait one by one)
        auto chain = [&](int k0, int k1) {
            int k = k0;
            for (; k + 8 <= k1; k += 8) {
                float wv[8];
#pragma unroll
                for (int t = 0; t < 8; ++t) wv[t] = w[(size_t)(k + t) * m.H1];
#pragma unroll
                for (int t = 0; t < 8; ++t) acc = __fmaf_rn(wv[t], xs[k + t], acc);
            }
            for (; k < k1; ++k) acc = __fmaf_rn(w[(size_t)k * m.H1], xs[k], acc);
        };
        chain(0, m.P + 1);
        m.Spre[(size_t)d * m.H1 + j] = acc;
        chain(m.P + 1, m.F - 2);
        m.A[(size_t)d * m.H1 + j] = acc;
        m.Abf[(size_t)d * m.H1 + j] = __bfloat16_as_ushort(__float2bfloat16_rn(acc));
    }
}

// ---------------------------------------------------------------------------
// The shared SIMT tile: up to TILE_ROWS rows, each a (query, deployment) pair
// or a sequential-table entry.  For every row it completes layer 1 from a
// deployment prefix and the two query features, runs layer 2 (register-tiled,
// K ascending in chunks of SIMT_KC), layer 3 and the softplus heads.  Output:
// sp[NH r + 0] = TTFT, sp[NH r + 1] = TPOT and, with three heads,
// sp[NH r + 2] = N_out.
//
// Thread map: warp w owns rows 8w .. 8w + 7 and lane l owns columns
// 128 j + VW l + v (v < VW = min(CPT, 4), j < CPT / VW): a lane reads its
// rows' layer-1 values as two 16-byte broadcasts and its W2 columns as
// vectors that are contiguous across the warp.  Shared memory: the layer-1
// chunk [KC][TILE_ROWS] (k-major) and two W2 chunks [KC][32 CPT] (rows of W2
// transposed; the next chunk's cp.async copies run while this one is used),
// then h2 [TILE_ROWS][H2 + 1] in the same space; W3 [NH][H2] in w3s.

constexpr int TILE_ROWS = 64;

// Barrier of the tile's SIMT_THREADS threads only (named barrier 1), so a
// block may run other warps beside the tile.
__device__ __forceinline__ void tile_sync() {
    asm volatile("bar.sync 1, %0;" ::"n"(SIMT_THREADS) : "memory");
}

// n rounded up to a multiple of 4, then to an odd multiple of 4: rows of
// this stride, read by a warp as 16-byte vectors (one row per lane), fall in
// distinct banks across each wavefront's 8 lanes.
__host__ __device__ constexpr int odd_units(int n) {
    return (((n + 3) & ~3) >> 2) & 1 ? (n + 3) & ~3 : ((n + 3) & ~3) + 4;
}

__host__ __device__ constexpr int tile_width(int H2) {
    return H2 <= 32 ? 32 : H2 <= 64 ? 64 : H2 <= 128 ? 128 : 256;
}

__host__ __device__ constexpr size_t tile_floats_for(int H2) {
    return (size_t)SIMT_KC * TILE_ROWS + 2 * (size_t)SIMT_KC * tile_width(H2) >
                   (size_t)TILE_ROWS * odd_units(H2)
               ? (size_t)SIMT_KC * TILE_ROWS + 2 * (size_t)SIMT_KC * tile_width(H2)
               : (size_t)TILE_ROWS * odd_units(H2);
}

// Rows k0 .. k0 + kc - 1 of W2 transposed into dst [kc][W] by 16-byte
// asynchronous copies (W2T rows are H2p floats, 16-byte aligned); one group.
__device__ __forceinline__ void w2_chunk_async(const Model &m, int k0, int kc, float *dst, int W) {
    const int gpr = m.H2p >> 2;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(dst);
    for (int g = threadIdx.x; g < kc * gpr; g += SIMT_THREADS) {
        const int kk = g / gpr, c4 = g - kk * gpr;
        const float *src = m.W2T + (size_t)(k0 + kk) * m.H2p + 4 * c4;
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                         base + (uint32_t)(4 * (kk * W + 4 * c4))),
                     "l"(__cvta_generic_to_global(src))
                     : "memory");
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
}

// The tile's weights that no row depends on: W3 for the head chains, the two
// query columns of W1 (both visible after the first barrier of the K loop)
// and the first W2 chunk (one cp.async group).  pair_mlp runs this itself
// unless the caller did, e.g. before waiting for a preceding kernel.
template <int CPT>
__device__ void pair_mlp_stage(const Model &m, float *tile, float *w3s, float *w1q) {
    const int tid = threadIdx.x, H1 = m.H1, H2 = m.H2, F = m.F;
    for (int i = tid; i < m.NH * H2; i += SIMT_THREADS) w3s[i] = m.W3[i];
    for (int k = tid; k < H1; k += SIMT_THREADS) {
        w1q[k] = m.W1[(size_t)k * F + F - 2];
        w1q[H1 + k] = m.W1[(size_t)k * F + F - 1];
    }
    w2_chunk_async(m, 0, min(SIMT_KC, H1), tile + SIMT_KC * TILE_ROWS, 32 * CPT);
}

template <int CPT, class Rows>
__device__ void pair_mlp(const Model &m, int R, const Rows &rows, const float *us,
                         const float *vs, float *tile, float *w3s, float *w1q, float *sp,
                         bool staged = false) {
    constexpr int VW = CPT < 4 ? CPT : 4, W = 32 * CPT;
    static_assert(SIMT_THREADS == 4 * TILE_ROWS, "layer-1 map: 4 threads per row");
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int H1 = m.H1, H2 = m.H2;
    float *h1T = tile;
    float *w2b = tile + SIMT_KC * TILE_ROWS;

    if (!staged) pair_mlp_stage<CPT>(m, tile, w3s, w1q);
    // layer-1 map: thread t fills row t % 64 at k offsets t / 64 + 4 j of a chunk
    const int r1 = tid % TILE_ROWS, kq = tid / TILE_ROWS;
    const bool rv = r1 < R;
    const float *pr = rv ? rows.prefix(r1) : m.W1;
    const float uq = rv ? us[rows.query(r1)] : 0.f, vq = rv ? vs[rows.query(r1)] : 0.f;
    tile_sync();
    float acc[8][CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        const int n = 128 * (j / VW) + VW * lane + j % VW;
        const float b = n < H2 ? m.b2[n] : 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i][j] = b;
    }
    const bool active = 8 * warp < R;

    for (int k0 = 0, it = 0; k0 < H1; k0 += SIMT_KC, ++it) {
        const int kc = min(SIMT_KC, H1 - k0);
        // layer 1, query suffix: h1 = relu(fma(w_out, v, fma(w_in, u, prefix)));
        // rows at or past R hold 0; a thread's prefix loads are issued together
        float pv[SIMT_KC / 4];
#pragma unroll
        for (int j = 0; j < SIMT_KC / 4; ++j) {
            const int kk = kq + 4 * j;
            pv[j] = rv && kk < kc ? pr[k0 + kk] : 0.f;
        }
#pragma unroll
        for (int j = 0; j < SIMT_KC / 4; ++j) {
            const int kk = kq + 4 * j;
            float a = 0.f;
            if (rv && kk < kc) {
                a = __fmaf_rn(w1q[k0 + kk], uq, pv[j]);
                a = __fmaf_rn(w1q[H1 + k0 + kk], vq, a);
                a = a > 0.f ? a : 0.f;
            }
            h1T[kk * TILE_ROWS + r1] = a;
        }
        // the next W2 chunk goes into the other buffer; this one must be complete
        if (k0 + SIMT_KC < H1) {
            w2_chunk_async(m, k0 + SIMT_KC, min(SIMT_KC, H1 - k0 - SIMT_KC),
                           w2b + ((it + 1) & 1) * SIMT_KC * W, W);
            asm volatile("cp.async.wait_group 1;" ::: "memory");
        } else {
            asm volatile("cp.async.wait_group 0;" ::: "memory");
        }
        tile_sync();
        if (active) {
            const float *wb = w2b + (it & 1) * SIMT_KC * W;
#pragma unroll 4
            for (int kk = 0; kk < kc; ++kk) {
                const float4 a0 = *reinterpret_cast<const float4 *>(h1T + kk * TILE_ROWS + 8 * warp);
                const float4 a1 =
                    *reinterpret_cast<const float4 *>(h1T + kk * TILE_ROWS + 8 * warp + 4);
                const float a[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
                float b[CPT];
                const float *wr = wb + kk * W + VW * lane;
#pragma unroll
                for (int v = 0; v < CPT / VW; ++v) {
                    if constexpr (VW == 4) {
                        const float4 t = *reinterpret_cast<const float4 *>(wr + 128 * v);
                        b[4 * v] = t.x;
                        b[4 * v + 1] = t.y;
                        b[4 * v + 2] = t.z;
                        b[4 * v + 3] = t.w;
                    } else if constexpr (VW == 2) {
                        const float2 t = *reinterpret_cast<const float2 *>(wr);
                        b[0] = t.x;
                        b[1] = t.y;
                    } else {
                        b[0] = wr[0];
                    }
                }
                // rows 2ip and 2ip + 1 in one packed fp32 FMA (fma.rn.f32x2:
                // each lane the same single rounding as __fmaf_rn)
#pragma unroll
                for (int ip = 0; ip < 4; ++ip) {
                    const float2 a2 = make_float2(a[2 * ip], a[2 * ip + 1]);
#pragma unroll
                    for (int j = 0; j < CPT; ++j) {
                        const float2 r = __ffma2_rn(make_float2(b[j], b[j]), a2,
                                                    make_float2(acc[2 * ip][j], acc[2 * ip + 1][j]));
                        acc[2 * ip][j] = r.x;
                        acc[2 * ip + 1][j] = r.y;
                    }
                }
            }
        }
        tile_sync();
    }

    float *h2s = tile;
    const int ld = odd_units(H2);
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int r = 8 * warp + i;
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            const int n = 128 * (j / VW) + VW * lane + j % VW;
            if (r < R && n < H2) {
                const float v = acc[i][j];
                h2s[r * ld + n] = v > 0.f ? v : 0.f;
            }
        }
    }
    tile_sync();
    for (int e = tid; e < m.NH * R; e += SIMT_THREADS) {
        // head chain o of row r, n ascending: eight n of operands as 16-byte
        // vectors before their FMAs (a chain step waiting on its own shared
        // loads costs several times its FMA)
        const int r = e / m.NH, o = e - r * m.NH;
        const float *w3 = w3s + (size_t)o * H2, *hr = h2s + (size_t)r * ld;
        float z = m.b3[o];
        int n = 0;
        if ((H2 & 3) == 0) {
            for (; n + 8 <= H2; n += 8) {
                const float4 h0 = *reinterpret_cast<const float4 *>(hr + n);
                const float4 h1 = *reinterpret_cast<const float4 *>(hr + n + 4);
                const float4 v0 = *reinterpret_cast<const float4 *>(w3 + n);
                const float4 v1 = *reinterpret_cast<const float4 *>(w3 + n + 4);
                z = __fmaf_rn(v0.x, h0.x, z);
                z = __fmaf_rn(v0.y, h0.y, z);
                z = __fmaf_rn(v0.z, h0.z, z);
                z = __fmaf_rn(v0.w, h0.w, z);
                z = __fmaf_rn(v1.x, h1.x, z);
                z = __fmaf_rn(v1.y, h1.y, z);
                z = __fmaf_rn(v1.z, h1.z, z);
                z = __fmaf_rn(v1.w, h1.w, z);
            }
        }
        for (; n < H2; ++n) z = __fmaf_rn(w3[n], hr[n], z);
        sp[e] = softplus_c(z);
    }
    tile_sync();
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

constexpr int ROUTE_QSTAGE = 4096;   // floats of the quality warp's staging space

struct RouteLayout {
    int QB, R;
    size_t us, vs, ol, qual, sp, C, U, w3, w1q, qstage, tile, total;  // float offsets
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
    o = (o + 3) & ~(size_t)3;   // W3 rows read as 16-byte vectors
    L.w3 = o; o += 3 * (size_t)H2;
    L.w1q = o; o += 2 * (size_t)MAX_H;
    o = (o + 3) & ~(size_t)3;
    L.qstage = o; o += ROUTE_QSTAGE;
    L.tile = o;
    o += tile_floats_for(H2);
    L.total = o;
    return L;
}

// K_route_simt runs the tile on warps 0-7 and the quality chains on warp 8,
// side by side.
constexpr int ROUTE_THREADS = SIMT_THREADS + 32;

template <int CPT>
__global__ void __launch_bounds__(ROUTE_THREADS, CPT <= 4 ? 3 : 2) k_route_simt(Model m, Queries q) {
    extern __shared__ float4 sm4[];
    float *sm = reinterpret_cast<float *>(sm4);
    const RouteLayout L = route_layout(m.D, m.M, m.H2);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int D = m.D, M = m.M, F = m.F, QB = L.QB, R = L.R;
    const int q0 = blockIdx.x * QB;
    float *us = sm + L.us, *vs = sm + L.vs, *ol = sm + L.ol, *qual = sm + L.qual;
    float *sp = sm + L.sp, *Cs = sm + L.C, *Us = sm + L.U;

    if (warp < SIMT_THREADS / 32) {
        // the two query slots on two warps (their fp64 chains run side by side)
        if (tid < QB) {
            const int qq = q0 + tid;
            us[tid] = qq < q.Q ? standardise(m.xform[F - 2], (double)q.in_len[qq], m.mu[F - 2],
                                             m.sd[F - 2])
                               : 0.f;
        } else if (tid >= 64 && tid < 64 + QB) {
            const int qi = tid - 64, qq = q0 + qi;
            const float o = qq < q.Q ? q.out_len[qq] : 0.f;
            vs[qi] = qq < q.Q ? standardise(m.xform[F - 1], (double)o, m.mu[F - 1], m.sd[F - 1])
                              : 0.f;
            ol[qi] = o;
        }
        tile_sync();
        RouteRows rows{m.A, D, m.H1};
        pair_mlp<CPT>(m, R, rows, us, vs, sm + L.tile, sm + L.w3, sm + L.w1q, sp);
    } else {
        // quality (QB M <= 64 chains) on the last warp, while the tile runs
        float qv[2];
        quality_group<32, 2>(m, q, q0, QB, sm + L.qstage, ROUTE_QSTAGE, lane, qv);
        if (lane < QB * M) qual[lane] = qv[0];
        if (lane + 32 < QB * M) qual[lane + 32] = qv[1];
    }
    __syncthreads();

    for (int r = tid; r < R; r += ROUTE_THREADS) {
        const int qi = r / D, d = r - qi * D;
        const float *h = sp + m.NH * r;   // TTFT, TPOT (, N_out)
        const float C = __fmaf_rn(m.NH == 3 ? h[2] : ol[qi], h[1], h[0]);
        const float Ql = qual[qi * M + m.dep_model[d]];
        Cs[r] = C;
        Us[r] = __fmaf_rn(-q.lam, C, __fmul_rn(q.wq, Ql));
        if (q.pair_C && q0 + qi < q.Q) q.pair_C[(size_t)(q0 + qi) * D + d] = C;
    }
    if (q.qual_out)
        for (int e = tid; e < QB * M; e += ROUTE_THREADS)
            if (q0 + e / M < q.Q) q.qual_out[(size_t)q0 * M + e] = qual[e];
    __syncthreads();

    for (int qi = warp; qi < QB; qi += ROUTE_THREADS / 32) {
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
// A table block takes an equal run of consecutive entries.

size_t seq_table_floats(int D, int Qs) { return tri_off(D, Qs, Qs); }

// Per-chunk auxiliary arrays (one scratch buffer, seq_aux_floats floats):
// quality [Qs][M], standardised query slots u [Qs] and v [Qs], and, for every
// deployment d and count c = 0 .. Qs of further picks, the standardised
// running count xr [D][Qs + 1] and the layer-1 prefix through slot F - 3
// pre [D][Qs + 1][H1] (the snapshot kernel's chain with running r_d + c).
struct SeqAux {
    float *qual, *us, *vs, *xr, *pre;
};

__host__ __device__ inline SeqAux seq_aux(float *aux, int D, int M, int Qs) {
    SeqAux a;
    a.qual = aux;
    a.us = aux + (size_t)Qs * M;
    a.vs = a.us + Qs;
    a.xr = a.vs + Qs;
    a.pre = a.xr + (((size_t)D * (Qs + 1) + 3) & ~(size_t)3);
    return a;
}

size_t seq_aux_floats(int D, int M, int H1, int Qs) {
    return (size_t)Qs * M + 2 * (size_t)Qs + (((size_t)D * (Qs + 1) + 3) & ~(size_t)3) +
           (size_t)D * (Qs + 1) * H1;
}

// K_seq_prep: the chunk's standardised features and layer-1 prefixes, each
// computed once (double arithmetic is scarce on this GPU, and every table
// block would otherwise repeat it).  Blocks [0, nuv): the query slots; then
// one block per deployment d and run of PREP_COUNTS counts c.
constexpr int PREP_THREADS = 128;
constexpr int PREP_COUNTS = 8;   // counts c per preparation block
__host__ __device__ inline int seq_prep_blocks_per_dep(int Qs) {
    return (Qs + PREP_COUNTS) / PREP_COUNTS;   // counts 0 .. Qs
}

__global__ void __launch_bounds__(PREP_THREADS)
k_seq_prep(Model m, Queries q, int Qs, float *aux, uint16_t *pre_bf, int32_t *dmv) {
    umma::grid_launch_dependents();
    const SeqAux a = seq_aux(aux, m.D, m.M, Qs);
    const int tid = threadIdx.x, F = m.F, P = m.P, H1 = m.H1;
    const int nuv = (2 * Qs + PREP_THREADS - 1) / PREP_THREADS;
    if ((int)blockIdx.x < nuv) {
        const int t = blockIdx.x * PREP_THREADS + tid;
        if (t < Qs) {
            a.us[t] = standardise(m.xform[F - 2], (double)q.in_len[t], m.mu[F - 2], m.sd[F - 2]);
        } else if (t < 2 * Qs) {
            const int i = t - Qs;
            a.vs[i] = standardise(m.xform[F - 1], (double)q.out_len[i], m.mu[F - 1], m.sd[F - 1]);
        }
        return;
    }
    // block: deployment d, counts c0 .. c0 + cn - 1
    const int nc = seq_prep_blocks_per_dep(Qs);
    const int gb = blockIdx.x - nuv, d = gb / nc, c0 = (gb - d * nc) * PREP_COUNTS;
    const int cn = Qs + 1 - c0 < PREP_COUNTS ? Qs + 1 - c0 : PREP_COUNTS;
    const int g0 = d * (Qs + 1) + c0;
    __shared__ float xr[PREP_COUNTS];
    if (tid < cn) {
        const float v = standardise(m.xform[P + 1], (double)(m.running[d] + c0 + tid), m.mu[P + 1],
                                    m.sd[P + 1]);
        xr[tid] = v;
        a.xr[g0 + tid] = v;
        if (dmv) dmv[g0 + tid] = m.dep_model[d];
    } else if (tid < PREP_COUNTS) {
        xr[tid] = 0.f;   // past the last count: computed, never stored
    }
    __syncthreads();
    // continue the chain from slot P + 1 (running) with the deployment's other
    // features, every count of the block at once (W1 read slot-major: a warp's
    // loads of one slot are contiguous)
    const float *x = m.X + (size_t)d * F;
    for (int j = tid; j < H1; j += PREP_THREADS) {
        const float s0 = m.Spre[(size_t)d * H1 + j], w = m.W1T[(size_t)(P + 1) * H1 + j];
        float acc[PREP_COUNTS];
#pragma unroll
        for (int c = 0; c < PREP_COUNTS; ++c) acc[c] = __fmaf_rn(w, xr[c], s0);
        // the remaining slots in order, their weights and features loaded
        // eight at a time ahead of the FMAs
        int k = P + 2;
        for (; k + 8 <= F - 2; k += 8) {
            float wv[8], xv[8];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                wv[t] = m.W1T[(size_t)(k + t) * H1 + j];
                xv[t] = x[k + t];
            }
#pragma unroll
            for (int t = 0; t < 8; ++t)
#pragma unroll
                for (int c = 0; c < PREP_COUNTS; ++c) acc[c] = __fmaf_rn(wv[t], xv[t], acc[c]);
        }
        for (; k < F - 2; ++k) {
            const float wk = m.W1T[(size_t)k * H1 + j], xk = x[k];
#pragma unroll
            for (int c = 0; c < PREP_COUNTS; ++c) acc[c] = __fmaf_rn(wk, xk, acc[c]);
        }
#pragma unroll
        for (int c = 0; c < PREP_COUNTS; ++c) {
            if (c < cn) {
                a.pre[(size_t)(g0 + c) * H1 + j] = acc[c];
                if (pre_bf)
                    pre_bf[(size_t)(g0 + c) * H1 + j] = __bfloat16_as_ushort(__float2bfloat16_rn(acc[c]));
            }
        }
    }
}

// Table rows of one block: row r is table entry t0 + r, i.e. (c, d, i) with
// prefix pre[d][c] and query slot i (decoded into shared memory).
struct FlatRows {
    const float *pre;
    const int *gi, *qi;
    int H1;
    __device__ const float *prefix(int r) const { return pre + (size_t)gi[r] * H1; }
    __device__ int query(int r) const { return qi[r]; }
};

struct SeqLayout {
    size_t us, vs, gi, qi, sp, w3, w1q, tile, total;
};

__host__ __device__ inline SeqLayout seq_layout(int H2) {
    SeqLayout L;
    size_t o = 0;
    L.us = o; o += SEQ_MAX_CHUNK;
    L.vs = o; o += SEQ_MAX_CHUNK;
    L.gi = o; o += TILE_ROWS;
    L.qi = o; o += TILE_ROWS;
    L.sp = o; o += 3 * TILE_ROWS;
    o = (o + 3) & ~(size_t)3;   // W3 rows read as 16-byte vectors
    L.w3 = o; o += 3 * (size_t)H2;
    L.w1q = o; o += 2 * (size_t)MAX_H;
    o = (o + 3) & ~(size_t)3;
    L.tile = o;
    o += tile_floats_for(H2);
    L.total = o;
    return L;
}

// Queries per quality block of the sequential table (at most 256 chains).
__host__ __device__ inline int seq_qual_rows(int M) {
    const int n = SIMT_THREADS / M;
    return n < 1 ? 1 : (n > 8 ? 8 : n);
}

// K_seq_table: blocks [0, nb_qual) compute the chunk's quality; the others
// take rows_per_block consecutive table entries each (the last block fewer),
// so that every SM gets the same number of rows.
template <int CPT>
__global__ void __launch_bounds__(SIMT_THREADS, CPT <= 4 ? 3 : 2)
k_seq_table(Model m, Queries q, int Qs, int nb_qual, int rows_per_block, float *ctab,
            float *aux) {
    extern __shared__ float4 sm4[];
    float *sm = reinterpret_cast<float *>(sm4);
    const int tid = threadIdx.x;
    const int D = m.D, M = m.M;
    const SeqLayout L = seq_layout(m.H2);
    const SeqAux A = seq_aux(aux, D, M, Qs);
    // launched as a programmatic dependent of the preparation kernel: the
    // chain may be scheduled now; the quality blocks need nothing from the
    // preparation kernel, the table blocks wait for it below
    umma::grid_launch_dependents();
    if ((int)blockIdx.x < nb_qual) {
        // quality of the chunk's queries [q0, q0 + nq), staged through the whole
        // shared space
        const int nq = seq_qual_rows(M), q0 = (int)blockIdx.x * nq;
        const float v = quality_staged(m, q, q0, nq, sm, (int)L.total);
        if (tid < nq * M && q0 + tid / M < Qs) A.qual[(size_t)q0 * M + tid] = v;
        return;
    }
    const int T = (int)tri_off(D, Qs, Qs);
    const int t0 = ((int)blockIdx.x - nb_qual) * rows_per_block;
    const int R = min(rows_per_block, T - t0);
    float *us = sm + L.us, *vs = sm + L.vs, *sp = sm + L.sp;
    int *gi = reinterpret_cast<int *>(sm + L.gi), *qi = reinterpret_cast<int *>(sm + L.qi);
    for (int r = tid; r < R; r += SIMT_THREADS) {
        // entry t: the count c with tri_off(c) <= t < tri_off(c + 1), then d and i
        const int t = t0 + r;
        int lo = 0, hi = Qs - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if ((int)tri_off(D, Qs, mid) <= t) lo = mid;
            else hi = mid - 1;
        }
        const int off = t - (int)tri_off(D, Qs, lo), len = Qs - lo, d = off / len;
        gi[r] = d * (Qs + 1) + lo;
        qi[r] = lo + off - d * len;
    }
    // the weights need nothing from the preparation kernel
    pair_mlp_stage<CPT>(m, sm + L.tile, sm + L.w3, sm + L.w1q);
    umma::grid_dependency_wait();    // the preparation kernel's features and prefixes
    for (int i = tid; i < Qs; i += SIMT_THREADS) {
        us[i] = A.us[i];
        vs[i] = A.vs[i];
    }
    __syncthreads();

    FlatRows rows{A.pre, gi, qi, m.H1};
    pair_mlp<CPT>(m, R, rows, us, vs, sm + L.tile, sm + L.w3, sm + L.w1q, sp, true);

    for (int r = tid; r < R; r += SIMT_THREADS) {
        const float *h = sp + m.NH * r;
        ctab[t0 + r] = __fmaf_rn(m.NH == 3 ? h[2] : q.out_len[qi[r]], h[1], h[0]);
    }
}

// Chain shared memory (4-byte words): dep_model and picks [MAX_D] ints each,
// the table [T rounded up to 4] (16-byte aligned), the chunk's quality
// [Qs][M], budgets [Qs] and the walk's outputs (chosen, latency, utility)
// [3][Qs].
constexpr int CHAIN_THREADS = 1024;

__host__ __device__ inline size_t chain_tab_floats(int D, int Qs) {
    return (tri_off(D, Qs, Qs) + 3) & ~(size_t)3;
}

// The decision maker's candidate order as one 40-bit integer: class + 1
// (bits 38-39), the key within the class (bits 6-37: larger U for a
// feasible candidate, smaller C for an infeasible one, as order-preserving
// integers) and 63 - d (bits 0-5), so that the largest value is the best
// candidate and ties go to the lowest deployment.  Same classes as make_cand.
// Written with selects only: the walk is one warp's dependent chain, and a
// divergent branch there costs more than the few extra instructions.
__device__ __forceinline__ uint64_t cand_key(float C, float U, int d, float slo) {
    const bool nan = C != C;
    const bool feas = C <= slo && U == U;       // false for a NaN cost
    const uint32_t kU = order_key(U), kC = ~order_key(C);
    uint32_t key = feas ? kU : kC, cls = feas ? 3u : 2u;
    key = nan ? 1u : key;
    cls = nan ? 1u : cls;
    const uint32_t hi = (cls << 6) | (key >> 26), lo = (key << 6) | (uint32_t)(63 - d);
    return ((uint64_t)hi << 32) | lo;
}

// HI: deployments 32 .. 63 exist (D > 32); without them every lane of the
// walk carries one deployment and the second half of the step is compiled out.
// BIG: only the table's first `tsm` entries (the rows of the first counts)
// fit in shared memory; the walk reads the rest from global memory (L2).
template <bool HI, bool BIG>
__global__ void __launch_bounds__(CHAIN_THREADS)
k_seq_chain(Model m, Queries q, int Qs, const float *ctab, float *aux, const float *qsrc,
            int qstride, int tsm) {
    extern __shared__ float4 sm4[];
    float *sm = reinterpret_cast<float *>(sm4);
    const int tid = threadIdx.x, lane = tid & 31;
    const int D = m.D, M = m.M, F = m.F, H1 = m.H1, P = m.P;
    const SeqAux A = seq_aux(aux, D, M, Qs);
    const size_t T = tri_off(D, Qs, Qs);
    int *dm = reinterpret_cast<int *>(sm), *cnt = dm + MAX_D;
    float *tab = sm + 2 * MAX_D;
    float *qs = tab + (BIG ? (size_t)tsm : chain_tab_floats(D, Qs)), *slo = qs + (size_t)Qs * M;
    const size_t Ts = BIG ? (size_t)tsm : T;    // entries staged in shared memory
    // entry e of the table: shared memory, or (BIG, e >= tsm) global memory
    auto at = [&](int e) -> float {
        if constexpr (BIG) {
            return e < tsm ? tab[e] : __ldcg(ctab + e);
        } else {
            return tab[e];
        }
    };
    float *o_lat = slo + Qs, *o_util = o_lat + Qs;
    int *o_ch = reinterpret_cast<int *>(o_util + Qs);

    // launched as a programmatic dependent of the table kernel: budgets and
    // the model map first, then wait for the table (and, through it, for the
    // preparation kernel)
    for (int i = tid; i < Qs; i += CHAIN_THREADS) slo[i] = query_budget(q, i);
    for (int e = tid; e < D; e += CHAIN_THREADS) dm[e] = m.dep_model[e];
    umma::grid_dependency_wait();
    const uint32_t tab_s = (uint32_t)__cvta_generic_to_shared(tab);
    // the triangular table, by 16-byte asynchronous copies (both sides
    // 16-byte aligned)
    for (size_t e = tid; e < Ts / 4; e += CHAIN_THREADS)
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(tab_s + (uint32_t)(16 * e)),
                     "l"(__cvta_generic_to_global(ctab + 4 * e))
                     : "memory");
    for (size_t e = Ts / 4 * 4 + tid; e < Ts; e += CHAIN_THREADS) tab[e] = __ldcg(ctab + e);
    asm volatile("cp.async.commit_group;" ::: "memory");
    for (int e = tid; e < Qs * M; e += CHAIN_THREADS) {
        const int i = e / M;
        qs[e] = __ldcg(qsrc + (size_t)i * qstride + e - i * M);
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();

    if (tid < 32) {
        // The walk.  Lane l holds deployments d0 = l and d1 = l + 32 with their
        // picks so far (c0, c1); entry (c, d, i) is tab[tab_row(c, d) + i].
        // While step i is decided, step i + 1's entries at the current count
        // and at one more pick are loaded and turned into candidate keys, so a
        // step is a choice between two ready keys, a 64-bit max over the warp
        // (two reductions) and the winner's index from the low bits.  Lanes
        // without a deployment shadow deployment D - 1 (valid addresses) and
        // keep key 0, below every candidate; the row of one more pick advances
        // by D (Qs - c) - d - 1 after a pick.  The step has no branch: the last
        // step loads its own column again (valid entries, unused), and a pick
        // moves the rows by selects.
        const unsigned full = 0xffffffffu;
        const int d0 = lane, d1 = lane + 32;
        const bool h0 = d0 < D, h1 = HI && d1 < D;
        const int e0 = h0 ? d0 : D - 1, e1 = h1 ? d1 : D - 1;
        const int m0 = dm[e0], m1 = HI ? dm[e1] : 0;
        const float lam = q.lam, wq = q.wq;
        int c0 = 0, c1 = 0;
        int r0 = tab_row(D, Qs, 0, e0), r1 = HI ? tab_row(D, Qs, 0, e1) : 0;
        int r0p = r0 + D * Qs - e0 - 1, r1p = HI ? r1 + D * Qs - e1 - 1 : 0;
        // this step's candidate of each deployment: cost, utility, key
        float C0, U0, C1 = 0.f, U1 = 0.f;
        uint64_t K0, K1 = 0;
        {
            const float b = slo[0];
            C0 = at(r0);
            U0 = __fmaf_rn(-lam, C0, __fmul_rn(wq, qs[m0]));
            K0 = cand_key(C0, U0, d0, b);
            K0 = h0 ? K0 : 0;
            if (HI) {
                C1 = at(r1);
                U1 = __fmaf_rn(-lam, C1, __fmul_rn(wq, qs[m1]));
                K1 = cand_key(C1, U1, d1, b);
                K1 = h1 ? K1 : 0;
            }
        }
        for (int i = 0; i < Qs; ++i) {
            // step j = i + 1's candidates: s = same count, p = after one more
            // pick (at the last step, j = i: this step's entries again)
            const bool more = i + 1 < Qs;
            const int j = more ? i + 1 : i;
            const float b = slo[j];
            const float wQ0 = __fmul_rn(wq, qs[j * M + m0]);
            const float C0s = at(r0 + j), C0p = at((more ? r0p : r0) + j);
            const float U0s = __fmaf_rn(-lam, C0s, wQ0), U0p = __fmaf_rn(-lam, C0p, wQ0);
            uint64_t K0s = cand_key(C0s, U0s, d0, b), K0p = cand_key(C0p, U0p, d0, b);
            K0s = h0 ? K0s : 0;
            K0p = h0 ? K0p : 0;
            float C1s = 0.f, U1s = 0.f, C1p = 0.f, U1p = 0.f;
            uint64_t K1s = 0, K1p = 0;
            if (HI) {
                const float wQ1 = __fmul_rn(wq, qs[j * M + m1]);
                C1s = at(r1 + j);
                C1p = at((more ? r1p : r1) + j);
                U1s = __fmaf_rn(-lam, C1s, wQ1);
                U1p = __fmaf_rn(-lam, C1p, wQ1);
                K1s = cand_key(C1s, U1s, d1, b);
                K1p = cand_key(C1p, U1p, d1, b);
                K1s = h1 ? K1s : 0;
                K1p = h1 ? K1p : 0;
            }
            // step i: the warp's largest key
            const uint64_t kl = HI && K1 > K0 ? K1 : K0;
            const uint32_t hi = __reduce_max_sync(full, (uint32_t)(kl >> 32));
            const uint32_t lo =
                __reduce_max_sync(full, (uint32_t)(kl >> 32) == hi ? (uint32_t)kl : 0u);
            const int wd = 63 - (int)(lo & 63u);
            const bool ok = (hi >> 6) >= 2u;    // class feasible or infeasible, not NaN
            const bool p0 = ok && wd == d0, p1 = HI && ok && wd == d1;
            if (lane == 0) o_ch[i] = ok ? wd : -1;
            if (p0 || p1) {
                o_lat[i] = p0 ? C0 : C1;
                o_util[i] = p0 ? U0 : U1;
            }
            if (!ok && lane == 0) {
                o_lat[i] = __int_as_float(0x7fc00000);
                o_util[i] = __int_as_float(0x7fc00000);
            }
            c0 += p0 ? 1 : 0;
            const int n0 = r0p + D * (Qs - c0) - e0 - 1;
            r0 = p0 ? r0p : r0;
            r0p = p0 ? n0 : r0p;
            C0 = p0 ? C0p : C0s;
            U0 = p0 ? U0p : U0s;
            K0 = p0 ? K0p : K0s;
            if (HI) {
                c1 += p1 ? 1 : 0;
                const int n1 = r1p + D * (Qs - c1) - e1 - 1;
                r1 = p1 ? r1p : r1;
                r1p = p1 ? n1 : r1p;
                C1 = p1 ? C1p : C1s;
                U1 = p1 ? U1p : U1s;
                K1 = p1 ? K1p : K1s;
            }
        }
        if (h0) cnt[d0] = c0;
        if (h1) cnt[d1] = c1;
    }
    __syncthreads();
    for (int i = tid; i < Qs; i += CHAIN_THREADS) {
        q.lat[i] = o_lat[i];
        q.util[i] = o_util[i];
        if (q.inputs_host) {
            // outputs in host memory: the host may poll chosen with acquire
            // loads, so it is stored last, with release semantics at system
            // scope
            asm volatile("st.release.sys.global.b32 [%0], %1;" ::"l"(q.chosen + i), "r"(o_ch[i])
                         : "memory");
        } else {
            q.chosen[i] = o_ch[i];
        }
    }
    __syncthreads();

    // persist the picks and refresh the state they touch: the standardised
    // running count and the layer-1 prefix are the preparation kernel's values
    // for the final count
    for (int d = tid; d < D; d += CHAIN_THREADS) {
        m.running[d] += cnt[d];
        m.X[(size_t)d * F + P + 1] = A.xr[(size_t)d * (Qs + 1) + cnt[d]];
    }
    for (int e = tid; e < D * H1; e += CHAIN_THREADS) {
        const int d = e / H1, j = e - d * H1;
        const float v = A.pre[((size_t)d * (Qs + 1) + cnt[d]) * H1 + j];
        m.A[e] = v;
        m.Abf[e] = __bfloat16_as_ushort(__float2bfloat16_rn(v));
    }
}

// ---------------------------------------------------------------------------
// K_route_pairs: the small-batch (latency) variant.  The (query, deployment)
// pairs p = qq D + d are taken in groups of PAIR_G consecutive pairs, and a
// group's layer 2 is split by columns over ncb column blocks, in one of two
// shapes.  Split (PAIR_COLS columns per block, when groups are many): each
// block stages its W2 columns k-major and the group's layer-1 rows in shared
// memory, runs its columns' serial chains (warp w: columns 4w .. 4w + 3,
// lane: pair, so a W2 load is a broadcast) and stores them to a scratch h2
// [groups][H2][PAIR_G].  Fused (PAIR_FUSED_COLS columns per block, when every
// block of the grid has an SM of its own, e.g. one query): each block stages
// its W2 rows, the pairs' deployment prefixes and W1's query columns, and
// rebuilds every layer-1 unit inside the layer-2 chains (warp w: columns 2w,
// 2w + 1), storing h2 rows [groups][PAIR_G][H2].  The last column block of a
// group (arrival counter, self-resetting) copies the group's h2 back with
// 16-byte async copies and runs the head chains and the cost of Eq. 2.
// Quality blocks run the per-(query, model) chains from shared memory.  A
// query is decided by the block that completes its count of D pairs and
// qblocks quality blocks (self-resetting).  Same canonical order as the
// kernels above in both shapes: every chain is the same sequence of roundings.

struct PairArgs {
    float *pairC;       // [Q][D] scratch
    float *qualS;       // [Q][M] scratch
    float *h2;          // [groups][H2][PAIR_G] scratch
    int32_t *count;     // [Q] arrivals, zero between calls
    int32_t *gcount;    // [groups] column-block arrivals, zero between calls
    int qblocks;        // quality blocks per query
    int ncb;            // column blocks per group
    int cols;           // layer-2 columns per column block: PAIR_FUSED_COLS or PAIR_COLS
};

constexpr int PAIR_MPB = 8;    // models per quality block
constexpr int PAIR_G = 32;     // pairs per group
constexpr int PAIR_COLS = 32;  // layer-2 columns per block, split shape
constexpr int PAIR_FUSED_COLS = 8;   // layer-2 columns per block, fused shape

__device__ void pair_select(const Model &m, const Queries &q, const PairArgs &a, int qq) {
    // one warp: utility, SLO mask, argmax over the query's stored costs
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
        q.lat[qq] = ok ? best.C : __int_as_float(0x7fc00000);
        q.util[qq] = ok ? best.U : __int_as_float(0x7fc00000);
        a.count[qq] = 0;
        const int32_t v = ok ? best.d : -1;
        if (q.inputs_host) {
            // outputs in mapped host memory: the host polls chosen with
            // acquire loads, so chosen is stored with release semantics at
            // system scope, after latency and utility
            asm volatile("st.release.sys.global.b32 [%0], %1;" ::"l"(q.chosen + qq), "r"(v)
                         : "memory");
        } else {
            q.chosen[qq] = v;
        }
    }
}

__host__ __device__ inline int pair_groups(int npair) { return (npair + PAIR_G - 1) / PAIR_G; }

// Shared-memory layout of a fused-shape column block (floats; every region
// 16-byte aligned), and of the group's last block over the same space.  Rows
// that a warp reads as 16-byte vectors, one row per lane, have a stride of an
// odd number of 16-byte units, so that the 8 lanes of each wavefront fall in
// distinct banks.
struct PairSmem {
    int ldk, lda, ld2;          // W2 / W1-column row stride; prefix and layer-2 row strides
    int w2, as, w1;             // column block: W2 rows, prefix rows, W1's query columns
    int h2, w3;                 // last block: layer-2 rows, W3
    int total;
};

__host__ __device__ inline PairSmem pair_smem(int H1, int H2) {
    PairSmem L;
    L.ldk = (H1 + 3) & ~3;
    L.lda = (H1 & 3) == 0 ? odd_units(H1) : H1;
    L.ld2 = odd_units(H2);
    int o = 3 * PAIR_G;                     // qu, qv, qo
    L.w2 = o;
    o += PAIR_FUSED_COLS * L.ldk;
    L.as = o;
    o += (PAIR_G * L.lda + 3) & ~3;
    L.w1 = o;
    o += 2 * L.ldk;
    L.h2 = 3 * PAIR_G;
    L.w3 = L.h2 + PAIR_G * L.ld2;
    const int fin = L.w3 + 3 * H2;
    L.total = o > fin ? o : fin;
    return L;
}

// Layers 1 and 2 of pair p (deployment prefix row ar, query slots u, v) for
// the block's columns c0, c0 + 1: each layer-1 unit is rebuilt where
// layer 2 consumes it (same two FMAs and ReLU as everywhere), and each
// layer-2 chain is bias, then k ascending.  Shared-memory operands come as
// 16-byte vectors, eight k at a time ahead of their FMAs: on this GPU a
// chain step waiting on its own shared loads costs several times its FMA.
// Stores relu(h2) into the group's scratch rows [PAIR_G][H2].
__device__ __forceinline__ void pair_layers(const Model &m, const PairArgs &a, const PairSmem &L,
                                            const float *w2c, const float *ar, const float *w1s,
                                            float u, float v, int g, int n0, int nb, int c0,
                                            int p) {
    constexpr int NC = 2;
    const int H1 = m.H1, H2 = m.H2;
    float acc[NC];
    const float *wr[NC];
#pragma unroll
    for (int j = 0; j < NC; ++j) {
        const int c = c0 + j;
        acc[j] = c < nb ? m.b2[n0 + c] : 0.f;
        wr[j] = w2c + (size_t)(c < nb ? c : 0) * L.ldk;
    }
    const float *wi = w1s, *wo = w1s + L.ldk;
    int k = 0;
    if ((H1 & 3) == 0) {
        for (; k + 8 <= H1; k += 8) {
            const float4 a0 = *reinterpret_cast<const float4 *>(ar + k);
            const float4 a1 = *reinterpret_cast<const float4 *>(ar + k + 4);
            const float4 i0 = *reinterpret_cast<const float4 *>(wi + k);
            const float4 i1 = *reinterpret_cast<const float4 *>(wi + k + 4);
            const float4 o0 = *reinterpret_cast<const float4 *>(wo + k);
            const float4 o1 = *reinterpret_cast<const float4 *>(wo + k + 4);
            float4 w0[NC], w1[NC];
#pragma unroll
            for (int j = 0; j < NC; ++j) {
                w0[j] = *reinterpret_cast<const float4 *>(wr[j] + k);
                w1[j] = *reinterpret_cast<const float4 *>(wr[j] + k + 4);
            }
            const float av[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
            const float iv[8] = {i0.x, i0.y, i0.z, i0.w, i1.x, i1.y, i1.z, i1.w};
            const float ov[8] = {o0.x, o0.y, o0.z, o0.w, o1.x, o1.y, o1.z, o1.w};
            float h[8];
#pragma unroll
            for (int t = 0; t < 8; ++t) {
                const float x = __fmaf_rn(ov[t], v, __fmaf_rn(iv[t], u, av[t]));
                h[t] = x > 0.f ? x : 0.f;
            }
#pragma unroll
            for (int j = 0; j < NC; ++j) {
                acc[j] = __fmaf_rn(w0[j].x, h[0], acc[j]);
                acc[j] = __fmaf_rn(w0[j].y, h[1], acc[j]);
                acc[j] = __fmaf_rn(w0[j].z, h[2], acc[j]);
                acc[j] = __fmaf_rn(w0[j].w, h[3], acc[j]);
                acc[j] = __fmaf_rn(w1[j].x, h[4], acc[j]);
                acc[j] = __fmaf_rn(w1[j].y, h[5], acc[j]);
                acc[j] = __fmaf_rn(w1[j].z, h[6], acc[j]);
                acc[j] = __fmaf_rn(w1[j].w, h[7], acc[j]);
            }
        }
    }
    for (; k < H1; ++k) {
        const float x = __fmaf_rn(wo[k], v, __fmaf_rn(wi[k], u, ar[k]));
        const float h = x > 0.f ? x : 0.f;
#pragma unroll
        for (int j = 0; j < NC; ++j) acc[j] = __fmaf_rn(wr[j][k], h, acc[j]);
    }
    float *dst = a.h2 + ((size_t)g * PAIR_G + p) * H2 + n0;
#pragma unroll
    for (int j = 0; j < NC; ++j)
        if (c0 + j < nb) dst[c0 + j] = acc[j] > 0.f ? acc[j] : 0.f;
    __threadfence();   // before the group's arrival
}

// The decision for each query of a group: its pairs arrive; the warp that
// completes the query's count (pairs and quality blocks) decides it.
__device__ __forceinline__ void pair_decide(const Model &m, const Queries &q, const PairArgs &a,
                                            int p0, int np, int q0, int nq) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, D = m.D;
    for (int ql = warp; ql < nq; ql += SIMT_THREADS / 32) {
        const int qq = q0 + ql;
        const int cnt = min(p0 + np, (qq + 1) * D) - max(p0, qq * D);
        int done = 0;
        if (lane == 0) done = atomicAdd(&a.count[qq], cnt) + cnt == D + a.qblocks;
        done = __shfl_sync(0xffffffffu, done, 0);
        if (done) {
            __threadfence();
            pair_select(m, q, a, qq);
        }
    }
}

// Column block, split shape (many groups): W2 columns n0 .. n0 + 31 k-major,
// layer 1 written once per (pair, unit), layer-2 chains of 4 columns per warp
// (lane = pair), h2 scratch [groups][H2][PAIR_G]; the group's last column
// block runs the heads.
__device__ __forceinline__ void pair_cols_split(const Model &m, const Queries &q, const PairArgs &a,
                                             float *sm, int *s_last_p) {
    int &s_last = *s_last_p;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int F = m.F, H1 = m.H1, H2 = m.H2, D = m.D;
    const int npair = q.Q * D;
    const int g = blockIdx.x / a.ncb, cb = blockIdx.x - g * a.ncb;
    const int p0 = g * PAIR_G, np = min(PAIR_G, npair - p0);
    const int q0 = p0 / D, nq = (p0 + np - 1) / D - q0 + 1;   // queries touched, <= PAIR_G
    const int n0 = cb * PAIR_COLS, nb = min(PAIR_COLS, H2 - n0);
    float *qu = sm, *qv = sm + PAIR_G, *qo = sm + 2 * PAIR_G;
    float *w2s = sm + 3 * PAIR_G;               // [H1][PAIR_COLS]
    const int ld1 = H1 | 1;                     // odd: rows of 4 pairs in distinct banks
    float *h1s = w2s + (size_t)H1 * PAIR_COLS;  // [PAIR_G][ld1]
    // W2 columns n0 .. n0 + 31 of every k (only within the padded row)
    {
        const int c4n = min(PAIR_COLS, m.H2p - n0) >> 2;
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(w2s);
        for (int e = tid; e < H1 * c4n; e += SIMT_THREADS) {
            const int k = e / c4n, c4 = e - k * c4n;
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                             base + (uint32_t)(4 * (k * PAIR_COLS + 4 * c4))),
                         "l"(__cvta_generic_to_global(m.W2T + (size_t)k * m.H2p + n0 + 4 * c4)) : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    // the query slots of the group's queries (fp64 chains side by side)
    if (tid < nq) {
        qu[tid] = standardise(m.xform[F - 2], (double)q.in_len[q0 + tid], m.mu[F - 2], m.sd[F - 2]);
    } else if (tid >= 32 && tid < 32 + nq) {
        const float o = q.out_len[q0 + tid - 32];
        qv[tid - 32] = standardise(m.xform[F - 1], (double)o, m.mu[F - 1], m.sd[F - 1]);
        qo[tid - 32] = o;
    }
    // this thread's unit k of layer 1 for every pair of the group: the
    // prefix loads first, all in flight together
    const int k = tid;
    const bool hk = k < H1;
    float av[PAIR_G];
    {
        int qq = q0, d = p0 - q0 * D;
#pragma unroll
        for (int p = 0; p < PAIR_G; ++p) {
            av[p] = hk && p < np ? m.A[(size_t)d * H1 + k] : 0.f;
            if (++d == D) {
                d = 0;
                ++qq;
            }
        }
    }
    const float wi = hk ? m.W1T[(size_t)(F - 2) * H1 + k] : 0.f;
    const float wo = hk ? m.W1T[(size_t)(F - 1) * H1 + k] : 0.f;
    __syncthreads();
    if (hk) {
        int ql = 0, d = p0 - q0 * D;
#pragma unroll
        for (int p = 0; p < PAIR_G; ++p) {
            if (p < np) {
                float x = __fmaf_rn(wi, qu[ql], av[p]);
                x = __fmaf_rn(wo, qv[ql], x);
                h1s[p * ld1 + k] = x > 0.f ? x : 0.f;
            }
            if (++d == D) {
                d = 0;
                ++ql;
            }
        }
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
    // layer 2: thread (pair p = lane, columns c .. c + 3 of warp w), serial over k
    {
        const int p = lane, c = 4 * warp;
        if (p < np && c < nb) {
            float acc[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) acc[j] = c + j < nb ? m.b2[n0 + c + j] : 0.f;
            const float *hr = h1s + p * ld1;
            const float *wr = w2s + c;
#pragma unroll 8
            for (int kk = 0; kk < H1; ++kk) {
                const float4 w = *reinterpret_cast<const float4 *>(wr + kk * PAIR_COLS);
                const float h = hr[kk];
                acc[0] = __fmaf_rn(w.x, h, acc[0]);
                acc[1] = __fmaf_rn(w.y, h, acc[1]);
                acc[2] = __fmaf_rn(w.z, h, acc[2]);
                acc[3] = __fmaf_rn(w.w, h, acc[3]);
            }
            float *dst = a.h2 + ((size_t)g * H2 + n0 + c) * PAIR_G + p;
#pragma unroll
            for (int j = 0; j < 4; ++j)
                if (c + j < nb) dst[j * PAIR_G] = acc[j] > 0.f ? acc[j] : 0.f;
            __threadfence();   // before the group's arrival below
        }
    }
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        s_last = atomicAdd(&a.gcount[g], 1) == a.ncb - 1;
    }
    __syncthreads();
    if (!s_last) return;
    // the group's last column block: heads and cost of every pair
    __threadfence();
    float *h2s = w2s;                            // [H2][PAIR_G]
    float *w3s = h2s + (size_t)H2 * PAIR_G;      // [NH][H2]
    {
        // the group's whole block (rows of pairs past np are not read),
        // L2 to shared memory by 16-byte copies that skip L1
        const uint32_t base = (uint32_t)__cvta_generic_to_shared(h2s);
        const float *src = a.h2 + (size_t)g * H2 * PAIR_G;
        for (int e = tid; e < H2 * PAIR_G / 4; e += SIMT_THREADS)
            asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(base + 16u * e),
                         "l"(__cvta_generic_to_global(src + 4 * e)) : "memory");
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    for (int i = tid; i < m.NH * H2; i += SIMT_THREADS) w3s[i] = m.W3[i];
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
    __shared__ float hd[PAIR_G * 3];
    if (warp < m.NH) {
        // head o = warp of pair p = lane: W3 reads are broadcasts, h2
        // reads consecutive words
        const int o = warp, p = lane;
        const float *w3 = w3s + (size_t)o * H2;
        float z = m.b3[o];
#pragma unroll 8
        for (int n = 0; n < H2; ++n) z = __fmaf_rn(w3[n], h2s[n * PAIR_G + p], z);
        if (p < np) hd[p * m.NH + o] = softplus_c(z);
    }
    __syncthreads();
    for (int p = tid; p < np; p += SIMT_THREADS) {
        const int qq = (p0 + p) / D, NH = m.NH;
        a.pairC[p0 + p] =
            __fmaf_rn(NH == 3 ? hd[p * NH + 2] : qo[qq - q0], hd[p * NH + 1], hd[p * NH]);
    }
    if (tid == 0) a.gcount[g] = 0;
    __threadfence();
    __syncthreads();
    pair_decide(m, q, a, p0, np, q0, nq);
}

// Column block, fused shape (few groups, so that every block has an SM of
// its own): the block's 8 W2 rows, each pair's deployment prefix row and
// W1's query columns staged by asynchronous copies behind the query slots'
// loads; each layer-1 unit rebuilt where layer 2 consumes it (no layer-1
// pass); h2 scratch [groups][PAIR_G][H2], a row per pair, so that the last
// block's head chains read it as vectors.
__device__ __forceinline__ void pair_cols_fused(const Model &m, const Queries &q, const PairArgs &a,
                                             float *sm, int *s_last_p) {
    int &s_last = *s_last_p;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int F = m.F, H1 = m.H1, H2 = m.H2, D = m.D;
    const int npair = q.Q * D;
    const int g = blockIdx.x / a.ncb, cb = blockIdx.x - g * a.ncb;
    const int p0 = g * PAIR_G, np = min(PAIR_G, npair - p0);
    const int q0 = p0 / D, nq = (p0 + np - 1) / D - q0 + 1;   // queries touched, <= PAIR_G
    const int cols = a.cols, n0 = cb * cols, nb = min(cols, H2 - n0);
    const PairSmem L = pair_smem(H1, H2);
    float *qu = sm, *qv = sm + PAIR_G, *qo = sm + 2 * PAIR_G;
    float *w2c = sm + L.w2;    // [cols][ldk]: W2 rows n0 .. n0 + cols - 1
    float *as = sm + L.as;     // [PAIR_G][lda]: each pair's deployment prefix
    float *w1s = sm + L.w1;    // [2][ldk]: W1's two query columns
    // the query slots' raw lengths first: their double-precision chains below
    // are this block's longest wait
    float iv = 0.f, ov = 0.f;
    if (tid < nq) iv = q.in_len[q0 + tid];
    else if (tid >= 32 && tid < 32 + nq) ov = q.out_len[q0 + tid - 32];
    {
        // pair p of the group is deployment (p0 + p) mod D; 16-byte copies
        // where the rows allow, else 4-byte ones
        const uint32_t wb = (uint32_t)__cvta_generic_to_shared(w2c);
        const uint32_t ab = (uint32_t)__cvta_generic_to_shared(as);
        const int d0 = p0 - q0 * D;
        if ((H1 & 3) == 0) {
            const int r4 = H1 >> 2;
            for (int e = tid; e < nb * r4; e += SIMT_THREADS) {
                const int c = e / r4, j = e - c * r4;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                                 wb + (uint32_t)(4 * (c * L.ldk + 4 * j))),
                             "l"(__cvta_generic_to_global(m.W2 + (size_t)(n0 + c) * H1 + 4 * j)) : "memory");
            }
            for (int e = tid; e < np * r4; e += SIMT_THREADS) {
                const int p = e / r4, j = e - p * r4;
                int d = d0 + p;
                d -= (d / D) * D;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                                 ab + (uint32_t)(4 * (p * L.lda + 4 * j))),
                             "l"(__cvta_generic_to_global(m.A + (size_t)d * H1 + 4 * j)) : "memory");
            }
        } else {
            for (int e = tid; e < nb * H1; e += SIMT_THREADS) {
                const int c = e / H1, j = e - c * H1;
                asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                                 wb + (uint32_t)(4 * (c * L.ldk + j))),
                             "l"(__cvta_generic_to_global(m.W2 + (size_t)(n0 + c) * H1 + j)) : "memory");
            }
            for (int e = tid; e < np * H1; e += SIMT_THREADS) {
                const int p = e / H1, j = e - p * H1;
                int d = d0 + p;
                d -= (d / D) * D;
                asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                                 ab + (uint32_t)(4 * (p * L.lda + j))),
                             "l"(__cvta_generic_to_global(m.A + (size_t)d * H1 + j)) : "memory");
            }
        }
        const uint32_t w1b = (uint32_t)__cvta_generic_to_shared(w1s);
        for (int e = tid; e < 2 * H1; e += SIMT_THREADS) {
            const int r = e / H1, j = e - r * H1;
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(
                             w1b + (uint32_t)(4 * (r * L.ldk + j))),
                         "l"(__cvta_generic_to_global(m.W1T + (size_t)(F - 2 + r) * H1 + j)) : "memory");
        }
        asm volatile("cp.async.commit_group;" ::: "memory");
    }
    // the query slots of the group's queries (fp64 chains side by side)
    if (tid < nq) {
        qu[tid] = standardise(m.xform[F - 2], (double)iv, m.mu[F - 2], m.sd[F - 2]);
    } else if (tid >= 32 && tid < 32 + nq) {
        qv[tid - 32] = standardise(m.xform[F - 1], (double)ov, m.mu[F - 1], m.sd[F - 1]);
        qo[tid - 32] = ov;
    }
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
    // layers 1 and 2: lane = pair p, warp w = columns 2w, 2w + 1
    if (lane < np && 2 * warp < nb) {
        const int p = lane, ql = (p0 + p) / D - q0;
        pair_layers(m, a, L, w2c, as + (size_t)p * L.lda, w1s, qu[ql], qv[ql], g, n0, nb,
                    2 * warp, p);
    }
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        s_last = atomicAdd(&a.gcount[g], 1) == a.ncb - 1;
    }
    __syncthreads();
    if (!s_last) return;
    // the group's last column block: heads and cost of every pair
    __threadfence();
    float *h2s = sm + L.h2;     // [PAIR_G][ld2]: layer 2, a row per pair
    float *w3s = sm + L.w3;     // [NH][H2]
    {
        // the group's rows, L2 to shared memory by copies that skip L1
        const float *src = a.h2 + (size_t)g * PAIR_G * H2;
        if ((H2 & 3) == 0) {
            const uint32_t base = (uint32_t)__cvta_generic_to_shared(h2s);
            const int r4 = H2 >> 2;
            for (int e = tid; e < np * r4; e += SIMT_THREADS) {
                const int p = e / r4, j = e - p * r4;
                asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                                 base + (uint32_t)(4 * (p * L.ld2 + 4 * j))),
                             "l"(__cvta_generic_to_global(src + (size_t)p * H2 + 4 * j)) : "memory");
            }
            asm volatile("cp.async.commit_group;" ::: "memory");
        } else {
            for (int e = tid; e < np * H2; e += SIMT_THREADS) {
                const int p = e / H2, j = e - p * H2;
                h2s[p * L.ld2 + j] = __ldcg(src + (size_t)p * H2 + j);
            }
        }
    }
    for (int i = tid; i < m.NH * H2; i += SIMT_THREADS) w3s[i] = m.W3[i];
    asm volatile("cp.async.wait_all;" ::: "memory");
    __syncthreads();
    __shared__ float hd[PAIR_G * 3];
    if (warp < m.NH && lane < np) {
        // head o = warp, pair p = lane: W3 reads are broadcasts, each lane
        // reads its own row of layer 2, four n per vector
        const int o = warp, p = lane;
        const float *w3 = w3s + (size_t)o * H2, *hr = h2s + (size_t)p * L.ld2;
        float z = m.b3[o];
        int n = 0;
        if ((H2 & 3) == 0) {
            for (; n + 8 <= H2; n += 8) {
                const float4 h0 = *reinterpret_cast<const float4 *>(hr + n);
                const float4 h1 = *reinterpret_cast<const float4 *>(hr + n + 4);
                const float4 v0 = *reinterpret_cast<const float4 *>(w3 + n);
                const float4 v1 = *reinterpret_cast<const float4 *>(w3 + n + 4);
                z = __fmaf_rn(v0.x, h0.x, z);
                z = __fmaf_rn(v0.y, h0.y, z);
                z = __fmaf_rn(v0.z, h0.z, z);
                z = __fmaf_rn(v0.w, h0.w, z);
                z = __fmaf_rn(v1.x, h1.x, z);
                z = __fmaf_rn(v1.y, h1.y, z);
                z = __fmaf_rn(v1.z, h1.z, z);
                z = __fmaf_rn(v1.w, h1.w, z);
            }
        }
        for (; n < H2; ++n) z = __fmaf_rn(w3[n], hr[n], z);
        hd[p * m.NH + o] = softplus_c(z);
    }
    __syncthreads();
    for (int p = tid; p < np; p += SIMT_THREADS) {
        const int qq = (p0 + p) / D, NH = m.NH;
        a.pairC[p0 + p] =
            __fmaf_rn(NH == 3 ? hd[p * NH + 2] : qo[qq - q0], hd[p * NH + 1], hd[p * NH]);
    }
    if (tid == 0) a.gcount[g] = 0;
    __threadfence();
    __syncthreads();
    pair_decide(m, q, a, p0, np, q0, nq);
}

__global__ void __launch_bounds__(SIMT_THREADS) k_route_pairs(Model m, Queries q, PairArgs a) {
    extern __shared__ float4 sm4[];   // 16-byte aligned: operands arrive as 16-byte copies
    float *sm = reinterpret_cast<float *>(sm4);
    __shared__ int s_last;
    const int tid = threadIdx.x;
    const int D = m.D, M = m.M;
    const int npair = q.Q * D, ncolb = pair_groups(npair) * a.ncb;
    if ((int)blockIdx.x < ncolb) {
        if (a.cols == PAIR_COLS) pair_cols_split(m, q, a, sm, &s_last);
        else pair_cols_fused(m, q, a, sm, &s_last);
        return;
    }
    // quality of models [m0, m0 + PAIR_MPB) for one query
    const int b = blockIdx.x - ncolb;
    const int qq = b / a.qblocks;
    const int m0 = (b - qq * a.qblocks) * PAIR_MPB, mn = min(PAIR_MPB, M - m0), E = m.E;
    // emb row [E] and the block's model columns as [E / 4][mn][4] (E is a
    // multiple of 8), so that a chain reads 4 consecutive k of its column as
    // one 16-byte load and the mn chains' loads fall in distinct banks; a
    // thread's staging loads are issued before its stores
    float *er = sm, *mb = sm + E;
    const size_t row = (size_t)qq * E;
    for (int k0 = 0; k0 < E; k0 += SIMT_THREADS) {
        const int k = k0 + tid;
        const bool ok = k < E;
        float v[PAIR_MPB];
        const float ev = ok ? emb_at(q.emb, q.emb_bf16, row + k) : 0.f;
#pragma unroll
        for (int j = 0; j < PAIR_MPB; ++j) v[j] = ok && j < mn ? m.memb[(size_t)k * M + m0 + j] : 0.f;
        if (ok) {
            er[k] = ev;
#pragma unroll
            for (int j = 0; j < PAIR_MPB; ++j)
                if (j < mn) mb[((size_t)(k >> 2) * mn + j) * 4 + (k & 3)] = v[j];
        }
    }
    __syncthreads();
    if (tid < mn) {
        const float4 *c = reinterpret_cast<const float4 *>(mb) + tid;
        const float4 *e4 = reinterpret_cast<const float4 *>(er);
        float s = 0.f;
        // E is a multiple of 8: two 4-term groups' operands, then their FMAs
        for (int k4 = 0; k4 < E / 4; k4 += 2) {
            const float4 x0 = e4[k4], y0 = c[(size_t)k4 * mn];
            const float4 x1 = e4[k4 + 1], y1 = c[(size_t)(k4 + 1) * mn];
            s = __fmaf_rn(x0.x, y0.x, s);
            s = __fmaf_rn(x0.y, y0.y, s);
            s = __fmaf_rn(x0.z, y0.z, s);
            s = __fmaf_rn(x0.w, y0.w, s);
            s = __fmaf_rn(x1.x, y1.x, s);
            s = __fmaf_rn(x1.y, y1.y, s);
            s = __fmaf_rn(x1.z, y1.z, s);
            s = __fmaf_rn(x1.w, y1.w, s);
        }
        a.qualS[(size_t)qq * M + m0 + tid] = sigmoid_c(s);
        __threadfence();
    }
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        s_last = atomicAdd(&a.count[qq], 1) + 1 == D + a.qblocks;
    }
    __syncthreads();
    if (s_last && tid < 32) {
        __threadfence();
        pair_select(m, q, a, qq);
    }
}

// ---------------------------------------------------------------------------
// K_select_multi: the decision maker for several lambdas over stored scores.
// One warp per query: lane l holds deployments l and l + 32 (D <= 64), loads
// their costs and quality once, and for every lambda forms each candidate's
// 40-bit key (the candidate order of the sequential chain, the same order as
// make_cand / better) and takes the warp's largest with two 32-bit
// reductions; lane k keeps lambda k's decision: 55 us for 8 lambdas over
// 65,536 queries at D = 64 on GB300.  (A warp per (query, lambda), each with
// its own warp reduction, took ~115 us; a thread per query with a running
// best per lambda 99 us: too few warps, and divergent comparisons.)
__global__ void __launch_bounds__(SIMT_THREADS)
k_select_multi(Model m, Queries q, const float *C, const float *qual, int qstride, Lambdas L,
               int ostride) {
    const int qq = (blockIdx.x * SIMT_THREADS + threadIdx.x) >> 5, lane = threadIdx.x & 31;
    if (qq >= q.Q) return;   // whole warps
    const unsigned full = 0xffffffffu;
    const float slo = query_budget(q, qq);
    const int d0 = lane, d1 = lane + 32;
    const bool h0 = d0 < m.D, h1 = d1 < m.D;
    const float *cr = C + (size_t)qq * m.D, *qr = qual + (size_t)qq * qstride;
    const float c0 = h0 ? cr[d0] : 0.f, c1 = h1 ? cr[d1] : 0.f;
    const float g0 = h0 ? qr[m.dep_model[d0]] : 0.f, g1 = h1 ? qr[m.dep_model[d1]] : 0.f;
    const float nan = __int_as_float(0x7fc00000);
    int od = -1;
    float oc = nan, ou = nan;
    for (int k = 0; k < L.K; ++k) {
        const float lam = L.lam[k], wq = L.wq[k];
        const float u0 = __fmaf_rn(-lam, c0, __fmul_rn(wq, g0));
        const float u1 = __fmaf_rn(-lam, c1, __fmul_rn(wq, g1));
        const uint64_t k0 = h0 ? cand_key(c0, u0, d0, slo) : 0, k1 = h1 ? cand_key(c1, u1, d1, slo) : 0;
        const uint64_t kl = k1 > k0 ? k1 : k0;
        const uint32_t hi = __reduce_max_sync(full, (uint32_t)(kl >> 32));
        const uint32_t lo = __reduce_max_sync(full, (uint32_t)(kl >> 32) == hi ? (uint32_t)kl : 0u);
        const int wd = 63 - (int)(lo & 63u);
        const bool ok = (hi >> 6) >= 2u;    // class feasible or infeasible, not NaN
        // the winner's cost and utility, from the lane that holds it
        const float wc = __shfl_sync(full, wd >= 32 ? c1 : c0, wd & 31);
        const float wu = __shfl_sync(full, wd >= 32 ? u1 : u0, wd & 31);
        if (lane == k) {
            od = ok ? wd : -1;
            oc = ok ? wc : nan;
            ou = ok ? wu : nan;
        }
    }
    if (lane < L.K) {
        const size_t o = (size_t)lane * ostride + qq;
        q.chosen[o] = od;
        q.lat[o] = oc;
        q.util[o] = ou;
    }
}

// ---------------------------------------------------------------------------
// host launchers

static int cpt_for(int H2) { return H2 <= 32 ? 1 : H2 <= 64 ? 2 : H2 <= 128 ? 4 : 8; }

size_t route_simt_smem(const Model &m) {
    return route_layout(m.D, m.M, m.H2).total * sizeof(float);
}

size_t seq_table_smem(const Model &m) {
    return seq_layout(m.H2).total * sizeof(float);
}

static size_t chain_smem(int D, int M, int Qs) {
    return (2 * MAX_D + chain_tab_floats(D, Qs) + (size_t)Qs * M + 4 * (size_t)Qs) * sizeof(float);
}


int seq_chunk(const Model &m) {
    int Qs = SEQ_MAX_CHUNK;
    while (Qs > 1 && chain_smem(m.D, m.M, Qs) > (size_t)SEQ_CHAIN_SMEM) --Qs;
    return Qs;
}

// Launch configuration of a programmatic dependent launch: the grid may be
// scheduled before the previous kernel in the stream has finished; it calls
// griddepcontrol.wait before it reads that kernel's results.
static cudaLaunchAttribute g_pdl_attr = [] {
    cudaLaunchAttribute a = {};
    a.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    a.val.programmaticStreamSerializationAllowed = 1;
    return a;
}();

static cudaLaunchConfig_t dependent_launch(int grid, int block, size_t smem, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)block);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = &g_pdl_attr;
    cfg.numAttrs = 1;
    return cfg;
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
    if (e == cudaSuccess) e = opt_in(k_seq_chain<false, false>, SEQ_CHAIN_SMEM + 1024);
    if (e == cudaSuccess) e = opt_in(k_seq_chain<true, false>, SEQ_CHAIN_SMEM + 1024);
    if (e == cudaSuccess) e = opt_in(k_seq_chain<false, true>, SEQ_CHAIN_SMEM + 1024);
    if (e == cudaSuccess) e = opt_in(k_seq_chain<true, true>, SEQ_CHAIN_SMEM + 1024);
    if (e == cudaSuccess) e = opt_in(k_route_pairs, big);
    return e;
}

cudaError_t launch_snapshot(const Model &m, const uint32_t *stage, cudaStream_t s) {
    k_snapshot<<<m.D, SIMT_THREADS, (size_t)m.F * sizeof(float), s>>>(m, stage);
    return cudaGetLastError();
}

cudaError_t launch_route_simt(const Model &m, const Queries &q, cudaStream_t s) {
    if (q.Q <= 0) return cudaSuccess;
    const RouteLayout L = route_layout(m.D, m.M, m.H2);
    const int blocks = (q.Q + L.QB - 1) / L.QB;
    const size_t smem = L.total * sizeof(float);
    switch (cpt_for(m.H2)) {
        case 1: k_route_simt<1><<<blocks, ROUTE_THREADS, smem, s>>>(m, q); break;
        case 2: k_route_simt<2><<<blocks, ROUTE_THREADS, smem, s>>>(m, q); break;
        case 4: k_route_simt<4><<<blocks, ROUTE_THREADS, smem, s>>>(m, q); break;
        default: k_route_simt<8><<<blocks, ROUTE_THREADS, smem, s>>>(m, q); break;
    }
    return cudaGetLastError();
}

size_t route_pairs_smem(const Model &m) {
    const size_t fused = (size_t)pair_smem(m.H1, m.H2).total;
    const size_t split = 3 * PAIR_G + (size_t)m.H1 * PAIR_COLS + (size_t)PAIR_G * (m.H1 | 1);
    const size_t fin = 3 * PAIR_G + (size_t)m.H2 * PAIR_G + (size_t)m.NH * m.H2;
    size_t blk = fused > split ? fused : split;
    blk = blk > fin ? blk : fin;
    const size_t qual = (size_t)m.E * (1 + PAIR_MPB);
    return (blk > qual ? blk : qual) * sizeof(float);
}

cudaError_t launch_route_pairs(const Model &m, const Queries &q, float *pairC, float *qualS,
                               float *h2, int32_t *count, int nsm, cudaStream_t s) {
    if (q.Q <= 0) return cudaSuccess;
    if ((long)q.Q * m.D > PAIRS_MAX_PAIRS) return cudaErrorInvalidValue;
    PairArgs a;
    a.pairC = pairC;
    a.qualS = qualS;
    a.h2 = h2;
    a.count = count;
    a.gcount = count + PAIRS_MAX_PAIRS;
    a.qblocks = (m.M + PAIR_MPB - 1) / PAIR_MPB;
    // The fused shape, 8 columns per block, when the whole grid still has an
    // SM per block: a layer-2 chain step there waits mostly on its shared
    // loads, so narrower blocks (fewer chains sharing an SM's shared memory)
    // finish sooner; with more groups the split shape's 32 columns per block
    // keep the grid to one wave.
    const int groups = pair_groups(q.Q * m.D);
    a.cols = (long)groups * ((m.H2 + PAIR_FUSED_COLS - 1) / PAIR_FUSED_COLS) +
                         (long)q.Q * a.qblocks <= nsm
                 ? PAIR_FUSED_COLS
                 : PAIR_COLS;
    a.ncb = (m.H2 + a.cols - 1) / a.cols;
    const int blocks = pair_groups(q.Q * m.D) * a.ncb + q.Q * a.qblocks;
    k_route_pairs<<<blocks, SIMT_THREADS, route_pairs_smem(m), s>>>(m, q, a);
    return cudaGetLastError();
}

cudaError_t launch_select_multi(const Model &m, const Queries &q, const float *C,
                                const float *qual, int qstride, const Lambdas &L, int ostride,
                                cudaStream_t s) {
    if (q.Q <= 0 || L.K <= 0 || L.K > MAX_LAMBDAS) return q.Q <= 0 || L.K <= 0 ? cudaSuccess : cudaErrorInvalidValue;
    const long threads = (long)q.Q * 32;   // a warp per query
    const int blocks = (int)((threads + SIMT_THREADS - 1) / SIMT_THREADS);
    k_select_multi<<<blocks, SIMT_THREADS, 0, s>>>(m, q, C, qual, qstride, L, ostride);
    return cudaGetLastError();
}

cudaError_t launch_seq_table(const Model &m, const Queries &q, int Qs, int slots, float *ctab,
                             float *aux, cudaStream_t s) {
    const int nuv = (2 * Qs + PREP_THREADS - 1) / PREP_THREADS;
    k_seq_prep<<<nuv + m.D * seq_prep_blocks_per_dep(Qs), PREP_THREADS, 0, s>>>(m, q, Qs, aux, nullptr, nullptr);
    // rows per table block: a multiple of 8 (whole warps of the tile) that
    // spreads the table evenly over the blocks resident at once
    const int T = (int)tri_off(m.D, Qs, Qs);
    const int nb_qual = (Qs + seq_qual_rows(m.M) - 1) / seq_qual_rows(m.M);
    const int want = slots - nb_qual > 1 ? slots - nb_qual : 1;
    int rpb = ((T + want - 1) / want + 7) / 8 * 8;
    rpb = rpb < 8 ? 8 : (rpb > TILE_ROWS ? TILE_ROWS : rpb);
    const int blocks = nb_qual + (T + rpb - 1) / rpb;
    cudaLaunchConfig_t cfg = dependent_launch(blocks, SIMT_THREADS, seq_layout(m.H2).total * sizeof(float), s);
    switch (cpt_for(m.H2)) {
        case 1: return cudaLaunchKernelEx(&cfg, k_seq_table<1>, m, q, Qs, nb_qual, rpb, ctab, aux);
        case 2: return cudaLaunchKernelEx(&cfg, k_seq_table<2>, m, q, Qs, nb_qual, rpb, ctab, aux);
        case 4: return cudaLaunchKernelEx(&cfg, k_seq_table<4>, m, q, Qs, nb_qual, rpb, ctab, aux);
        default: return cudaLaunchKernelEx(&cfg, k_seq_table<8>, m, q, Qs, nb_qual, rpb, ctab, aux);
    }
}

int seq_table_slots(const Model &m) {
    int dev = 0, nsm = 0, per = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return 1;
    const size_t smem = seq_layout(m.H2).total * sizeof(float);
    cudaError_t e;
    switch (cpt_for(m.H2)) {
        case 1: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_seq_table<1>, SIMT_THREADS, smem); break;
        case 2: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_seq_table<2>, SIMT_THREADS, smem); break;
        case 4: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_seq_table<4>, SIMT_THREADS, smem); break;
        default: e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, k_seq_table<8>, SIMT_THREADS, smem); break;
    }
    if (e != cudaSuccess || per < 1) per = 1;
    return nsm * per;
}

cudaError_t launch_seq_chain(const Model &m, const Queries &q, int Qs, const float *ctab,
                             float *aux, cudaStream_t s) {
    cudaLaunchConfig_t cfg = dependent_launch(1, CHAIN_THREADS, chain_smem(m.D, m.M, Qs), s);
    const SeqAux A = seq_aux(aux, m.D, m.M, Qs);
    if (m.D > 32)
        return cudaLaunchKernelEx(&cfg, k_seq_chain<true, false>, m, q, Qs, ctab, aux,
                                  (const float *)A.qual, m.M, 0);
    return cudaLaunchKernelEx(&cfg, k_seq_chain<false, false>, m, q, Qs, ctab, aux,
                              (const float *)A.qual, m.M, 0);
}

cudaError_t launch_seq_prep_tc(const Model &m, const Queries &q, int Qs, float *aux,
                               uint16_t *pre_bf, int32_t *dmv, cudaStream_t s) {
    const int nuv = (2 * Qs + PREP_THREADS - 1) / PREP_THREADS;
    k_seq_prep<<<nuv + m.D * seq_prep_blocks_per_dep(Qs), PREP_THREADS, 0, s>>>(m, q, Qs, aux, pre_bf, dmv);
    return cudaGetLastError();
}

cudaError_t launch_seq_chain_tc(const Model &m, const Queries &q, int Qs, const float *ctab,
                                float *aux, const float *qual, int qstride, cudaStream_t s) {
    if (chain_smem(m.D, m.M, Qs) <= (size_t)SEQ_CHAIN_SMEM) {
        cudaLaunchConfig_t cfg = dependent_launch(1, CHAIN_THREADS, chain_smem(m.D, m.M, Qs), s);
        if (m.D > 32)
            return cudaLaunchKernelEx(&cfg, k_seq_chain<true, false>, m, q, Qs, ctab, aux, qual,
                                      qstride, 0);
        return cudaLaunchKernelEx(&cfg, k_seq_chain<false, false>, m, q, Qs, ctab, aux, qual,
                                  qstride, 0);
    }
    // the table's first rows in shared memory, the rest read from L2
    const size_t rest = chain_smem(m.D, m.M, Qs) - chain_tab_floats(m.D, Qs) * sizeof(float);
    if (rest + 4 * sizeof(float) > (size_t)SEQ_CHAIN_SMEM) return cudaErrorInvalidValue;
    const int tsm = (int)(((size_t)SEQ_CHAIN_SMEM - rest) / sizeof(float)) & ~3;
    cudaLaunchConfig_t cfg =
        dependent_launch(1, CHAIN_THREADS, rest + (size_t)tsm * sizeof(float), s);
    if (m.D > 32)
        return cudaLaunchKernelEx(&cfg, k_seq_chain<true, true>, m, q, Qs, ctab, aux, qual,
                                  qstride, tsm);
    return cudaLaunchKernelEx(&cfg, k_seq_chain<false, true>, m, q, Qs, ctab, aux, qual, qstride,
                              tsm);
}

}  // namespace hwr

