// bf16 tensor-core kernels (tcgen05 + TMA) of the route-scoring path.
//
// K_qual_tc  quality contraction of Sec. 3.2 "Quality Predictor":
//            S = Qemb [Q x E] . Memb [E x M] on the tensor cores (M padded to
//            16 or 32), query tiles streamed by TMA, model embeddings resident
//            in shared memory, accumulators in TMEM; epilogue sigmoid -> qual
//            [Q][Mpad] fp32.  Memory bound: it streams the embeddings once.
// K_mlp_tc   the latency predictor of Eq. 1 for every (query, deployment)
//            pair, then Eq. 2 and the decision maker of Eq. 3.  Per tile of
//            128 queries and per deployment d, producer warps build the layer-1
//            activations relu(A_d + W1[:, in] u_q + W1[:, out] v_q) as bf16
//            straight into the UMMA operand layout in shared memory (A_d is the
//            query-independent prefix of layer 1 computed per snapshot); one
//            thread issues the layer-2 MMA against W2 resident in shared
//            memory into a double-buffered TMEM accumulator; epilogue warps
//            (one TMEM lane = one query) apply bias + ReLU, the two output
//            heads, softplus, the cost, the utility and the SLO mask, and
//            keep the running argmax over d in registers.
//
// Warp roles are fixed per CTA; CTAs are persistent over query tiles.  Every
// mbarrier wait is bounded (umma.cuh): on a timeout the CTA stops, drains what
// it issued, frees its TMEM and reports HWR_ERR_TIMEOUT through the status
// word.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>
#include <string.h>

#include "hwr_internal.cuh"
#include "select.cuh"
#include "umma.cuh"

namespace hwr {

using namespace umma;

namespace {

constexpr int BM = 128;                         // queries per tile
constexpr int KCH = 64;                         // bf16 K elements per 128-byte row
constexpr uint32_t CHUNK_BYTES = BM * KCH * 2;  // one A chunk: 16 KB
constexpr int QUAL_THREADS = 192;               // w0 TMA, w1 MMA, w2-5 epilogue
constexpr int QUAL_STAGES = 8;
constexpr int MLP_THREADS = 448;                // w0 MMA, w1-4 epilogue, w5-12 producers, w13 prefix loader
constexpr int MLP_PRODUCERS = 256;
constexpr int MLP_MAX_STAGES = 8;
constexpr uint32_t SMEM_LIMIT = 227 * 1024;

int g_num_sms = 0;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

}  // namespace

// ---------------------------------------------------------------------------
// host-side shared-memory images (K-major, 128-byte swizzle): the K extent is
// cut into chunks of 64 bf16 (128 bytes); chunk c holds one 128-byte row per
// matrix row n, and inside each row the 16-byte granule g is stored at
// position g ^ (n % 8).  Chunks follow each other.

static inline size_t sw128_index(int rows, int n, int k) {
    const int c = k >> 6, kk = k & 63, g = kk >> 3, e = kk & 7;
    return (size_t)c * rows * 64 + (size_t)n * 64 + (size_t)((g ^ (n & 7)) << 3) + e;
}

size_t tc_w2img_elems(int H1, int H2) { return (size_t)H1 * H2; }
size_t tc_membimg_elems(int Mpad, int Epad) { return (size_t)Mpad * Epad; }

void tc_build_w2img(const uint16_t *W2, int H1, int H2, uint16_t *img) {
    for (int n = 0; n < H2; ++n)
        for (int k = 0; k < H1; ++k) img[sw128_index(H2, n, k)] = W2[(size_t)n * H1 + k];
}

void tc_build_membimg(const uint16_t *memb_EM, int E, int M, int Mpad, int Epad,
                      uint16_t *img) {
    memset(img, 0, (size_t)Mpad * Epad * sizeof(uint16_t));
    for (int m = 0; m < M; ++m)
        for (int k = 0; k < E; ++k) img[sw128_index(Mpad, m, k)] = memb_EM[(size_t)k * M + m];
}

// ---------------------------------------------------------------------------
// shared-memory layouts (byte offsets from a 1024-aligned base)

struct QualLayout {
    uint32_t memb, stages, bars, misc, total;
};

__host__ __device__ inline QualLayout qual_layout(int Mpad, int Epad) {
    QualLayout L;
    uint32_t o = 0;
    L.memb = o;
    o += (uint32_t)Mpad * Epad * 2;
    o = (o + 1023) & ~1023u;
    L.stages = o;
    o += QUAL_STAGES * CHUNK_BYTES;
    L.bars = o;
    o += (2 * QUAL_STAGES + 6) * 8;
    L.misc = o;
    o += 16;
    L.total = o + 1024;  // slack for aligning the dynamic base
    return L;
}

constexpr int APRE_SLOTS = 4;   // deployment-prefix ring (layer-1 A_d rows)

struct MlpLayout {
    uint32_t w2, ring, qual, consts, w1q, uvs, apre, bars, misc, total;
    int ns;
};

constexpr int MLP_BARS = 2 * MLP_MAX_STAGES + 6 + 2 * APRE_SLOTS + 4;

// Layout with ns ring stages of 16 KB.  head_smem: the output-layer
// constants b2, W3 also in shared memory (kernels without a fixed H2 read
// them there; the others take them from the kernel-parameter bank).
__host__ __device__ inline MlpLayout mlp_layout_ns(int H1, int H2, int Mpad, int D, int ns,
                                                   bool head_smem) {
    MlpLayout L;
    L.ns = ns;
    uint32_t o = 0;
    L.w2 = o;                                   // W2 image (B operand)
    o += (uint32_t)H1 * H2 * 2;
    o = (o + 1023) & ~1023u;
    L.ring = o;                                 // A-operand ring
    o += (uint32_t)(ns > 0 ? ns : 0) * CHUNK_BYTES;
    L.qual = o;                                 // quality rows of the tile
    o += BM * (Mpad + 1) * 4;
    L.consts = o;                               // [b2, W3 (<= 3 rows)], b3, dep_model
    o += (head_smem ? 4 * H2 * 4 : 0) + 16 + D * 4;
    o = (o + 15) & ~15u;
    L.w1q = o;                                  // W1's query columns, pairs interleaved
    o += (uint32_t)H1 * 2 * 4;
    L.uvs = o;                                  // standardised query slots [2][2][BM]
    o += 2 * 2 * BM * 4;
    L.apre = o;                                 // deployment-prefix ring
    o += APRE_SLOTS * H1 * 2;
    L.bars = o;
    o += MLP_BARS * 8;
    L.misc = o;
    o += 16;
    L.total = o + 1024;                         // slack for aligning the dynamic base
    return L;
}

// As many ring stages as fit (at most MLP_MAX_STAGES).
__host__ __device__ inline MlpLayout mlp_layout(int H1, int H2, int Mpad, int D, bool head_smem) {
    const uint32_t base = mlp_layout_ns(H1, H2, Mpad, D, 0, head_smem).total;
    int ns = base < SMEM_LIMIT ? (int)((SMEM_LIMIT - base) / CHUNK_BYTES) : 0;
    return mlp_layout_ns(H1, H2, Mpad, D, ns > MLP_MAX_STAGES ? MLP_MAX_STAGES : ns, head_smem);
}

// The predictor kernel has a variant with H2 fixed at compile time for these
// widths (output-layer constants in the parameter bank).
__host__ __device__ inline bool mlp_fixed_h2(int H2) { return H2 == 128 || H2 == 256; }

__device__ __forceinline__ uint8_t *align1024(uint8_t *p) {
    const uint32_t a = smem_u32(p);
    return p + (((a + 1023) & ~1023u) - a);
}

// Bounded wait that ignores the abort flag: used only to drain copies and
// MMAs this CTA itself issued before it frees its resources.
__device__ __forceinline__ void drain_wait(uint64_t *bar, uint32_t parity) {
    const long long t0 = clock64();
    while (!mbar_try_wait(bar, parity) && clock64() - t0 < WAIT_CYCLES) {
    }
}

__device__ __forceinline__ float softplus_fast(float z) {
    return fmaxf(z, 0.f) + log1pf(__expf(-fabsf(z)));
}

__device__ __forceinline__ float standardise_fast(uint8_t code, float v, float mu, float sd) {
    const float t = code == 1 ? log1pf(v) : (code == 2 ? logf(v) : v);
    return (t - mu) / sd;
}

// ---------------------------------------------------------------------------
// K_qual_tc

__global__ void __launch_bounds__(QUAL_THREADS, 1)
k_qual_tc(const __grid_constant__ CUtensorMap tmap, TcModel m, int Q, float *qual,
          int32_t *status, int early, const uint32_t *done, uint32_t done_target) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    const QualLayout L = qual_layout(m.Mpad, m.Epad);
    uint8_t *membs = sm + L.memb, *stages = sm + L.stages;
    uint64_t *full = (uint64_t *)(sm + L.bars), *empty = full + QUAL_STAGES;
    uint64_t *accf = empty + QUAL_STAGES, *acce = accf + 2, *wbar = acce + 2, *dbar = wbar + 1;
    uint32_t *tslot = (uint32_t *)(sm + L.misc);
    volatile int *abort_f = (volatile int *)(tslot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nch = m.Epad / KCH, ntiles = (Q + BM - 1) / BM, Mpad = m.Mpad;
    const uint32_t membytes = (uint32_t)Mpad * m.Epad * 2;

    if (threadIdx.x == 0) {
        for (int s = 0; s < QUAL_STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&accf[b], 1);
            mbar_init(&acce[b], 128);
        }
        mbar_init(wbar, 1);
        mbar_init(dbar, 1);
        *abort_f = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(tslot, 64);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;
    // Launched as a programmatic dependent of the kernel before it on the
    // stream (normally the previous route's predictor): this grid reads only
    // the query embeddings, which were complete before that kernel began, and
    // writes its own quality buffer (two alternate between calls), so it runs
    // alongside that kernel.  It waits for that kernel's completion only at
    // the end.  Its own dependent, the predictor of this call, touches memory
    // that the kernels before may write (outputs, scratch) only after waiting
    // for this grid's completion, so with `early` it may be scheduled at once:
    // its set-up, weight load and first layer-2 steps then overlap this grid
    // and the kernel before.  Without `early` (the kernel before lets its own
    // dependents start early and writes what the predictor reads first, or
    // the caller's inputs may alias earlier outputs) only at the end.
    if (early) grid_launch_dependents();

    if (warp == 0 && lane == 0) {
        // producer: model embeddings once, then query tiles chunk by chunk
        tma_prefetch_desc(&tmap);
        mbar_arrive_expect_tx(wbar, membytes);
        for (uint32_t off = 0; off < membytes; off += 16384)
            bulk_g2s(membs + off, (const uint8_t *)m.membimg + off,
                     membytes - off < 16384 ? membytes - off : 16384, wbar);
        uint32_t n = 0;
        bool ok = true;
        for (int t = blockIdx.x; ok && t < ntiles; t += gridDim.x)
            for (int c = 0; c < nch; ++c, ++n) {
                const int s = n % QUAL_STAGES;
                ok = mbar_wait(&empty[s], ((n / QUAL_STAGES) & 1) ^ 1, abort_f, status);
                if (!ok) break;
                mbar_arrive_expect_tx(&full[s], CHUNK_BYTES);
                tma_load_2d(stages + s * CHUNK_BYTES, &tmap, &full[s], c * KCH, t * BM);
            }
        // drain the loads still in flight before the CTA can exit
        const uint32_t first = n > QUAL_STAGES ? n - QUAL_STAGES : 0;
        for (uint32_t j = first; j < n; ++j) drain_wait(&full[j % QUAL_STAGES], (j / QUAL_STAGES) & 1);
        drain_wait(wbar, 0);
    } else if (warp == 1 && lane == 0) {
        // MMA issuer
        bool ok = mbar_wait(wbar, 0, abort_f, status);
        const uint32_t idesc = idesc_bf16_f32(BM, Mpad);
        uint32_t n = 0, lt = 0;
        for (int t = blockIdx.x; ok && t < ntiles; t += gridDim.x, ++lt) {
            const int b = lt & 1;
            ok = mbar_wait(&acce[b], ((lt >> 1) & 1) ^ 1, abort_f, status);
            if (!ok) break;
            tc_fence_after();
            for (int c = 0; c < nch; ++c, ++n) {
                const int s = n % QUAL_STAGES;
                ok = mbar_wait(&full[s], (n / QUAL_STAGES) & 1, abort_f, status);
                if (!ok) break;
                tc_fence_after();
                const uint64_t ad = sdesc_sw128(smem_u32(stages + s * CHUNK_BYTES));
                const uint64_t bd = sdesc_sw128(smem_u32(membs + (uint32_t)c * Mpad * 128));
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    mma_bf16(tmem + b * 32, ad + 2 * k, bd + 2 * k, idesc, (c | k) != 0);
                mma_commit(&empty[s]);
            }
            if (!ok) break;
            mma_commit(&accf[b]);
        }
        // every MMA this thread issued must land before TMEM is freed
        mma_commit(dbar);
        drain_wait(dbar, 0);
    } else if (warp >= 2) {
        // epilogue: TMEM lane = query row of the tile
        const int quad = warp & 3, r = quad * 32 + lane;
        const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
        uint32_t lt = 0;
        bool ok = true, may_store = done == nullptr;
        for (int t = blockIdx.x; t < ntiles; t += gridDim.x, ++lt) {
            const int b = lt & 1;
            ok = mbar_wait(&accf[b], (lt >> 1) & 1, abort_f, status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            tc_fence_after();
            uint32_t v[32];
            uint32_t v16[16];
            tmem_ld16(tmem + lane_base + b * 32, v16);
            tmem_wait_ld16(v16);
#pragma unroll
            for (int i = 0; i < 16; ++i) v[i] = v16[i];
            if (Mpad == 32) {
                tmem_ld16(tmem + lane_base + b * 32 + 16, v16);
                tmem_wait_ld16(v16);
#pragma unroll
                for (int i = 0; i < 16; ++i) v[16 + i] = v16[i];
            }
            tc_fence_before();
            mbar_arrive(&acce[b]);
            if (!may_store) {
                // This buffer was last read by the predictor two routes back
                // (the buffers alternate), which may still run when this grid
                // starts: before the first store, every predictor CTA launched
                // before the most recent predictor has finished.
                if (lane == 0) ok = count_wait(done, done_target, abort_f, status);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                __syncwarp();
                may_store = true;
                if (!ok) break;
            }
            const int row = t * BM + r;
            if (row < Q) {
                float4 *dst = (float4 *)(qual + (size_t)row * Mpad);
                for (int i = 0; i < Mpad; i += 4) {
                    float4 o;
                    o.x = i + 0 < m.M ? 1.f / (1.f + expf(-__uint_as_float(v[i + 0]))) : 0.f;
                    o.y = i + 1 < m.M ? 1.f / (1.f + expf(-__uint_as_float(v[i + 1]))) : 0.f;
                    o.z = i + 2 < m.M ? 1.f / (1.f + expf(-__uint_as_float(v[i + 2]))) : 0.f;
                    o.w = i + 3 < m.M ? 1.f / (1.f + expf(-__uint_as_float(v[i + 3]))) : 0.f;
                    dst[i >> 2] = o;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    grid_dependency_wait();
    if (!early) grid_launch_dependents();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, 64);
    }
}

// ---------------------------------------------------------------------------
// K_mlp_tc
//
// Work unit = (query tile, part of the deployment range).  The first nwhole
// tiles are units of all D deployments; each remaining tile is split into
// nsplit parts, dealt after them (so the split tiles even out the last,
// partial round over the CTAs).  A part leaves its per-row best candidate in
// `part` and the last of a row's parts to arrive (per-row atomic counter)
// merges them; whole tiles write their decisions directly.

struct Unit {
    int tile, d0, d1;
};

__host__ __device__ __forceinline__ int unit_part(int u, int ntiles, int nwhole) {
    return u < nwhole ? 0 : (u - nwhole) / (ntiles - nwhole);
}

__host__ __device__ __forceinline__ Unit unit_of(int u, int ntiles, int nwhole, int nsplit,
                                                 int D) {
    Unit x;
    if (u < nwhole) {
        x.tile = u;
        x.d0 = 0;
        x.d1 = D;
        return x;
    }
    const int v = u - nwhole, ntail = ntiles - nwhole, part = v / ntail;
    x.tile = nwhole + (v - part * ntail);
    x.d0 = part * D / nsplit;
    x.d1 = (part + 1) * D / nsplit;
    return x;
}

// bf16 pairs in 32-bit registers: relu(a * b + c), and float pair -> bf16 pair
__device__ __forceinline__ uint32_t hfma2_relu(uint32_t a, uint32_t b, uint32_t c) {
    uint32_t d;
    asm("fma.rn.relu.bf16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
    return d;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t d;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
    return d;
}

// Four columns of the second hidden layer into the output heads.  With
// nb = -b2, relu(acc + b2) = max(acc, nb) + b2 exactly, so
// sum_n w[n] relu(acc[n] + b2[n]) = sum_n w[n] max(acc[n], nb[n]) + sum_n w[n] b2[n];
// the constant second sum is folded into the head bias b3 on the host (in
// double), which leaves one max per column and packed FMAs for the heads.
template <int NH>
__device__ __forceinline__ void head_pair(const uint32_t *v, int j, const float4 &nb,
                                          const float4 &w0, const float4 &w1, const float4 &w2,
                                          float2 &t0a, float2 &t0b, float2 &t1a, float2 &t1b,
                                          float2 &t2a, float2 &t2b) {
    float2 x01, x23;
    x01.x = fmaxf(__uint_as_float(v[j]), nb.x);
    x01.y = fmaxf(__uint_as_float(v[j + 1]), nb.y);
    x23.x = fmaxf(__uint_as_float(v[j + 2]), nb.z);
    x23.y = fmaxf(__uint_as_float(v[j + 3]), nb.w);
    t0a = __ffma2_rn(x01, make_float2(w0.x, w0.y), t0a);
    t0b = __ffma2_rn(x23, make_float2(w0.z, w0.w), t0b);
    t1a = __ffma2_rn(x01, make_float2(w1.x, w1.y), t1a);
    t1b = __ffma2_rn(x23, make_float2(w1.z, w1.w), t1b);
    if constexpr (NH == 3) {
        t2a = __ffma2_rn(x01, make_float2(w2.x, w2.y), t2a);
        t2b = __ffma2_rn(x23, make_float2(w2.z, w2.w), t2b);
    }
}

// Standardised query slots of query `row` into slot r of a [2][BM] buffer
// (u: input length, v: output length), then arrive on `full`.
__device__ __forceinline__ void put_slots(const TcModel &m, const Queries &q, int row, int r,
                                          float *uv, uint64_t *full) {
    const bool v = row < q.Q;
    uv[r] = v ? standardise_fast(m.xf_in, q.in_len[row], m.mu_in, m.sd_in) : 0.f;
    uv[BM + r] = v ? standardise_fast(m.xf_out, q.out_len[row], m.mu_out, m.sd_out) : 0.f;
    mbar_arrive(full);
}

// Output-layer constants passed by value: they sit in the kernel-parameter
// constant bank, so the fully unrolled epilogue reads them as instruction
// operands instead of shared-memory loads.  nb2 = -b2; b3 holds the head
// biases plus sum_n W3[o][n] b2[n] (see head_pair).
struct HeadConsts {
    float nb2[MAX_H], w0[MAX_H], w1[MAX_H], w2[MAX_H], b3[3];
};

template <int H2T, int NH>
__global__ void __launch_bounds__(MLP_THREADS, 1)
k_mlp_tc(TcModel m, Queries q, const __grid_constant__ HeadConsts hc,
         const float *__restrict__ qual, int nwhole, int nsplit, int4 *part, int32_t *count,
         int32_t *status, uint32_t *done) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr bool FIXED = H2T > 0;
    const int H1 = m.H1, H2 = FIXED ? H2T : m.H2, D = m.D, Mpad = m.Mpad, QS = Mpad + 1;
    const MlpLayout L = mlp_layout(H1, H2, Mpad, D, !FIXED);
    const int NS = L.ns;
    uint8_t *w2s = sm + L.w2, *ring = sm + L.ring;
    float *qs = (float *)(sm + L.qual);
    // b2 (negated), W3 rows: only without a fixed H2
    float *b2s = (float *)(sm + L.consts), *w30s = b2s + H2, *w31s = w30s + H2;
    float *w32s = w31s + H2, *b3s = FIXED ? b2s : w32s + H2;
    int *dms = (int *)(b3s + 4);
    float *uvs = (float *)(sm + L.uvs);        // [buffer][u / v][row]
    uint64_t *full = (uint64_t *)(sm + L.bars), *empty = full + MLP_MAX_STAGES;
    uint64_t *accf = empty + MLP_MAX_STAGES, *acce = accf + 2, *wbar = acce + 2, *dbar = wbar + 1;
    uint64_t *afull = dbar + 1, *afree = afull + APRE_SLOTS;   // prefix ring
    uint64_t *uvfull = afree + APRE_SLOTS, *uvfree = uvfull + 2;   // query slots
    uint8_t *apre = sm + L.apre;
    uint32_t *tslot = (uint32_t *)(sm + L.misc);
    volatile int *abort_f = (volatile int *)(tslot + 1);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int nch = H1 / KCH, ntiles = (q.Q + BM - 1) / BM, nunits = nwhole + (ntiles - nwhole) * nsplit;
    const uint32_t tcols = 2 * H2 <= 32 ? 32 : 2 * H2 <= 64 ? 64 : 2 * H2 <= 128 ? 128
                                                : 2 * H2 <= 256 ? 256 : 512;

    if (tid == 0) {
        for (int s = 0; s < NS; ++s) {
            mbar_init(&full[s], MLP_PRODUCERS);
            mbar_init(&empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&accf[b], 1);
            mbar_init(&acce[b], 128);
        }
        mbar_init(wbar, 1);
        mbar_init(dbar, 1);
        for (int j = 0; j < APRE_SLOTS; ++j) {
            mbar_init(&afull[j], 1);
            mbar_init(&afree[j], MLP_PRODUCERS);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&uvfull[b], 128);
            mbar_init(&uvfree[b], MLP_PRODUCERS / 32);
        }
        *abort_f = 0;
        fence_mbar_init();
    }
    if (!FIXED) {
        for (int i = tid; i < H2; i += MLP_THREADS) {
            b2s[i] = hc.nb2[i];
            w30s[i] = m.W3[i];
            w31s[i] = m.W3[H2 + i];
            w32s[i] = NH == 3 ? m.W3[2 * H2 + i] : 0.f;
        }
    }
    if (tid < NH) b3s[tid] = hc.b3[tid];
    for (int i = tid; i < D; i += MLP_THREADS) dms[i] = m.dep_model[i];
    // W1's two query columns as {W1[k][in], W1[k+1][in], W1[k][out], W1[k+1][out]}
    // per pair of rows k: one 16-byte load serves a pair for every query row
    float4 *w1qs = (float4 *)(sm + L.w1q);
    for (int i = tid; i < H1 / 2; i += MLP_THREADS)
        w1qs[i] = make_float4(m.W1q[2 * i], m.W1q[2 * i + 1], m.W1q[H1 + 2 * i], m.W1q[H1 + 2 * i + 1]);
    if (warp == 0) {
        tmem_alloc(tslot, tcols);
        tmem_relinquish();
    }
    // the next route's quality kernel may be scheduled now: it waits for this
    // grid's completion before it touches memory
    grid_launch_dependents();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tslot;

    if (warp == 0 && lane == 0) {
        // ---- MMA issuer: W2 once, then one layer-2 MMA chain per step -----
        const uint32_t wbytes = (uint32_t)H1 * H2 * 2;
        mbar_arrive_expect_tx(wbar, wbytes);
        for (uint32_t off = 0; off < wbytes; off += 16384)
            bulk_g2s(w2s + off, (const uint8_t *)m.W2img + off,
                     wbytes - off < 16384 ? wbytes - off : 16384, wbar);
        bool ok = mbar_wait(wbar, 0, abort_f, status);
        const uint32_t idesc = idesc_bf16_f32(BM, H2);
        uint32_t g = 0, ph = 0;
        int s = 0;
        for (int u = blockIdx.x; ok && u < nunits; u += gridDim.x) {
            const Unit un = unit_of(u, ntiles, nwhole, nsplit, D);
            for (int d = un.d0; d < un.d1; ++d, ++g) {
                const int b = g & 1;
                ok = mbar_wait(&acce[b], ((g >> 1) & 1) ^ 1, abort_f, status);
                if (!ok) break;
                tc_fence_after();
                const uint32_t dt = tmem + (uint32_t)b * H2;
                for (int c = 0; c < nch; ++c) {
                    ok = mbar_wait(&full[s], ph, abort_f, status);
                    if (!ok) break;
                    tc_fence_after();
                    const uint64_t ad = sdesc_sw128(smem_u32(ring + s * CHUNK_BYTES));
                    const uint64_t bd = sdesc_sw128(smem_u32(w2s + (uint32_t)c * H2 * 128));
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_bf16(dt, ad + 2 * k, bd + 2 * k, idesc, (c | k) != 0);
                    mma_commit(&empty[s]);
                    if (++s == NS) {
                        s = 0;
                        ph ^= 1;
                    }
                }
                if (!ok) break;
                mma_commit(&accf[b]);
            }
        }
        // everything this thread issued must land before TMEM is freed
        mma_commit(dbar);
        drain_wait(dbar, 0);
        drain_wait(wbar, 0);
    } else if (warp >= 1 && warp < 5) {
        // ---- epilogue: TMEM lane = query row of the tile ---------------------
        const int quad = warp & 3, r = quad * 32 + lane;
        const uint32_t lane_base = (uint32_t)(quad * 32) << 16;
        const float slo = q.slo, lam = q.lam, wq = q.wq, b30 = b3s[0], b31 = b3s[1];
        const float b32 = NH == 3 ? b3s[2] : 0.f;
        const float4 *b2v = (const float4 *)b2s, *w0v = (const float4 *)w30s,
                     *w1v = (const float4 *)w31s, *w2v = (const float4 *)w32s;
        const int ncol = H2 / 32;
        uint32_t g = 0;
        bool ok = true;
        // The standardised query slots u, v of row r for the producers (one
        // row per thread), one unit ahead: the local unit k uses buffer k & 1,
        // refilled once the producers have read it for unit k - 2.
        if (blockIdx.x < nunits)   // the lengths are inputs: no wait for the kernel before
            put_slots(m, q, unit_of(blockIdx.x, ntiles, nwhole, nsplit, D).tile * BM + r, r, uvs,
                      &uvfull[0]);
        // the quality matrix comes from the kernel before (a dependent launch
        // may start this grid before that one has finished)
        grid_dependency_wait();
        int lk = 0;
        for (int u = blockIdx.x; ok && u < nunits; u += gridDim.x, ++lk) {
            const Unit un = unit_of(u, ntiles, nwhole, nsplit, D);
            if (u + (int)gridDim.x < nunits) {
                const int k = lk + 1, b = k & 1;
                if (k >= 2) ok = mbar_wait(&uvfree[b], ((k >> 1) & 1) ^ 1, abort_f, status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                put_slots(m, q, unit_of(u + gridDim.x, ntiles, nwhole, nsplit, D).tile * BM + r, r,
                          uvs + 2 * b * BM, &uvfull[b]);
            }
            const int row = un.tile * BM + r;
            const bool valid = row < q.Q;
            const float ol = valid ? q.out_len[row] : 0.f;
            const float slo_r = valid ? query_budget(q, row) : slo;
            for (int i = 0; i < m.M; ++i)
                qs[r * QS + i] = valid ? qual[(size_t)row * Mpad + i] : 0.f;
            Cand best = no_cand();
            for (int d = un.d0; d < un.d1; ++d, ++g) {
                const int b = g & 1;
                ok = mbar_wait(&accf[b], (g >> 1) & 1, abort_f, status);
                ok = __all_sync(0xffffffffu, ok);
                if (!ok) break;
                tc_fence_after();
                const uint32_t base = tmem + lane_base + (uint32_t)b * H2;
                float2 t0a = make_float2(0.f, 0.f), t0b = t0a, t1a = t0a, t1b = t0a, t2a = t0a,
                       t2b = t0a;
                uint32_t va[32], vb[32];
                tmem_ld32(base, va);
                if constexpr (FIXED) {
                    constexpr int NC = H2T / 32;
#pragma unroll
                    for (int c = 0; c < NC; ++c) {
                        uint32_t(&cur)[32] = (c & 1) ? vb : va;
                        uint32_t(&nxt)[32] = (c & 1) ? va : vb;
                        tmem_wait_ld32(cur);
                        if (c + 1 < NC) tmem_ld32(base + (c + 1) * 32, nxt);
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            const int n = c * 32 + j;
                            head_pair<NH>(cur, j, make_float4(hc.nb2[n], hc.nb2[n + 1], hc.nb2[n + 2], hc.nb2[n + 3]),
                                          make_float4(hc.w0[n], hc.w0[n + 1], hc.w0[n + 2], hc.w0[n + 3]),
                                          make_float4(hc.w1[n], hc.w1[n + 1], hc.w1[n + 2], hc.w1[n + 3]),
                                          make_float4(hc.w2[n], hc.w2[n + 1], hc.w2[n + 2], hc.w2[n + 3]),
                                          t0a, t0b, t1a, t1b, t2a, t2b);
                        }
                    }
                } else {
                    for (int c = 0; c < ncol; c += 2) {
                        tmem_wait_ld32(va);
                        if (c + 1 < ncol) tmem_ld32(base + (c + 1) * 32, vb);
#pragma unroll
                        for (int j = 0; j < 32; j += 4) {
                            const int f = (c * 32 + j) >> 2;
                            head_pair<NH>(va, j, b2v[f], w0v[f], w1v[f], w2v[f], t0a, t0b, t1a, t1b,
                                          t2a, t2b);
                        }
                        if (c + 1 < ncol) {
                            tmem_wait_ld32(vb);
                            if (c + 2 < ncol) tmem_ld32(base + (c + 2) * 32, va);
#pragma unroll
                            for (int j = 0; j < 32; j += 4) {
                                const int f = ((c + 1) * 32 + j) >> 2;
                                head_pair<NH>(vb, j, b2v[f], w0v[f], w1v[f], w2v[f], t0a, t0b, t1a,
                                              t1b, t2a, t2b);
                            }
                        }
                    }
                }
                tc_fence_before();
                mbar_arrive(&acce[b]);
                const float z0 = (t0a.x + t0a.y) + (t0b.x + t0b.y) + b30;
                const float z1 = (t1a.x + t1a.y) + (t1b.x + t1b.y) + b31;
                const float z2 = (t2a.x + t2a.y) + (t2b.x + t2b.y) + b32;
                const float ttft = softplus_fast(z0), tpot = softplus_fast(z1);
                // N_out of Eq. 2: the third head, or the query's given length
                const float C = fmaf(NH == 3 ? softplus_fast(z2) : ol, tpot, ttft);
                const float U = fmaf(-lam, C, wq * qs[r * QS + dms[d]]);
                if (q.pair_C && valid) {
                    if (q.seq_n == 0) {
                        q.pair_C[(size_t)row * D + d] = C;
                    } else {
                        // (deployment, count) slot d: keep the entries with
                        // count <= query (the lanes of a warp write
                        // consecutive queries of one table row)
                        const int np = q.seq_n + 1, dd = d / np, cc = d - dd * np;
                        if (cc <= row) q.pair_C[tab_row(D / np, q.seq_n, cc, dd) + row] = C;
                    }
                }
                const Cand cd = make_cand(C, U, d, slo_r);
                if (better(cd, best)) best = cd;
            }
            if (!ok || !valid || q.no_select) continue;
            const int nparts = u < nwhole ? 1 : nsplit;
            if (nparts == 1) {
                const bool sel = best.cls > 0;
                q.chosen[row] = sel ? best.d : -1;
                q.lat[row] = sel ? best.C : __int_as_float(0x7fc00000);
                q.util[row] = sel ? best.U : __int_as_float(0x7fc00000);
                continue;
            }
            part[(size_t)unit_part(u, ntiles, nwhole) * q.Q + row] =
                make_int4(best.cls, best.d, __float_as_int(best.C), __float_as_int(best.U));
            // release: the record above is visible to whoever increments the
            // counter later; acquire: the last arrival sees every record
            int seen;
            asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;"
                         : "=r"(seen)
                         : "l"(count + row)
                         : "memory");
            if (seen == nparts - 1) {
                // last of this row's units: merge the parts (any order gives the
                // same result: the candidate order is total)
                Cand acc = no_cand();
                for (int pp = 0; pp < nparts; ++pp) {
                    const int4 x = __ldcg(&part[(size_t)pp * q.Q + row]);
                    Cand c;
                    c.cls = x.x;
                    c.d = x.y;
                    c.C = __int_as_float(x.z);
                    c.U = __int_as_float(x.w);
                    if (better(c, acc)) acc = c;
                }
                const bool sel = acc.cls > 0;
                q.chosen[row] = sel ? acc.d : -1;
                q.lat[row] = sel ? acc.C : __int_as_float(0x7fc00000);
                q.util[row] = sel ? acc.U : __int_as_float(0x7fc00000);
                count[row] = 0;
            }
        }
    } else if (warp >= 5 && warp < 13) {
        // ---- producers: layer-1 activations as bf16 UMMA operand tiles ------
        // Thread p owns granule gi = p % 8 (8 consecutive K) of every 64-wide K
        // chunk, for rows rb + 32 i (i < 4).  The query part of layer 1,
        // W1[:, in] u + W1[:, out] v, does not depend on the deployment: it is
        // built once per unit in registers (bf16 pairs) and every step then
        // needs one fused add + ReLU per pair: relu(1 * B + A_d).
        const int p = tid - 160, gi = p & 7, rb = p >> 3;
        // shared-memory offset of granule gi of row rb in a stage (K-major,
        // 128-byte swizzle); row rb + 32 i sits 4 atoms (4096 bytes) further
        const uint32_t offs0 = (uint32_t)(rb >> 3) * 1024 + (uint32_t)(rb & 7) * 128 +
                               (uint32_t)((gi ^ (rb & 7)) << 4);
        const uint32_t one2 = 0x3F803F80u;  // (1.0, 1.0) in bf16
        uint32_t Bq[4][4][4];
        uint32_t ph = 0;
        int s = 0;
        bool ok = true;
        // Deployment prefixes A_d come through the 4-slot shared-memory ring
        // the loader warp fills; each producer frees a slot (afree) once it has
        // built every chunk from its granules.  dn counts this CTA's deployments.
        const uint32_t abytes = (uint32_t)H1 * 2;
        uint32_t dn = 0;
        int lk = 0;
        for (int u = blockIdx.x; ok && u < nunits; u += gridDim.x, ++lk) {
            const Unit un = unit_of(u, ntiles, nwhole, nsplit, D);
            // standardised query slots of this thread's four rows, prepared by
            // the epilogue warps
            const int ub = lk & 1;
            ok = mbar_wait(&uvfull[ub], (lk >> 1) & 1, abort_f, status);
            ok = __all_sync(0xffffffffu, ok);
            if (!ok) break;
            float uu[4], vv[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uu[i] = uvs[(2 * ub) * BM + rb + 32 * i];
                vv[i] = uvs[(2 * ub + 1) * BM + rb + 32 * i];
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&uvfree[ub]);
            // the query part of this thread's granules: W1 pairs from shared
            // memory, each used for the four rows, as packed fp32 products
            // (per lane: fma(v, W1[out], u * W1[in]))
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                if (c < nch) {
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float4 w = w1qs[c * (KCH / 2) + gi * 4 + e];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const float2 pr = __fmul2_rn(make_float2(uu[i], uu[i]), make_float2(w.x, w.y));
                            const float2 h = __ffma2_rn(make_float2(vv[i], vv[i]), make_float2(w.z, w.w), pr);
                            Bq[i][c][e] = pack_bf16x2(h.x, h.y);
                        }
                    }
                }
            }

            for (int d = un.d0; ok && d < un.d1; ++d, ++dn) {
                const int j = dn & (APRE_SLOTS - 1);
                ok = ok && mbar_wait(&afull[j], (dn / APRE_SLOTS) & 1, abort_f, status);
                if (!ok) break;
                const uint4 *As = (const uint4 *)(apre + j * abytes);
                // two chunks per round: one wait / fence / arrive cycle covers
                // both, halving the serial latency each producer warp pays
#pragma unroll
                for (int c = 0; c < 4; c += 2) {
                    if (c < nch && ok) {
                        const bool two = c + 1 < nch;
                        // this round's prefix granules (loaded before the waits)
                        uint4 a[2];
                        a[0] = As[c * 8 + gi];
                        if (two) a[1] = As[(c + 1) * 8 + gi];
                        const int s1 = s + 1 == NS ? 0 : s + 1;
                        const uint32_t ph1 = s + 1 == NS ? ph ^ 1 : ph;
                        ok = mbar_wait(&empty[s], ph ^ 1, abort_f, status);
                        if (ok && two) ok = mbar_wait(&empty[s1], ph1 ^ 1, abort_f, status);
                        if (ok) {
#pragma unroll
                            for (int cc = 0; cc < 2; ++cc) {
                                if (cc == 0 || two) {
                                    const uint4 av = a[cc];
                                    const uint32_t st = smem_u32(ring + (cc ? s1 : s) * CHUNK_BYTES);
#pragma unroll
                                    for (int i = 0; i < 4; ++i) {
                                        const uint32_t h0 = hfma2_relu(Bq[i][c + cc][0], one2, av.x);
                                        const uint32_t h1 = hfma2_relu(Bq[i][c + cc][1], one2, av.y);
                                        const uint32_t h2 = hfma2_relu(Bq[i][c + cc][2], one2, av.z);
                                        const uint32_t h3 = hfma2_relu(Bq[i][c + cc][3], one2, av.w);
                                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(
                                                         st + offs0 + 4096u * i),
                                                     "r"(h0), "r"(h1), "r"(h2), "r"(h3)
                                                     : "memory");
                                    }
                                }
                            }
                            fence_proxy_async_smem();
                            if (!m.test_stall) {
                                mbar_arrive(&full[s]);
                                if (two) mbar_arrive(&full[s1]);
                            }
                            s = s1;
                            ph = ph1;
                            if (two && ++s == NS) {
                                s = 0;
                                ph ^= 1;
                            }
                        }
                    }
                }
                // the slot is freed only after the chunks above have used every
                // granule read from it, so those shared-memory reads are complete
                // before the loader's next bulk copy can overwrite it
                mbar_arrive(&afree[j]);
            }
        }
    } else if (warp == 13 && lane == 0) {
        // ---- prefix loader: the layer-1 deployment prefix of every step of
        // this CTA's units, in order, into the 4-slot ring (bulk copies,
        // completion on afull; a slot is reused once afree says all producers
        // have read it) ------------------------------------------------------
        const uint32_t abytes = (uint32_t)H1 * 2;
        uint32_t issued = 0;
        bool ok = true;
        for (int u = blockIdx.x; ok && u < nunits; u += gridDim.x) {
            const Unit un = unit_of(u, ntiles, nwhole, nsplit, D);
            for (int d = un.d0; d < un.d1; ++d, ++issued) {
                const int j = issued & (APRE_SLOTS - 1);
                if (issued >= APRE_SLOTS)
                    ok = mbar_wait(&afree[j], ((issued / APRE_SLOTS) & 1) ^ 1, abort_f, status);
                if (!ok) break;
                mbar_arrive_expect_tx(&afull[j], abytes);
                bulk_g2s(apre + j * abytes, (const uint8_t *)m.Abf + (size_t)d * abytes, abytes,
                         &afull[j]);
            }
        }
        // the last copies may still be in flight: they land before the CTA exits
        for (uint32_t k = issued > APRE_SLOTS ? issued - APRE_SLOTS : 0; k < issued; ++k)
            drain_wait(&afull[k & (APRE_SLOTS - 1)], (k / APRE_SLOTS) & 1);
    }
    tc_fence_before();
    __syncthreads();
    // every global access of this CTA is done: count it for the quality kernel
    // that will next overwrite the quality buffer this grid read
    if (done && tid == 0) count_release(done);
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, tcols);
    }
}

// ---------------------------------------------------------------------------
// host side

bool tc_supported(int M, int H1, int H2, int E) {
    if (M < 1 || M > 32) return false;
    if (H1 < 64 || H1 > 256 || H1 % 64) return false;
    if (H2 < 32 || H2 > 256 || H2 % 32) return false;
    if (E < 8 || E % 8) return false;
    const int Mpad = M <= 16 ? 16 : 32, Epad = (E + 63) / 64 * 64;
    if (qual_layout(Mpad, Epad).total > SMEM_LIMIT) return false;
    const MlpLayout L = mlp_layout(H1, H2, Mpad, 64, !mlp_fixed_h2(H2));
    return L.ns >= 2 && L.total <= SMEM_LIMIT;
}

cudaError_t tc_prepare() {
    if (!g_num_sms) {
        int dev = 0;
        cudaError_t e = cudaGetDevice(&dev);
        if (e == cudaSuccess) e = cudaDeviceGetAttribute(&g_num_sms, cudaDevAttrMultiProcessorCount, dev);
        if (e != cudaSuccess) return e;
    }
    if (!g_encode) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult qr;
        cudaError_t e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                         cudaEnableDefault, &qr);
        if (e != cudaSuccess) return e;
        if (qr != cudaDriverEntryPointSuccess || !fn) return cudaErrorNotSupported;
        g_encode = (PFN_cuTensorMapEncodeTiled_v12000)fn;
    }
    cudaError_t e = cudaFuncSetAttribute(k_qual_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         SMEM_LIMIT);
    const auto attr = cudaFuncAttributeMaxDynamicSharedMemorySize;
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_mlp_tc<0, 2>, attr, SMEM_LIMIT);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_mlp_tc<128, 2>, attr, SMEM_LIMIT);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_mlp_tc<256, 2>, attr, SMEM_LIMIT);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_mlp_tc<0, 3>, attr, SMEM_LIMIT);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_mlp_tc<128, 3>, attr, SMEM_LIMIT);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(k_mlp_tc<256, 3>, attr, SMEM_LIMIT);
    return e;
}

cudaError_t launch_qual_tc(const TcModel &m, const Queries &q, float *qual, int32_t *status,
                           cudaStream_t s, bool dependent, bool early, int free_sms,
                           const uint32_t *done, uint32_t done_target) {
    if (q.Q <= 0) return cudaSuccess;
    CUtensorMap map;
    const cuuint64_t dims[2] = {(cuuint64_t)m.E, (cuuint64_t)q.Q};
    const cuuint64_t strides[1] = {(cuuint64_t)m.E * 2};
    const cuuint32_t box[2] = {KCH, BM};
    const cuuint32_t estr[2] = {1, 1};
    CUresult r = g_encode(&map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(q.emb),
                          dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                          CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    // as many CTAs as give every CTA the same number of tiles (512 tiles on
    // 152 SMs: 128 CTAs of 4 tiles, not 152 with a last round on 56)
    const int ntiles = (q.Q + BM - 1) / BM;
    int rounds = (ntiles + g_num_sms - 1) / g_num_sms;
    // a small batch on the SMs the predictor leaves free, at most two tiles
    // each: the predictor's CTAs then find their SMs free as the previous
    // predictor's leave (4,096 queries at D = 32: 16 CTAs of 2 tiles beside
    // 128 predictor CTAs, 24.8 -> 19.6 us per call back to back; with three or
    // more tiles per CTA the longer quality kernel costs a lone call more
    // than the overlap gives)
    if (early && free_sms >= 8 && ntiles <= 2 * free_sms) rounds = (ntiles + free_sms - 1) / free_sms;
    const int grid = (ntiles + rounds - 1) / rounds;
    const QualLayout L = qual_layout(m.Mpad, m.Epad);
    // programmatic dependent launch (when `qual` is not read by the kernel
    // before it): the grid runs alongside that kernel and waits for it at
    // its end
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(QUAL_THREADS);
    cfg.dynamicSmemBytes = L.total;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = dependent ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, k_qual_tc, map, m, q.Q, qual, status, early ? 1 : 0, done,
                              done_target);
}

cudaError_t launch_mlp_tc_scores(const TcModel &m, const Queries &q, const float *qual,
                                 int32_t *status, cudaStream_t s, uint32_t *done, int *ctas) {
    *ctas = 0;
    if (q.Q <= 0) return cudaSuccess;
    if (q.Q > BM || !q.no_select || !q.pair_C) return cudaErrorInvalidValue;
    if (q.seq_n && (q.seq_n != q.Q || m.D % (q.seq_n + 1))) return cudaErrorInvalidValue;
    // one tile: split its deployments into one part per SM
    const int sms = g_num_sms > 0 ? g_num_sms : 1;
    const MlpSplit sp{0, m.D < sms ? m.D : sms};
    return launch_mlp_tc(m, q, qual, sp, nullptr, nullptr, status, s, done, ctas);
}

// Unit decomposition that minimises the busiest CTA's cost in deployment
// steps: R rounds of whole tiles (one per SM each), then the remaining tiles
// in ns parts, dealt round-robin.  A unit also pays a fixed setup cost, larger
// for split tiles (the part record and the merge), from per-unit timings of
// the kernel on GB300.
MlpSplit tc_mlp_split(const TcModel &m, int Q, int max_split) {
    constexpr double SETUP_WHOLE = 0.7, SETUP_SPLIT = 2.5;   // in deployment steps
    const int ntiles = (Q + BM - 1) / BM, sms = g_num_sms > 0 ? g_num_sms : 1, D = m.D;
    MlpSplit best{0, 1};
    double best_cost = 1e300;
    long best_units = 0;
    for (int R = 0; R * sms <= ntiles; ++R) {
        const int nwhole = R * sms, ntail = ntiles - nwhole;
        for (int ns = 1; ns <= max_split && ns <= D; ++ns) {
            if (ntail == 0 && ns > 1) break;
            const long tail_units = (long)ntail * ns, units = nwhole + tail_units;
            if (units == 0) continue;
            const long grid = units < sms ? units : sms;
            const double per = ns > 1 ? (double)((D + ns - 1) / ns) + SETUP_SPLIT : D + SETUP_WHOLE;
            const double cost = R * (D + SETUP_WHOLE) + (double)((tail_units + grid - 1) / grid) * per;
            if (cost < best_cost - 1e-9 || (cost < best_cost + 1e-9 && units < best_units)) {
                best_cost = cost;
                best = MlpSplit{nwhole, ns};
                best_units = units;
            }
        }
    }
    return best;
}

int tc_mlp_free_sms(int Q, const MlpSplit &sp) {
    const int ntiles = (Q + BM - 1) / BM;
    const long units = sp.nwhole + (long)(ntiles - sp.nwhole) * sp.nsplit;
    return units < g_num_sms ? g_num_sms - (int)units : 0;
}

cudaError_t launch_mlp_tc(const TcModel &m, const Queries &q, const float *qual,
                          const MlpSplit &sp, void *part, int32_t *count, int32_t *status,
                          cudaStream_t s, uint32_t *done, int *ctas) {
    *ctas = 0;
    if (q.Q <= 0) return cudaSuccess;
    const int ntiles = (q.Q + BM - 1) / BM;
    if (sp.nwhole < 0 || sp.nwhole > ntiles || sp.nsplit < 1) return cudaErrorInvalidValue;
    const long units = sp.nwhole + (long)(ntiles - sp.nwhole) * sp.nsplit;
    const int grid = units < g_num_sms ? (int)units : g_num_sms;
    const MlpLayout L = mlp_layout(m.H1, m.H2, m.Mpad, m.D, !mlp_fixed_h2(m.H2));
    const HeadConsts &hc = *m.head;
    int4 *pt = (int4 *)part;
    // programmatic dependent launch: the grid may start while the quality
    // kernel before it on the stream finishes (its epilogue waits for it)
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(MLP_THREADS);
    cfg.dynamicSmemBytes = L.total;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    cudaError_t e;
#define HWR_MLP(H2T, NHT) \
    e = cudaLaunchKernelEx(&cfg, k_mlp_tc<H2T, NHT>, m, q, hc, qual, sp.nwhole, sp.nsplit, pt, \
                           count, status, done)
    if (m.NH == 3) {
        if (m.H2 == 256) HWR_MLP(256, 3);
        else if (m.H2 == 128) HWR_MLP(128, 3);
        else HWR_MLP(0, 3);
    } else {
        if (m.H2 == 256) HWR_MLP(256, 2);
        else if (m.H2 == 128) HWR_MLP(128, 2);
        else HWR_MLP(0, 2);
    }
#undef HWR_MLP
    if (e == cudaSuccess) *ctas = grid;
    return e;
}

size_t tc_head_consts_bytes() { return sizeof(HeadConsts); }

void tc_fill_head_consts(void *dst, const float *b2, const float *W3, const float *b3, int H2,
                         int NH) {
    HeadConsts *h = (HeadConsts *)dst;
    memset(h, 0, sizeof *h);
    for (int i = 0; i < H2; ++i) {
        h->nb2[i] = -b2[i];
        h->w0[i] = W3[i];
        h->w1[i] = W3[H2 + i];
        h->w2[i] = NH == 3 ? W3[2 * H2 + i] : 0.f;
    }
    for (int o = 0; o < NH; ++o) {
        double s = b3[o];
        for (int i = 0; i < H2; ++i) s += (double)W3[(size_t)o * H2 + i] * b2[i];
        h->b3[o] = (float)s;
    }
}

}  // namespace hwr
