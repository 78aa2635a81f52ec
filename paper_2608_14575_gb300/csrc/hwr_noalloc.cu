// hwr_route_batch_noalloc: routing without any allocation at call time.
//
// Some callers cannot allocate GPU memory when they route: a router embedded
// in an LLM serving process whose engine has reserved nearly all of HBM up
// front (its KV-cache pool), or a latency-critical serving loop that must not
// take cudaMalloc's device-wide synchronisation.  hwr_route_batch grows its
// scratch on demand with cudaMalloc; this entry point instead runs the same
// bf16 tensor-core kernels with their scratch in one fixed array that the
// library places in device memory when it is loaded.
//
// The array is shared by every call on a device and keeps the last call's
// contents; the per-row arrival counters, which must start at zero, are
// cleared (cudaMemsetAsync, not an allocation) on every call.  Two calls
// whose kernels overlap on the GPU -- on different streams, or on contexts
// of different threads -- race on the array: order them.
#include <stdio.h>

#include <mutex>

#include "hwr_internal.cuh"

hwr_status hwr_internal_fail(hwr_ctx *c, hwr_status s, const char *msg);
int hwr_internal_device(const hwr_ctx *c);
hwr_status hwr_internal_route_tensor_scratch(hwr_ctx *c, int32_t Q, const float *in_len,
                                             const float *out_len, const void *q_emb, float slo,
                                             float lambda, uint32_t flags, int32_t *chosen,
                                             float *pred_latency, float *utility, float *qual,
                                             void *part, int32_t *count, int max_split);

namespace {

constexpr int32_t NOALLOC_MAX_Q = HWR_NOALLOC_MAX_Q;
constexpr int NOALLOC_MAX_SPLIT = 4;
constexpr size_t QUAL_BYTES = (size_t)NOALLOC_MAX_Q * 32 * sizeof(float);   // [Q][Mpad <= 32]
constexpr size_t PART_BYTES = (size_t)NOALLOC_MAX_SPLIT * NOALLOC_MAX_Q * 16;
constexpr size_t COUNT_BYTES = (size_t)NOALLOC_MAX_Q * sizeof(int32_t);
constexpr size_t SCRATCH_BYTES = QUAL_BYTES + PART_BYTES + COUNT_BYTES;   // 6.1 MiB

constexpr int MAX_DEVICES = 64;
std::mutex g_mu;
unsigned char *g_dev_ptr[MAX_DEVICES];

}  // namespace

// The scratch.  In host code this name is only a stand-in for the symbol:
// its device address comes from cudaGetSymbolAddress, per device.
static __device__ __align__(256) unsigned char g_noalloc_scratch[SCRATCH_BYTES];

// Device address of the scratch on device `dev` (the current device),
// resolved on the first call made with that device current.
static cudaError_t scratch_on_device(int dev, unsigned char **out) {
    cudaError_t e;
    if (dev < 0 || dev >= MAX_DEVICES) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_dev_ptr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_dev_ptr[dev] = (unsigned char *)p;
    }
    *out = g_dev_ptr[dev];
    return cudaSuccess;
}

extern "C" hwr_status hwr_route_batch_noalloc(hwr_ctx *ctx, int32_t Q, const float *in_len,
                                              const float *out_len, const void *q_emb, float slo,
                                              float lambda, uint32_t flags, int32_t *chosen,
                                              float *pred_latency, float *utility) {
    if (!ctx) return HWR_ERR_INVALID_ARG;
    const uint32_t allowed = HWR_DEVICE_PTRS | HWR_ASYNC | HWR_SCORE_CONVEX;
    if (flags & ~allowed)
        return hwr_internal_fail(ctx, HWR_ERR_INVALID_ARG,
                                 "noalloc route accepts only HWR_DEVICE_PTRS, HWR_ASYNC and "
                                 "HWR_SCORE_CONVEX");
    if (Q < 0) return hwr_internal_fail(ctx, HWR_ERR_INVALID_ARG, "Q < 0");
    if (Q > NOALLOC_MAX_Q) {
        char msg[128];
        snprintf(msg, sizeof msg, "Q=%d exceeds the noalloc maximum of %d queries", Q,
                 NOALLOC_MAX_Q);
        return hwr_internal_fail(ctx, HWR_ERR_UNSUPPORTED, msg);
    }
    // the scratch of the context's own device: one device's array handed to
    // kernels on another would be the wrong memory
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return hwr_internal_fail(ctx, HWR_ERR_CUDA, "no current CUDA device");
    }
    if (dev != hwr_internal_device(ctx))
        return hwr_internal_fail(ctx, HWR_ERR_INVALID_ARG,
                                 "the current CUDA device is not the context's device");
    unsigned char *base = nullptr;
    const cudaError_t e = scratch_on_device(dev, &base);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return hwr_internal_fail(ctx, HWR_ERR_CUDA, "cannot resolve the noalloc scratch address");
    }
    float *qual = (float *)base;
    void *part = base + QUAL_BYTES;
    int32_t *count = (int32_t *)(base + QUAL_BYTES + PART_BYTES);
    return hwr_internal_route_tensor_scratch(ctx, Q, in_len, out_len, q_emb, slo, lambda, flags,
                                             chosen, pred_latency, utility, qual, part, count,
                                             NOALLOC_MAX_SPLIT);
}
