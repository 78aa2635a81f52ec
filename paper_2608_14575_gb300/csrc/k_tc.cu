// bf16 tensor-core kernels (tcgen05 + TMA) of the route-scoring path.
#include <string.h>

#include "hwr_internal.cuh"

namespace hwr {

// Shared-memory operand images for UMMA, K-major with the 128-byte swizzle:
// the K extent is cut into chunks of 64 bf16 (128 bytes); chunk c holds one
// 128-byte row per matrix row n, and inside each row the 16-byte granule g
// is stored at position g ^ (n % 8).  Chunks follow each other.
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

bool tc_supported(int, int, int, int) { return false; }

cudaError_t tc_prepare() { return cudaSuccess; }

cudaError_t launch_qual_tc(const TcModel &, const Queries &, float *, int32_t *, cudaStream_t) {
    return cudaErrorNotSupported;
}

cudaError_t launch_mlp_tc(const TcModel &, const Queries &, const float *, int32_t *, cudaStream_t) {
    return cudaErrorNotSupported;
}

}  // namespace hwr
