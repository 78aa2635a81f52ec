// The decision maker's reduction (HW-Router Sec. 3.2 (4), Eq. 3), shared by
// the SIMT and tensor-core kernels.
#pragma once

namespace hwr {

// Candidate of the decision maker.  cls 2: feasible (C <= SLO, U defined),
// ordered by larger U; cls 1: defined C, ordered by smaller C; cls 0: NaN C;
// cls -1: no candidate.  Ties go to the lower deployment index.  This is a
// strict total order, so a tree reduction returns the same deployment as a
// left-to-right scan.
struct Cand {
    int cls;
    int d;
    float C, U;
};

__device__ __forceinline__ Cand make_cand(float C, float U, int d, float slo) {
    Cand c;
    c.d = d;
    c.C = C;
    c.U = U;
    if (C != C) c.cls = 0;
    else if (C <= slo && U == U) c.cls = 2;
    else c.cls = 1;
    return c;
}

__device__ __forceinline__ bool better(const Cand &a, const Cand &b) {
    if (a.cls != b.cls) return a.cls > b.cls;
    if (a.cls == 2) {
        if (a.U > b.U) return true;
        if (a.U < b.U) return false;
    } else if (a.cls == 1) {
        if (a.C < b.C) return true;
        if (a.C > b.C) return false;
    }
    return a.d < b.d;
}

// 32-bit key that orders non-NaN floats as the floats compare (+0 and -0
// map to the same key).
__device__ __forceinline__ uint32_t order_key(float x) {
    uint32_t u = __float_as_uint(x);
    u = (u << 1) == 0u ? 0u : u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Best candidate of a full warp under `better`, on every lane.  Three warp
// reductions: the best class, then within it the best key (larger U for
// class 2, smaller C for class 1), then the lowest deployment among the
// lanes holding that key; C and U come from the lane that holds the winner.
// Keys of participating lanes are never 0 (a NaN would be needed), so the 0
// of the other lanes never wins.
__device__ __forceinline__ Cand warp_best(Cand c) {
    const unsigned full = 0xffffffffu;
    const int cls = (int)__reduce_max_sync(full, (unsigned)(c.cls + 1)) - 1;
    uint32_t key = 0u;
    if (c.cls == cls) key = cls == 2 ? order_key(c.U) : cls == 1 ? ~order_key(c.C) : 1u;
    const uint32_t kmax = __reduce_max_sync(full, key);
    const bool tied = c.cls == cls && key == kmax;
    const uint32_t dmin = __reduce_min_sync(full, tied ? (uint32_t)c.d : 0xffffffffu);
    const int src = __ffs(__ballot_sync(full, tied && (uint32_t)c.d == dmin)) - 1;
    Cand b;
    b.cls = cls;
    b.d = (int)dmin;
    b.C = __shfl_sync(full, c.C, src);
    b.U = __shfl_sync(full, c.U, src);
    return b;
}

__device__ __forceinline__ Cand no_cand() {
    Cand c;
    c.cls = -1;
    c.d = 0x7fffffff;
    c.C = 0.f;
    c.U = 0.f;
    return c;
}

}  // namespace hwr
