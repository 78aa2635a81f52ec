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

__device__ __forceinline__ Cand warp_best(Cand c) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
        Cand o;
        o.cls = __shfl_xor_sync(0xffffffffu, c.cls, off);
        o.d = __shfl_xor_sync(0xffffffffu, c.d, off);
        o.C = __shfl_xor_sync(0xffffffffu, c.C, off);
        o.U = __shfl_xor_sync(0xffffffffu, c.U, off);
        if (better(o, c)) c = o;
    }
    return c;
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
