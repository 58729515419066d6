// gs_decide.cuh -- the keep decision of section 3 and the cap threshold of
// Algorithm 3, shared by the chunked kernels (gs_kernels.cu) and the
// cluster-resident small-input kernel (gs_small.cu) so that both decide
// every coordinate with the same arithmetic.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "gs_device.cuh"

namespace gs {
namespace {

// cap_threshold kept out of line in the solve kernels: it is called from
// several places, and inlining each copy (with its loops) bloats the code the
// solve's single busy warp has to fetch.
__device__ __noinline__ float cap_threshold_call(double lam) { return cap_threshold(lam); }

// cap_threshold by a whole warp (all 32 lanes, same lam; every lane gets the
// result): the 32 floats around the fp32 reciprocal of lam are tested side by
// side, one fp64 product each.  fl64(lam a) >= 1 is monotone in a, so the
// ballot is one run of ones from some lane up; when that lane is not lane 0
// the smallest qualifying float lies in the window (the reciprocal is within
// a few ulps of it), else the serial search decides.
__device__ __forceinline__ float warp_cap_threshold(double lam) {
    const int lane = threadIdx.x & 31;
    const float f = (float)lam;
    if (lam > 0.0 && f > 0.0f && f < 3.0e38f) {
        const uint32_t b0 = __float_as_uint(__frcp_rn(f));
        if (b0 > 16u && b0 < 0x7F7FFFFFu - 16u) {
            const uint32_t b = b0 - 16u + (uint32_t)lane;
            const uint32_t bal = __ballot_sync(0xFFFFFFFFu, lam * (double)__uint_as_float(b) >= 1.0);
            if (bal != 0u && (bal & 1u) == 0u) return __uint_as_float(b0 - 16u + (uint32_t)(__ffs(bal) - 1));
        }
    }
    return cap_threshold_call(lam);
}

// ---------------------------------------------------------------------------
// Decision for one candidate: Z_i = [u_i < p_i] with p_i = min(fl64(lam |g_i|), 1)
// and u_i = x 2^-32 (section 3).  fp32 decides whenever u is more than 2^-21
// away from p; closer calls are settled in fp64.  Kept values
// are g_i / p_i: g_i itself when capped, else sign(g_i) / lambda (the
// constant-value form of section 5.3).
// ---------------------------------------------------------------------------
// The exact fp64 comparison, kept out of line so that the compiler cannot
// evaluate it (fp64 is slow on this part) for the common, certain calls.
__device__ __noinline__ bool exact_keep(uint32_t x, double lam, float a) {
    return (double)x * 0x1p-32 < lam * (double)a;
}

struct Decider {
    double lam;
    float lam32, a_cap, inv_lam32;
    __device__ __forceinline__ bool operator()(float gv, uint32_t x, float& val) const {
        const float a = fabsf(gv);
        if (a >= a_cap) {
            val = gv;
            return true;
        }
        // 1 + u lies in [uf, uf + 2^-23) with uf exact; 1 + p is within 2^-23 of
        // pf.  Outside a 2^-21 band the fp32 comparison is certain; inside it
        // (probability ~2^-20 per candidate) fp64 decides.
        const float uf = unit_plus_one(x);
        const float pf = fmaf(lam32, a, 1.0f);
        bool keep;
        if (uf + 0x1p-21f < pf) keep = true;
        else if (uf - 0x1p-21f > pf) keep = false;
        else keep = exact_keep(x, lam, a);
        val = copysignf(inv_lam32, gv);
        return keep;
    }
};

}  // namespace
}  // namespace gs
