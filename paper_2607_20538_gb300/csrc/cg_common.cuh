// cg_common.cuh -- device-side definitions shared by the libcodecgauge kernels.
// (GPU path only; the CPU oracle has its own, independent code.)
#pragma once

#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "../../include/codecgauge.h"

namespace cg {

// Kernels accumulate CG_FLAG_* bits into a per-device status word whose address the
// host passes in (see cg_api.cu).
__device__ __forceinline__ void raise_flag(int32_t* status, int32_t f) {
    if (f) atomicOr(status, f);
}

__device__ __forceinline__ float bf16_bits_to_float(uint32_t b) {
    return __uint_as_float(b << 16);
}

__device__ __forceinline__ bool bf16_nonfinite(uint32_t b) {
    return ((b >> 7) & 0xffu) == 0xffu;
}

// fp32 -> fp16 bits, round to nearest even.
__device__ __forceinline__ uint32_t f2h_bits(float f) {
    return (uint32_t)__half_as_ushort(__float2half_rn(f));
}

__device__ __forceinline__ float h2f_bits(uint32_t h) {
    return __half2float(__ushort_as_half((unsigned short)h));
}

__device__ __forceinline__ bool h_is_inf(uint32_t h) { return (h & 0x7fffu) == 0x7c00u; }

// Block scale/zero of the asymmetric min/max rule: s = fp16((max-min)/qmax), m = fp16(min).
// Returns packed half2 bits {s (low 16), m (high 16)} and sets *flag on fp16 overflow.
__device__ __forceinline__ uint32_t scale_zero(float mn, float mx, float qmax, int32_t* flag) {
    float s32 = __fdiv_rn(__fsub_rn(mx, mn), qmax);
    uint32_t s16 = f2h_bits(s32), m16 = f2h_bits(mn);
    if (h_is_inf(s16) || h_is_inf(m16)) *flag |= CG_FLAG_FP16_OVERFLOW;
    return s16 | (m16 << 16);
}

// Code of one value given the decoded fp16 scale s and zero m (both as fp32).
__device__ __forceinline__ uint32_t quant_code(float z, float s, float m, int qmax) {
    if (s == 0.0f) return 0u;
    float t = __fdiv_rn(__fsub_rn(z, m), s);
    int q = __float2int_rn(t);  // round half to even
    q = q < 0 ? 0 : (q > qmax ? qmax : q);
    return (uint32_t)q;
}

// Pairwise fp32 sum of 8 products a[k] * b[k] (k = 0..7), the leaves of the library's
// fixed summation order; explicit round-to-nearest ops so nothing is contracted.
__device__ __forceinline__ float tree8(const float (&a)[8], const float (&b)[8]) {
    const float p0 = __fmul_rn(a[0], b[0]), p1 = __fmul_rn(a[1], b[1]), p2 = __fmul_rn(a[2], b[2]),
                p3 = __fmul_rn(a[3], b[3]), p4 = __fmul_rn(a[4], b[4]), p5 = __fmul_rn(a[5], b[5]),
                p6 = __fmul_rn(a[6], b[6]), p7 = __fmul_rn(a[7], b[7]);
    return __fadd_rn(__fadd_rn(__fadd_rn(p0, p1), __fadd_rn(p2, p3)), __fadd_rn(__fadd_rn(p4, p5), __fadd_rn(p6, p7)));
}

// Pairwise combination of n (a power of two <= 16) partial sums s[0..n), in place.
__device__ __forceinline__ float tree_combine(float (&s)[16], int n) {
#pragma unroll
    for (int w = 1; w < 16; w *= 2) {
#pragma unroll
        for (int i = 0; i + w < 16; i += 2 * w)
            if (w < n && i + w < n) s[i] = __fadd_rn(s[i], s[i + w]);
    }
    return s[0];
}

// KIVI split: quantized tokens form whole groups of Gt; the newest T - nq >= R stay raw.
__host__ __device__ __forceinline__ int64_t kivi_nq(int64_t T, int64_t R, int64_t Gt) {
    return T <= R ? 0 : ((T - R) / Gt) * Gt;
}

// Byte/element strides that place one row (one token of one (l, s, b, h)) of the packed
// outputs; row offset = base + l*sL + s*sS + b*sB + h*sH + (t >> tshift)*sT. A shift of 4
// maps the 16 tokens of a block-uniform tile to the tile's one set of scales.
struct RowMap {
    int64_t base, sL, sS, sB, sH, sT;
    int tshift;
    __host__ __device__ __forceinline__ int64_t at(int l, int s, int b, int h, int64_t t) const {
        return base + l * sL + s * sS + b * sB + h * sH + (t >> tshift) * sT;
    }
};

}  // namespace cg
