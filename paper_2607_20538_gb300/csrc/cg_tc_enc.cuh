// cg_tc_enc.cuh -- pieces shared by the tensor-core encoders (cg_tc.cu: KIVI keys,
// cg_tc_rows.cu: block-uniform rows and KIVI value rows), head dim d = 128.
//
// The rotation z~ = x G^T runs on tcgen05 with G split exactly into three bf16 terms
// (hi + lo + lo2, exact for normal fp32 values; any residual is bounded). The library
// defines z as a fixed-order fp32 sum (pairwise summation of the products;
// include/codecgauge.h), so for every output channel i the converter bounds
// |z~_i - z_i| / ||x_group||_2 by
//     e_i = (c_order + c_tc) ||G_i||_2 + ||G_i - sum of split terms||_2,
// c_order = (1 + log2 g) u the rounding bound of the fixed order, c_tc a bound on the
// tensor-core fp32 accumulation: the MMAs accumulate the split's two small terms first
// (partial sums below 2^-7 of ||G_i|| ||x||, 2 n_hi K-steps) and the leading term last
// (n_hi = K / 16 steps), so c_tc = (n_hi + 4 + 2 n_hi / 128) u, 4 u covering the rounding
// inside each MMA and of the result; the measured |z~ - Gx| stays below 2.4 u ||G_i|| ||x||
// (g = 32 and 128; random, Hadamard and DCT gauges). Candidates that the bound leaves
// undecided are recomputed exactly in the library's order (run_jobs).
#pragma once

#include <cuda_bf16.h>

#include "cg_sm100.cuh"
#include "cg_tc_common.cuh"

namespace cg {
namespace tce {

using namespace sm100;
using tc::kD;

constexpr int kNPass = 3;             // bf16 terms of the gauge split
constexpr int kSegBufs = 4;           // gauge-set slots of the per-block bound coefficients
constexpr float kU = 5.9604645e-08f;  // 2^-24
constexpr float kMagic = 12582912.0f; // 1.5 * 2^23: adding it rounds to an integer (RNE)

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

__device__ __forceinline__ float min3f(float a, float b, float c) {
    float r;
    asm("min.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}
__device__ __forceinline__ float max3f(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}

// Rows of the gauge channels whose error bounds block bk's values: the whole gauge group
// when the group spans the block, else the block's own channels.
__host__ __device__ __forceinline__ void bound_range(int bk, int g, int blk, int& lo, int& hi) {
    if (g >= blk) {
        lo = ((bk * blk) / g) * g;
        hi = lo + g;
    } else {
        lo = bk * blk;
        hi = lo + blk;
    }
}

// One warp-wide round of exact recomputation of the queued gauge-space values (job word:
// row | col << 8; the value goes to the next word), in the library's fixed order. A team
// of T = g/4 lanes computes one value: lane j forms the products of channels 4j..4j+3 and
// their pairwise sum, and the team combines its partial sums with xor-shuffles, which
// follows the same pairwise tree. Each lane loads the operands of kSlots values before any
// arithmetic, so one memory round trip serves kSlots x (32 / T) values. `stage` is the
// staged bf16 tile (two 64-column halves, 128-byte swizzle), Gf the gauge set in global
// memory.
template <int kSlots>
__device__ __forceinline__ void run_jobs(uint32_t* qjob, int nq, const unsigned char* stage, const float* Gf, int g,
                                      int lane) {
    const int lgT = 29 - __clz(g);  // log2(g / 4); g in {8, ..., 128}
    const int T = 1 << lgT, teams = 32 >> lgT;
    const int tm = lane >> lgT, j = lane & (T - 1);
    for (int base = 0; base < nq; base += kSlots * teams) {
        uint2 xv[kSlots];
        float4 gv[kSlots];
#pragma unroll
        for (int k = 0; k < kSlots; k++) {
            const int c = base + k * teams + tm;
            const uint32_t jb = qjob[2 * (c < nq ? c : 0)];
            const int row = (int)(jb & 0xffu), col = (int)((jb >> 8) & 0xffu);
            const int kk = (col & ~(g - 1)) + 4 * j;  // first channel of this lane's products
            xv[k] = *reinterpret_cast<const uint2*>(stage + (kk >> 6) * 16384 + row * 128 +
                                                    ((((kk & 63) >> 3) ^ (row & 7)) << 4) + (kk & 7) * 2);
            gv[k] = ldg_hint_f4(Gf + (size_t)col * g + 4 * j, policy_evict_last());  // kept in L2
        }
        float part[kSlots];
#pragma unroll
        for (int k = 0; k < kSlots; k++) {
            const float p0 = __fmul_rn(gv[k].x, bf_lo(xv[k].x)), p1 = __fmul_rn(gv[k].y, bf_hi(xv[k].x));
            const float p2 = __fmul_rn(gv[k].z, bf_lo(xv[k].y)), p3 = __fmul_rn(gv[k].w, bf_hi(xv[k].y));
            part[k] = __fadd_rn(__fadd_rn(p0, p1), __fadd_rn(p2, p3));
        }
        for (int w = 1; w < T; w <<= 1) {
#pragma unroll
            for (int k = 0; k < kSlots; k++) part[k] = __fadd_rn(part[k], __shfl_xor_sync(0xffffffffu, part[k], w));
        }
        if (j == 0) {
#pragma unroll
            for (int k = 0; k < kSlots; k++) {
                const int c = base + k * teams + tm;
                if (c < nq) qjob[2 * c + 1] = __float_as_uint(part[k]);
            }
        }
    }
}

// The constant part of a packed word built from y = 0x4B400000 + q: the wrapping sum of
// 0x4B400000 << s over the codes of a 32-code chunk that start in word w.
template <int BITS>
__host__ __device__ constexpr uint32_t pack_bias(int w) {
    uint32_t k = 0;
    for (int c = 0; c < 32; c++)
        if ((c * BITS) >> 5 == w) k += 0x4B400000u << ((c * BITS) & 31);
    return k;
}

__device__ __forceinline__ uint32_t scale16(float mx, float mn, float qmax) {
    return f2h_bits(__fdiv_rn(__fsub_rn(mx, mn), qmax));
}

// Overwrite the BITS-bit code at bit position `bit` of a packed row in global memory
// (the row was stored by this thread; the rare exact recomputes are patched in place).
template <int BITS>
__device__ __forceinline__ void patch_code(uint8_t* rowp, int bit, uint32_t q) {
    unsigned int* wp = reinterpret_cast<unsigned int*>(rowp) + (bit >> 5);
    const int off = bit & 31;
    const uint32_t msk = (1u << BITS) - 1u;
    atomicAnd(wp, ~(msk << off));
    atomicOr(wp, q << off);
    if (off + BITS > 32) {
        const int sh = 32 - off;
        atomicAnd(wp + 1, ~(msk >> sh));
        atomicOr(wp + 1, q >> sh);
    }
}

// Warm L2 with the gauge set of the unit after (l, s, h) in this CTA's walk order.
__device__ __forceinline__ void prefetch_next_gauges(const RowArgs& a, const tc::TileInfo& ti, int g, int lane) {
    int nl = ti.l, ns = ti.s, nh = ti.h + 1;
    if (nh == a.H) {
        nh = 0;
        if (++ns == a.s_lo + a.s_n) {
            ns = a.s_lo;
            nl++;
        }
    }
    if (nl < a.L) {
        const char* nG = reinterpret_cast<const char*>(a.G + ((int64_t)(nl * 2 + ns) * a.H + nh) * (int64_t)kD * g);
        for (int off = lane * 128; off < kD * g * 4; off += 32 * 128) asm volatile("prefetch.global.L2::evict_last [%0];" ::"l"(nG + off));
    }
}

// Converts rows of the gauge set Gf (d/g diagonal g x g blocks, fp32) into the MMA's B
// operand: output channel n is B row n, its K entries the gauge row. A lane takes the NQ
// rows n = lane + 32 q, q0 <= q < q0 + NQ, so one to four warps can share a set. The split
// is exact by truncation: hi = v with its low 16 bits cleared, lo the same of v - hi, lo2
// of the rest (for normal values nothing remains; a remainder is bounded below); the terms
// go to bsplit + (npass - 1 - t) * bsz, so the smallest is accumulated first (|lo| < 2^-7
// |hi|, |lo2| < 2^-14 |hi|). Layout: full K = 128 (`fullk`, block-diagonal for g < 128) in
// two 64-column SW128 halves of 16 KB, or one g-wide K block per group in a 64-column tile.
// Writes, per quantization block bk < nbk (keys: slot 0 for all rows), the largest bound
// coefficient e_i over this warp's rows that bound the block (emax[bk]) and the largest
// ||G_i|| among them (gmax[bk]); the readers take the maximum over the warps. Returns true
// when the split of every row of this warp is exact (no remainder: normal values).
template <bool KEYS, int NQ>
__device__ __forceinline__ bool convert_gauge_set(const float* Gf, int g, int blk, int nbk, bool fullk, uint32_t bsz,
                                                  unsigned char* bsplit, float* emax, float* gmax, int q0, int lane) {
    const int lg = 31 - __clz(g);
    const float c_order = (float)(1 + lg) * kU * 1.01f;
    const int n_hi = (KEYS ? 128 : (g < 16 ? 16 : g)) / 16;
    const float c_tc = ((float)n_hi + 4.0f + (float)((kNPass - 1) * n_hi) * (1.0f / 128.0f)) * kU;
    float e_row[NQ], s_g2[NQ], s_res2[NQ];
#pragma unroll
    for (int q = 0; q < NQ; q++) s_g2[q] = s_res2[q] = 0.0f;
    // eight values of each row per step; the next step's loads are in flight while this step
    // converts (a gauge change stalls the MMAs until the set is ready)
    float4 n0[NQ], n1[NQ];
#pragma unroll
    for (int q = 0; q < NQ; q++) {
        const float* Gr = Gf + (size_t)(lane + 32 * (q0 + q)) * g;
        n0[q] = __ldg(reinterpret_cast<const float4*>(Gr));
        n1[q] = __ldg(reinterpret_cast<const float4*>(Gr + 4));
    }
    for (int j = 0; j < g; j += 8) {
        float4 v0[NQ], v1[NQ];
#pragma unroll
        for (int q = 0; q < NQ; q++) {
            v0[q] = n0[q];
            v1[q] = n1[q];
        }
        if (j + 8 < g) {
#pragma unroll
            for (int q = 0; q < NQ; q++) {
                const float* Gr = Gf + (size_t)(lane + 32 * (q0 + q)) * g;
                n0[q] = __ldg(reinterpret_cast<const float4*>(Gr + j + 8));
                n1[q] = __ldg(reinterpret_cast<const float4*>(Gr + j + 12));
            }
        }
#pragma unroll
        for (int q = 0; q < NQ; q++) {
            const int n = lane + 32 * (q0 + q);  // B row = output channel
            const int k = (n / g) * g + j;
            const float v[8] = {v0[q].x, v0[q].y, v0[q].z, v0[q].w, v1[q].x, v1[q].y, v1[q].z, v1[q].w};
            uint32_t tb[3][8];  // term bit patterns (fp32 with the low 16 bits clear)
#pragma unroll
            for (int e = 0; e < 8; e++) {
                float rest = v[e];
                s_g2[q] = fmaf(v[e], v[e], s_g2[q]);
#pragma unroll
                for (int t = 0; t < 3; t++) {
                    tb[t][e] = __float_as_uint(rest) & 0xffff0000u;
                    rest = __fsub_rn(rest, __uint_as_float(tb[t][e]));  // exact
                }
                s_res2[q] = fmaf(rest, rest, s_res2[q]);
            }
#pragma unroll
            for (int t = 0; t < 3; t++) {
                unsigned char* region = bsplit + (kNPass - 1 - t) * bsz + (fullk ? (k >> 6) * 16384 : 0);
                *reinterpret_cast<uint4*>(region + sw128_offset(n, k & 63)) =
                    make_uint4(__byte_perm(tb[t][0], tb[t][1], 0x7632), __byte_perm(tb[t][2], tb[t][3], 0x7632),
                               __byte_perm(tb[t][4], tb[t][5], 0x7632), __byte_perm(tb[t][6], tb[t][7], 0x7632));
            }
        }
    }
#pragma unroll
    for (int q = 0; q < NQ; q++) e_row[q] = ((c_order + c_tc) * sqrtf(s_g2[q]) + sqrtf(s_res2[q])) * 1.001f + 1e-30f;
    // per quantization block: max of e over the rows that bound its values (keys: a block is
    // one channel over tokens, bounded by the max over all rows, slot 0)
#pragma unroll
    for (int bk = 0; bk < 4; bk++) {
        if (KEYS ? bk == 0 : bk < nbk) {
            int lo = 0, hi = 128;
            if (!KEYS) bound_range(bk, g, blk, lo, hi);
            float m = 0.0f, gm = 0.0f;  // gm: max_i ||G_i|| over the same rows, bounds |z~| / ||x||
#pragma unroll
            for (int q = 0; q < NQ; q++) {
                const int n = lane + 32 * (q0 + q);
                if (n >= lo && n < hi) {
                    m = fmaxf(m, e_row[q]);
                    gm = fmaxf(gm, sqrtf(s_g2[q]));
                }
            }
            for (int off = 16; off >= 1; off >>= 1) {
                m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
                gm = fmaxf(gm, __shfl_xor_sync(0xffffffffu, gm, off));
            }
            if (lane == 0) {
                emax[bk] = m;
                gmax[bk] = gm;
            }
        }
    }
    bool rem = false;
#pragma unroll
    for (int q = 0; q < NQ; q++) rem = rem || s_res2[q] != 0.0f;
    return !__any_sync(0xffffffffu, rem);
}

}  // namespace tce
}  // namespace cg
