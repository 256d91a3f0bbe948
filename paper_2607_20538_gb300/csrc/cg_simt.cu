// cg_simt.cu -- CUDA-core kernels of the encode/decode path.
//
// These kernels evaluate the gauge rotation Z = G X (Sec. 3) exactly as the library's
// quantization rule defines it (pairwise fp32 summation of the products), so scales,
// zeros and codes are reproducible to the bit. They serve every shape the library accepts and are the launch choice where a
// tile of tokens is too small or the group too small for the tensor-core kernels.
//
// Thread mapping (row kernels): one warp per token row; lane owns channels c = lane + 32k.
// The (l, s, h) gauge set sits in shared memory; one CTA handles 64 rows (b, t) that
// share it.
#include "cg_launch.h"

namespace cg {
namespace {

constexpr int kRowThreads = 256;
constexpr int kRowWarps = kRowThreads / 32;
constexpr int kRowsPerCta = 64;

__device__ __forceinline__ float seg_min(float v, int seg) {
    for (int off = seg >> 1; off >= 1; off >>= 1) v = fminf(v, __shfl_xor_sync(0xffffffffu, v, off));
    return v;
}
__device__ __forceinline__ float seg_max(float v, int seg) {
    for (int off = seg >> 1; off >= 1; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
    return v;
}

// One gauge-space coordinate sum_j G[i][j] x[j] in the library's fixed fp32 order:
// pairwise summation of the products. The 8-product leaves are summed as trees and merged
// in chunk order with a binary carry (the partial sum of 2^k chunks waits at level k), which
// reproduces the pairwise tree for a power-of-two count of chunks. Gcol[j * gstride] =
// G[i][j]; g a power of two in [8, 128].
__device__ __forceinline__ float gauge_coord(const float* Gcol, int gstride, const float* x, int g) {
    float l0 = 0.0f, l1 = 0.0f, l2 = 0.0f, l3 = 0.0f, v = 0.0f;
#pragma unroll 1
    for (int c = 0; c < g / 8; c++) {
        float a[8], b[8];
#pragma unroll
        for (int k = 0; k < 8; k++) {
            a[k] = Gcol[(8 * c + k) * gstride];
            b[k] = x[8 * c + k];
        }
        v = tree8(a, b);
        if (c & 1) {
            v = __fadd_rn(l0, v);
            if (c & 2) {
                v = __fadd_rn(l1, v);
                if (c & 4) {
                    v = __fadd_rn(l2, v);
                    if (c & 8) v = __fadd_rn(l3, v);
                    else l3 = v;
                } else {
                    l2 = v;
                }
            } else {
                l1 = v;
            }
        } else {
            l0 = v;
        }
    }
    return v;
}

// Extract the b-bit code that starts at bit p of a little-endian word stream.
__device__ __forceinline__ uint32_t extract_code(const uint32_t* w, int p, int bits) {
    int wi = p >> 5, off = p & 31;
    uint32_t v = w[wi] >> off;
    if (off + bits > 32) v |= w[wi + 1] << (32 - off);
    return v & ((1u << bits) - 1u);
}

// Word w of the little-endian stream in which code c sits at bits [c*bits, (c+1)*bits).
__device__ __forceinline__ uint32_t pack_word(const uint8_t* q, int w, int bits) {
    int bit0 = w * 32, c0 = bit0 / bits, c1 = (bit0 + 31) / bits;
    uint32_t word = 0;
    for (int c = c0; c <= c1; c++) {
        int p = c * bits - bit0;
        uint32_t v = q[c];
        word |= p >= 0 ? (v << p) : (v >> (-p));
    }
    return word;
}

// ------------------------------------------------------------------------------------
// Row encode: Z = G X, then per-token block min/max quantization and packing (or the raw
// fp32 Z for the no-compression rows).
// ------------------------------------------------------------------------------------
template <int NR>
__global__ void __launch_bounds__(kRowThreads) row_encode_kernel(RowArgs a) {
    constexpr int d = NR * 32;
    extern __shared__ __align__(16) unsigned char smem[];
    const int g = a.g;
    float* Gs = reinterpret_cast<float*>(smem);  // Gs[r][jj][i] = G_r[i][jj]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* xs = reinterpret_cast<float*>(smem + (size_t)d * g * 4) + warp * d;
    uint8_t* qs = smem + (size_t)d * g * 4 + (size_t)kRowWarps * d * 4 + warp * d;
    uint32_t* sm = reinterpret_cast<uint32_t*>(smem + (size_t)d * g * 4 + (size_t)kRowWarps * d * 5) + warp * 32;

    const int y = blockIdx.y;
    const int h = y % a.H;
    const int s = a.s_lo + (y / a.H) % a.s_n;
    const int l = y / (a.H * a.s_n);
    const float* Gsrc = a.G + ((int64_t)(l * 2 + s) * a.H + h) * (int64_t)d * g;
    for (int e = threadIdx.x; e < d * g; e += kRowThreads) {
        int r = e / (g * g), rem = e - r * g * g, i = rem / g, jj = rem - i * g;
        Gs[r * g * g + jj * g + i] = __ldg(Gsrc + e);
    }
    __syncthreads();

    const int64_t rows = (int64_t)a.B * a.t_count;
    const int64_t r0 = (int64_t)blockIdx.x * kRowsPerCta;
    const int bits = a.bits, blk = a.blk;
    const int qmax = (1 << bits) - 1;
    const float qmaxf = (float)qmax;
    int32_t flag = 0;

    for (int rr = warp; rr < kRowsPerCta; rr += kRowWarps) {
        const int64_t row = r0 + rr;
        if (row >= rows) break;
        const int b = (int)(row / a.t_count);
        const int64_t t = row - (int64_t)b * a.t_count;
        const uint16_t* xr = a.x + ((((int64_t)(l * 2 + s) * a.B + b) * a.H + h) * a.T_x + t) * d;
        float z[NR];
#pragma unroll
        for (int k = 0; k < NR; k++) {
            uint32_t xb = xr[lane + 32 * k];
            if (bf16_nonfinite(xb)) flag |= CG_FLAG_NONFINITE_INPUT;
            xs[lane + 32 * k] = bf16_bits_to_float(xb);
        }
        __syncwarp();
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k, r = c / g, i = c - r * g;
            z[k] = gauge_coord(Gs + r * g * g + i, g, xs + r * g, g);
        }
        const int64_t coff = a.cmap.at(l, s, b, h, t);
        if (a.none_mode) {
            float* zr = reinterpret_cast<float*>(a.codes + coff);
#pragma unroll
            for (int k = 0; k < NR; k++) zr[lane + 32 * k] = z[k];
            __syncwarp();
            continue;
        }
        // block ranges: segments of min(blk, 32) lanes per register, then registers
        const int seg = blk < 32 ? blk : 32;
        const int per = blk > 32 ? blk / 32 : 1;
        float mn[NR], mx[NR];
#pragma unroll
        for (int k = 0; k < NR; k++) {
            mn[k] = seg_min(z[k], seg);
            mx[k] = seg_max(z[k], seg);
        }
        if (per > 1) {
#pragma unroll
            for (int k = 0; k < NR; k++) {
                const int k0 = (k / per) * per;
                float a0 = mn[k0], a1 = mx[k0];
                for (int kk = 1; kk < per; kk++) {
                    a0 = fminf(a0, mn[k0 + kk]);
                    a1 = fmaxf(a1, mx[k0 + kk]);
                }
                mn[k] = a0;
                mx[k] = a1;
            }
        }
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k;
            const uint32_t sz = scale_zero(mn[k], mx[k], qmaxf, &flag);
            const float sc = h2f_bits(sz & 0xffffu), mz = h2f_bits(sz >> 16);
            qs[c] = (uint8_t)quant_code(z[k], sc, mz, qmax);
            if ((c % blk) == 0) sm[c / blk] = sz;
        }
        __syncwarp();
        uint32_t* cw = reinterpret_cast<uint32_t*>(a.codes + coff);
        const int nw = d * bits / 32;
        for (int w = lane; w < nw; w += 32) cw[w] = pack_word(qs, w, bits);
        const int nb = d / blk;
        if (lane < nb) a.scales[a.smap.at(l, s, b, h, t) + lane] = sm[lane];
        __syncwarp();
    }
    if (flag) raise_flag(a.status, flag);
}

// ------------------------------------------------------------------------------------
// Block-uniform tiles: Z = G X for the 16 tokens of a tile, then one min/max range per
// tile block (16 tokens x blk channels, Sec. 4.3 with T_b = 16 from Sec. 4.2), codes and
// packing in the per-token row layout, one {scale, zero} pair per tile block.
// One warp per tile; the CTA shares the (l, s, h) gauge set in shared memory.
// ------------------------------------------------------------------------------------
constexpr int kTileTokens = CG_TILE_TOKENS;
constexpr int kTileWarpsMax = 16;
constexpr size_t kSmemOptIn = 232448;  // 227 KB of dynamic shared memory per CTA

__host__ __device__ __forceinline__ size_t tile_warp_bytes(int d) {
    return (size_t)kTileTokens * d * 4 + (size_t)kTileTokens * d + 32 * 4;
}

// Binary-carry merge of the chunk sums of one pairwise sum (see gauge_coord).
__device__ __forceinline__ void carry_push(float& l0, float& l1, float& l2, float& l3, float& v, int c) {
    if (c & 1) {
        v = __fadd_rn(l0, v);
        if (c & 2) {
            v = __fadd_rn(l1, v);
            if (c & 4) {
                v = __fadd_rn(l2, v);
                if (c & 8) v = __fadd_rn(l3, v);
                else l3 = v;
            } else {
                l2 = v;
            }
        } else {
            l1 = v;
        }
    } else {
        l0 = v;
    }
}

// gauge_coord for four tokens at once: out[t] = sum_j G[i][j] x_t[j] in the library's
// pairwise order, x_t = x0 + t * xstride (16-byte aligned rows). Each gauge value loaded
// from shared memory serves the four tokens.
__device__ __forceinline__ void gauge_coord4(const float* Gcol, int gstride, const float* x0, int xstride, int g,
                                             float (&out)[4]) {
    float l0[4] = {}, l1[4] = {}, l2[4] = {}, l3[4] = {}, v[4] = {};
#pragma unroll 1
    for (int c = 0; c < g / 8; c++) {
        float a[8];
#pragma unroll
        for (int k = 0; k < 8; k++) a[k] = Gcol[(8 * c + k) * gstride];
#pragma unroll
        for (int t = 0; t < 4; t++) {
            const float4* xp = reinterpret_cast<const float4*>(x0 + t * xstride + 8 * c);
            const float4 u0 = xp[0], u1 = xp[1];
            const float b[8] = {u0.x, u0.y, u0.z, u0.w, u1.x, u1.y, u1.z, u1.w};
            v[t] = tree8(a, b);
            carry_push(l0[t], l1[t], l2[t], l3[t], v[t], c);
        }
    }
#pragma unroll
    for (int t = 0; t < 4; t++) out[t] = v[t];
}

template <int NR>
__global__ void __launch_bounds__(kTileWarpsMax * 32) tile_encode_kernel(RowArgs a) {
    constexpr int d = NR * 32;
    extern __shared__ __align__(16) unsigned char smem[];
    const int g = a.g;
    float* Gs = reinterpret_cast<float*>(smem);  // Gs[r][jj][i] = G_r[i][jj]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nwarps = blockDim.x >> 5;
    unsigned char* wbase = smem + (size_t)d * g * 4 + (size_t)warp * tile_warp_bytes(d);
    float* buf = reinterpret_cast<float*>(wbase);                         // [16][d]: x, then z
    uint8_t* qs = wbase + (size_t)kTileTokens * d * 4;                    // [16][d] codes
    uint32_t* smw = reinterpret_cast<uint32_t*>(qs + (size_t)kTileTokens * d);  // [d/blk] scales

    const int y = blockIdx.y;
    const int h = y % a.H;
    const int s = a.s_lo + (y / a.H) % a.s_n;
    const int l = y / (a.H * a.s_n);
    const float* Gsrc = a.G + ((int64_t)(l * 2 + s) * a.H + h) * (int64_t)d * g;
    for (int e = threadIdx.x; e < d * g; e += blockDim.x) {
        int r = e / (g * g), rem = e - r * g * g, i = rem / g, jj = rem - i * g;
        Gs[r * g * g + jj * g + i] = __ldg(Gsrc + e);
    }
    __syncthreads();

    const int64_t ntc = (a.t_count + kTileTokens - 1) / kTileTokens;  // tiles per unit in this call
    const int64_t total = (int64_t)a.B * ntc;
    const int64_t chunk = (total + gridDim.x - 1) / gridDim.x;
    const int64_t k0 = (int64_t)blockIdx.x * chunk;
    const int64_t k1 = k0 + chunk < total ? k0 + chunk : total;
    const int bits = a.bits, blk = a.blk;
    const int qmax = (1 << bits) - 1;
    const float qmaxf = (float)qmax;
    const int nw = d * bits / 32;  // packed words per token row
    int32_t flag = 0;

    for (int64_t tk = k0 + warp; tk < k1; tk += nwarps) {
        const int b = (int)(tk / ntc);
        const int64_t t_lo = (tk - (int64_t)b * ntc) * kTileTokens;
        const int nt = a.t_count - t_lo < kTileTokens ? (int)(a.t_count - t_lo) : kTileTokens;
        // the tile's tokens are nt consecutive rows of x: nt * d bf16, 16-byte chunks
        const uint4* xt = reinterpret_cast<const uint4*>(
            a.x + ((((int64_t)(l * 2 + s) * a.B + b) * a.H + h) * a.T_x + t_lo) * d);
        for (int e = lane; e < nt * d / 8; e += 32) {
            const uint4 v = __ldg(xt + e);
            const uint32_t w[4] = {v.x, v.y, v.z, v.w};
            float f[8];
#pragma unroll
            for (int k = 0; k < 4; k++) {
                const uint32_t lo = w[k] & 0xffffu, hi = w[k] >> 16;
                if (bf16_nonfinite(lo) || bf16_nonfinite(hi)) flag |= CG_FLAG_NONFINITE_INPUT;
                f[2 * k] = bf16_bits_to_float(lo);
                f[2 * k + 1] = bf16_bits_to_float(hi);
            }
            float4* dst = reinterpret_cast<float4*>(buf + 8 * e);
            dst[0] = make_float4(f[0], f[1], f[2], f[3]);
            dst[1] = make_float4(f[4], f[5], f[6], f[7]);
        }
        __syncwarp();
        // Z for four tokens at a time; each quad's z overwrites its x rows once all lanes
        // have read them
        for (int tq = 0; tq * 4 < nt; tq++) {
            float zq[NR][4];
#pragma unroll
            for (int k = 0; k < NR; k++) {
                const int c = lane + 32 * k, r = c / g, i = c - r * g;
                gauge_coord4(Gs + r * g * g + i, g, buf + (size_t)(4 * tq) * d + r * g, d, g, zq[k]);
            }
            __syncwarp();
#pragma unroll
            for (int t = 0; t < 4; t++)
                if (4 * tq + t < nt) {
#pragma unroll
                    for (int k = 0; k < NR; k++) buf[(4 * tq + t) * d + lane + 32 * k] = zq[k][t];
                }
            __syncwarp();
        }
        // tile block ranges: tokens per lane, then lanes (segments of min(blk, 32)), then
        // registers for blk > 32
        const int seg = blk < 32 ? blk : 32;
        const int per = blk > 32 ? blk / 32 : 1;
        float mn[NR], mx[NR];
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k;
            float lo = buf[c], hi = lo;
            for (int tt = 1; tt < nt; tt++) {
                const float v = buf[tt * d + c];
                lo = fminf(lo, v);
                hi = fmaxf(hi, v);
            }
            mn[k] = seg_min(lo, seg);
            mx[k] = seg_max(hi, seg);
        }
        if (per > 1) {
#pragma unroll
            for (int k = 0; k < NR; k++) {
                const int kb = (k / per) * per;
                float a0 = mn[kb], a1 = mx[kb];
                for (int kk = 1; kk < per; kk++) {
                    a0 = fminf(a0, mn[kb + kk]);
                    a1 = fmaxf(a1, mx[kb + kk]);
                }
                mn[k] = a0;
                mx[k] = a1;
            }
        }
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k;
            const uint32_t sz = scale_zero(mn[k], mx[k], qmaxf, &flag);
            const float sc = h2f_bits(sz & 0xffffu), mz = h2f_bits(sz >> 16);
            for (int tt = 0; tt < nt; tt++) qs[tt * d + c] = (uint8_t)quant_code(buf[tt * d + c], sc, mz, qmax);
            if ((c % blk) == 0) smw[c / blk] = sz;
        }
        __syncwarp();
        for (int e = lane; e < nt * nw; e += 32) {
            const int tt = e / nw, w = e - tt * nw;
            uint32_t* cw = reinterpret_cast<uint32_t*>(a.codes + a.cmap.at(l, s, b, h, t_lo + tt));
            cw[w] = pack_word(qs + tt * d, w, bits);
        }
        if (lane < d / blk) a.scales[a.smap.at(l, s, b, h, t_lo) + lane] = smw[lane];
        __syncwarp();
    }
    if (flag) raise_flag(a.status, flag);
}

// ------------------------------------------------------------------------------------
// Hadamard gauge by fast Walsh-Hadamard transform (the structured Hadamard control of
// Sec. 4.3, G = H_g / sqrt(g) in fp32 for every (l, s, h, r)), O(g log g) per group and no
// gauge tensor read. Every entry of G is +-c, c = fp32(1 / sqrt(g)), so the library's
// products are +-fl(c x_j), and the pairwise summation order over j (adjacent pairs first,
// halves last) is the butterfly order of the transform (stride 1 first, stride g/2 last):
// scaling x by c with rounding and then running the butterflies in fp32 gives exactly the
// library's z. One warp per token row; lane owns CPL = d/32 consecutive channels.
// ------------------------------------------------------------------------------------
template <int CPL>
__device__ __forceinline__ void fwht_lane(float (&v)[CPL], int g, int lane) {
#pragma unroll
    for (int h = 1; h < CPL; h <<= 1) {
        if (h >= g) break;
#pragma unroll
        for (int k = 0; k < CPL; k++)
            if (!(k & h)) {
                const float a = v[k], b = v[k + h];
                v[k] = __fadd_rn(a, b);
                v[k + h] = __fsub_rn(a, b);
            }
    }
    for (int h = CPL; h < g; h <<= 1) {
        const int m = h / CPL;
        const bool hi = (lane & m) != 0;
#pragma unroll
        for (int k = 0; k < CPL; k++) {
            const float o = __shfl_xor_sync(0xffffffffu, v[k], m);
            v[k] = hi ? __fsub_rn(o, v[k]) : __fadd_rn(v[k], o);
        }
    }
}

// CPL consecutive bf16 values (CPL * 2 bytes, naturally aligned) as raw bits.
template <int CPL>
__device__ __forceinline__ void load_bf16(const uint16_t* p, uint32_t (&out)[CPL]) {
    if (CPL == 8) {
        const uint4 v = *reinterpret_cast<const uint4*>(p);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int k = 0; k < CPL; k++) out[k] = (w[k >> 1] >> (16 * (k & 1))) & 0xffffu;
    } else if (CPL == 4) {
        const uint2 v = *reinterpret_cast<const uint2*>(p);
        const uint32_t w[2] = {v.x, v.y};
#pragma unroll
        for (int k = 0; k < CPL; k++) out[k] = (w[k >> 1] >> (16 * (k & 1))) & 0xffffu;
    } else if (CPL == 2) {
        const uint32_t w = *reinterpret_cast<const uint32_t*>(p);
        out[0] = w & 0xffffu;
        out[CPL - 1] = w >> 16;
    } else {
        out[0] = p[0];
    }
}

// The rule's code, clamp(rint(fl((z - m) / s)), 0, qmax), from a reciprocal product: the product
// is within a few ulp of the quotient, so it rounds to the same integer unless it lies within
// 2^-12 of a half-integer, where the exact division decides (rare).
__device__ __forceinline__ uint32_t quant_code_rcp(float z, float s, float m, float rcp, int qmax) {
    if (s == 0.0f) return 0u;
    const float d = __fsub_rn(z, m);
    float t = __fmul_rn(d, rcp);
    if (fabsf(t - floorf(t) - 0.5f) < 2.5e-4f) t = __fdiv_rn(d, s);
    int q = __float2int_rn(t);
    q = q < 0 ? 0 : (q > qmax ? qmax : q);
    return (uint32_t)q;
}

template <int CPL>
__global__ void __launch_bounds__(kRowThreads) hadamard_encode_kernel(RowArgs a, float c) {
    constexpr int d = CPL * 32;
    __shared__ uint8_t qs_all[kRowWarps][d];
    __shared__ uint32_t sm_all[kRowWarps][32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint8_t* qs = qs_all[warp];
    uint32_t* smw = sm_all[warp];
    const int g = a.g, bits = a.bits, blk = a.blk, qmax = (1 << bits) - 1;
    const float qmaxf = (float)qmax;
    const int lanes_per_blk = blk / CPL;  // block >= 8 >= CPL
    const int nb = d / blk, nw = d * bits / 32;
    // grid: x = (l, s, b, h) unit, y = token range; a warp takes tokens in steps of the y extent
    int u = blockIdx.x;
    const int h = u % a.H; u /= a.H;
    const int b = u % a.B; u /= a.B;
    const int s = a.s_lo + u % a.s_n;
    const int l = u / a.s_n;
    const uint16_t* xu = a.x + (((int64_t)(l * 2 + s) * a.B + b) * a.H + h) * a.T_x * d + CPL * lane;
    const int64_t stride = (int64_t)gridDim.y * kRowWarps;
    int32_t flag = 0;
    int64_t t = (int64_t)blockIdx.y * kRowWarps + warp;
    uint32_t xb[CPL];
    if (t < a.t_count) load_bf16<CPL>(xu + t * d, xb);
    for (; t < a.t_count; t += stride) {
        float v[CPL];
#pragma unroll
        for (int k = 0; k < CPL; k++) {
            if (bf16_nonfinite(xb[k])) flag |= CG_FLAG_NONFINITE_INPUT;
            v[k] = __fmul_rn(c, bf16_bits_to_float(xb[k]));
        }
        const int cl = l, cs = s, cb = b, ch_ = h;
        const int64_t ct = t;
        if (t + stride < a.t_count) load_bf16<CPL>(xu + (t + stride) * d, xb);  // next row
        fwht_lane<CPL>(v, g, lane);
        float mn = v[0], mx = v[0];
#pragma unroll
        for (int k = 1; k < CPL; k++) {
            mn = fminf(mn, v[k]);
            mx = fmaxf(mx, v[k]);
        }
        mn = seg_min(mn, lanes_per_blk);
        mx = seg_max(mx, lanes_per_blk);
        const uint32_t sz = scale_zero(mn, mx, qmaxf, &flag);
        const float sc = h2f_bits(sz & 0xffffu), mz = h2f_bits(sz >> 16);
        const float rcp = sc != 0.0f ? __frcp_rn(sc) : 0.0f;
#pragma unroll
        for (int k = 0; k < CPL; k++) qs[CPL * lane + k] = (uint8_t)quant_code_rcp(v[k], sc, mz, rcp, qmax);
        if (((CPL * lane) % blk) == 0) smw[(CPL * lane) / blk] = sz;
        __syncwarp();
        uint32_t* cw = reinterpret_cast<uint32_t*>(a.codes + a.cmap.at(cl, cs, cb, ch_, ct));
        for (int w = lane; w < nw; w += 32) cw[w] = pack_word(qs, w, bits);
        if (lane < nb) a.scales[a.smap.at(cl, cs, cb, ch_, ct) + lane] = smw[lane];
        __syncwarp();
    }
    if (flag) raise_flag(a.status, flag);
}

template <int CPL>
__global__ void __launch_bounds__(kRowThreads) hadamard_decode_kernel(RowArgs a, float c) {
    constexpr int d = CPL * 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = a.g, bits = a.bits, blk = a.blk;
    const int nw = d * bits / 32;
    const uint32_t mask = (1u << bits) - 1u;
    const int bit0 = CPL * lane * bits, wi = bit0 >> 5, sh = bit0 & 31;
    int u = blockIdx.x;  // grid as in the encode kernel
    const int h = u % a.H; u /= a.H;
    const int b = u % a.B; u /= a.B;
    const int s = a.s_lo + u % a.s_n;
    const int l = u / a.s_n;
    for (int64_t t = (int64_t)blockIdx.y * kRowWarps + warp; t < a.t_count; t += (int64_t)gridDim.y * kRowWarps) {
        // this lane's CPL codes: CPL * bits <= 64 bits starting at bit bit0 of the row
        const uint32_t* cw = reinterpret_cast<const uint32_t*>(a.codes + a.cmap.at(l, s, b, h, t));
        const uint32_t w0 = __ldg(cw + wi);
        const uint32_t w1 = wi + 1 < nw ? __ldg(cw + wi + 1) : 0u;
        const uint32_t w2 = wi + 2 < nw ? __ldg(cw + wi + 2) : 0u;
        const uint64_t lo = (((uint64_t)w1 << 32) | w0) >> sh;
        const uint64_t cv = sh ? (lo | ((uint64_t)w2 << (64 - sh))) : lo;
        const uint32_t sz = __ldg(a.scales + a.smap.at(l, s, b, h, t) + (CPL * lane) / blk);
        const float sc = h2f_bits(sz & 0xffffu), mz = h2f_bits(sz >> 16);
        float v[CPL];
#pragma unroll
        for (int k = 0; k < CPL; k++) v[k] = fmaf((float)((uint32_t)(cv >> (k * bits)) & mask), sc, mz);
        fwht_lane<CPL>(v, g, lane);  // H is symmetric: G^T zhat = c H zhat
        uint16_t* orow = a.out + ((((int64_t)(l * 2 + s) * a.B + b) * a.H + h) * a.T_x + t) * d + CPL * lane;
        uint32_t ob[CPL];
#pragma unroll
        for (int k = 0; k < CPL; k++) ob[k] = __bfloat16_as_ushort(__float2bfloat16_rn(c * v[k]));
        if (CPL == 8) {
            *reinterpret_cast<uint4*>(orow) = make_uint4(ob[0] | ob[1 % CPL] << 16, ob[2 % CPL] | ob[3 % CPL] << 16,
                                                         ob[4 % CPL] | ob[5 % CPL] << 16, ob[6 % CPL] | ob[7 % CPL] << 16);
        } else if (CPL == 4) {
            *reinterpret_cast<uint2*>(orow) = make_uint2(ob[0] | ob[1 % CPL] << 16, ob[2 % CPL] | ob[3 % CPL] << 16);
        } else if (CPL == 2) {
            *reinterpret_cast<uint32_t*>(orow) = ob[0] | ob[1 % CPL] << 16;
        } else {
            orow[0] = (uint16_t)ob[0];
        }
    }
}

// ------------------------------------------------------------------------------------
// Row decode: unpack, dequantize zhat = q*s + m, then Xhat = G^T Zhat, bf16 store.
// ------------------------------------------------------------------------------------
template <int NR>
__global__ void __launch_bounds__(kRowThreads) row_decode_kernel(RowArgs a) {
    constexpr int d = NR * 32;
    extern __shared__ __align__(16) unsigned char smem[];
    const int g = a.g;
    float* Gs = reinterpret_cast<float*>(smem);  // Gs[r][jj][i] = G_r[jj][i]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* zs = reinterpret_cast<float*>(smem + (size_t)d * g * 4) + warp * d;
    uint32_t* cwS = reinterpret_cast<uint32_t*>(smem + (size_t)d * g * 4 + (size_t)kRowWarps * d * 4) + warp * (d / 4 + 4);
    uint32_t* sm = reinterpret_cast<uint32_t*>(smem + (size_t)d * g * 4 + (size_t)kRowWarps * d * 4 +
                                               (size_t)kRowWarps * (d / 4 + 4) * 4) + warp * 32;

    const int y = blockIdx.y;
    const int h = y % a.H;
    const int s = a.s_lo + (y / a.H) % a.s_n;
    const int l = y / (a.H * a.s_n);
    const float* Gsrc = a.G + ((int64_t)(l * 2 + s) * a.H + h) * (int64_t)d * g;
    for (int e = threadIdx.x; e < d * g; e += kRowThreads) Gs[e] = __ldg(Gsrc + e);
    __syncthreads();

    const int64_t rows = (int64_t)a.B * a.t_count;
    const int64_t r0 = (int64_t)blockIdx.x * kRowsPerCta;
    const int bits = a.bits, blk = a.blk;

    for (int rr = warp; rr < kRowsPerCta; rr += kRowWarps) {
        const int64_t row = r0 + rr;
        if (row >= rows) break;
        const int b = (int)(row / a.t_count);
        const int64_t t = row - (int64_t)b * a.t_count;
        const int64_t coff = a.cmap.at(l, s, b, h, t);
        if (a.none_mode) {
            const float* zr = reinterpret_cast<const float*>(a.codes + coff);
#pragma unroll
            for (int k = 0; k < NR; k++) zs[lane + 32 * k] = zr[lane + 32 * k];
        } else {
            const uint32_t* cw = reinterpret_cast<const uint32_t*>(a.codes + coff);
            const int nw = d * bits / 32, nb = d / blk;
            for (int w = lane; w < nw; w += 32) cwS[w] = cw[w];
            if (lane < nb) sm[lane] = a.scales[a.smap.at(l, s, b, h, t) + lane];
            __syncwarp();
#pragma unroll
            for (int k = 0; k < NR; k++) {
                const int c = lane + 32 * k;
                const uint32_t q = extract_code(cwS, c * bits, bits);
                const uint32_t sz = sm[c / blk];
                zs[c] = fmaf((float)q, h2f_bits(sz & 0xffffu), h2f_bits(sz >> 16));
            }
        }
        __syncwarp();
        uint16_t* orow = a.out + ((((int64_t)(l * 2 + s) * a.B + b) * a.H + h) * a.T_x + t) * d;
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k, r = c / g, i = c - r * g;
            const float acc = gauge_coord(Gs + r * g * g + i, g, zs + r * g, g);
            orow[c] = __bfloat16_as_ushort(__float2bfloat16_rn(acc));
        }
        __syncwarp();
    }
}

// ------------------------------------------------------------------------------------
// KIVI keys: per-channel ranges over a group of Gt tokens (one CTA per (l, b, h, group)).
// ------------------------------------------------------------------------------------
template <int NR>
__global__ void __launch_bounds__(kRowThreads) key_encode_kernel(KeyArgs a) {
    constexpr int d = NR * 32;
    extern __shared__ __align__(16) unsigned char smem[];
    const int g = a.g, Gt = a.Gt, bits = a.bits;
    const int pay = Gt * bits / 8;
    float* Gs = reinterpret_cast<float*>(smem);                          // transposed
    float* Zs = reinterpret_cast<float*>(smem + (size_t)d * g * 4);      // [Gt][d]
    float* xsAll = Zs + (size_t)Gt * d;                                  // [warps][d]
    uint8_t* stage = reinterpret_cast<uint8_t*>(xsAll + kRowWarps * d);  // [d][pay]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* xs = xsAll + warp * d;

    const int64_t tg = blockIdx.x;
    const int bh = blockIdx.y % (a.B * a.H), l = blockIdx.y / (a.B * a.H);
    const int b = bh / a.H, h = bh % a.H;
    const float* Gsrc = a.G + ((int64_t)(l * 2 + 0) * a.H + h) * (int64_t)d * g;
    for (int e = threadIdx.x; e < d * g; e += kRowThreads) {
        int r = e / (g * g), rem = e - r * g * g, i = rem / g, jj = rem - i * g;
        Gs[r * g * g + jj * g + i] = __ldg(Gsrc + e);
    }
    __syncthreads();
    int32_t flag = 0;
    const uint16_t* X = a.x + ((((int64_t)(l * 2 + 0) * a.B + b) * a.H + h) * a.T + tg * Gt) * d;
    for (int t = warp; t < Gt; t += kRowWarps) {
#pragma unroll
        for (int k = 0; k < NR; k++) {
            uint32_t xb = X[(int64_t)t * d + lane + 32 * k];
            if (bf16_nonfinite(xb)) flag |= CG_FLAG_NONFINITE_INPUT;
            xs[lane + 32 * k] = bf16_bits_to_float(xb);
        }
        __syncwarp();
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k, r = c / g, i = c - r * g;
            Zs[(size_t)t * d + c] = gauge_coord(Gs + r * g * g + i, g, xs + r * g, g);
        }
        __syncwarp();
    }
    __syncthreads();
    const int qmax = (1 << bits) - 1;
    const float qmaxf = (float)qmax;
    const int64_t bhl = (int64_t)b * a.H + h;
    for (int c = threadIdx.x; c < d; c += kRowThreads) {
        float mn = Zs[c], mx = Zs[c];
        for (int t = 1; t < Gt; t++) {
            const float v = Zs[(size_t)t * d + c];
            mn = fminf(mn, v);
            mx = fmaxf(mx, v);
        }
        const uint32_t sz = scale_zero(mn, mx, qmaxf, &flag);
        const float sc = h2f_bits(sz & 0xffffu), mz = h2f_bits(sz >> 16);
        uint8_t* st = stage + (size_t)c * pay;
        uint64_t acc = 0;
        int nacc = 0, nbytes = 0;
        for (int t = 0; t < Gt; t++) {
            acc |= (uint64_t)quant_code(Zs[(size_t)t * d + c], sc, mz, qmax) << nacc;
            nacc += bits;
            while (nacc >= 8) {
                st[nbytes++] = (uint8_t)(acc & 0xffu);
                acc >>= 8;
                nacc -= 8;
            }
        }
        a.scales[(int64_t)l * a.layer_scales + bhl * a.key_scales_per_bh + tg * d + c] = sz;
    }
    __syncthreads();
    uint32_t* dst = reinterpret_cast<uint32_t*>(a.codes + (int64_t)l * a.layer_codes + bhl * a.key_codes_per_bh +
                                                tg * (int64_t)d * pay);
    const uint32_t* src = reinterpret_cast<const uint32_t*>(stage);
    for (int w = threadIdx.x; w < d * pay / 4; w += kRowThreads) dst[w] = src[w];
    if (flag) raise_flag(a.status, flag);
}

template <int NR>
__global__ void __launch_bounds__(kRowThreads) key_decode_kernel(KeyArgs a) {
    constexpr int d = NR * 32;
    extern __shared__ __align__(16) unsigned char smem[];
    const int g = a.g, Gt = a.Gt, bits = a.bits;
    const int pay = Gt * bits / 8;
    float* Gs = reinterpret_cast<float*>(smem);                      // untransposed
    float* Zs = reinterpret_cast<float*>(smem + (size_t)d * g * 4);  // [Gt][d]
    uint8_t* stage = reinterpret_cast<uint8_t*>(Zs + (size_t)Gt * d);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int64_t tg = blockIdx.x;
    const int bh = blockIdx.y % (a.B * a.H), l = blockIdx.y / (a.B * a.H);
    const int b = bh / a.H, h = bh % a.H;
    const int64_t bhl = (int64_t)b * a.H + h;
    const float* Gsrc = a.G + ((int64_t)(l * 2 + 0) * a.H + h) * (int64_t)d * g;
    for (int e = threadIdx.x; e < d * g; e += kRowThreads) Gs[e] = __ldg(Gsrc + e);
    const uint32_t* src = reinterpret_cast<const uint32_t*>(a.codes + (int64_t)l * a.layer_codes +
                                                            bhl * a.key_codes_per_bh + tg * (int64_t)d * pay);
    uint32_t* stw = reinterpret_cast<uint32_t*>(stage);
    for (int w = threadIdx.x; w < d * pay / 4; w += kRowThreads) stw[w] = src[w];
    __syncthreads();
    for (int c = threadIdx.x; c < d; c += kRowThreads) {
        const uint32_t sz = a.scales[(int64_t)l * a.layer_scales + bhl * a.key_scales_per_bh + tg * d + c];
        const float sc = h2f_bits(sz & 0xffffu), mz = h2f_bits(sz >> 16);
        const uint8_t* st = stage + (size_t)c * pay;
        for (int t = 0; t < Gt; t++) {
            const int p = t * bits;
            uint32_t v = st[p >> 3] >> (p & 7);
            if ((p & 7) + bits > 8) v |= (uint32_t)st[(p >> 3) + 1] << (8 - (p & 7));
            v &= (1u << bits) - 1u;
            Zs[(size_t)t * d + c] = fmaf((float)v, sc, mz);
        }
    }
    __syncthreads();
    uint16_t* O = a.out + ((((int64_t)(l * 2 + 0) * a.B + b) * a.H + h) * a.T + tg * Gt) * d;
    for (int t = warp; t < Gt; t += kRowWarps) {
        const float* zr = Zs + (size_t)t * d;
#pragma unroll
        for (int k = 0; k < NR; k++) {
            const int c = lane + 32 * k, r = c / g, i = c - r * g;
            const float acc = gauge_coord(Gs + r * g * g + i, g, zr + r * g, g);
            O[(int64_t)t * d + c] = __bfloat16_as_ushort(__float2bfloat16_rn(acc));
        }
    }
}

__global__ void residual_copy_kernel(ResidArgs a) {
    const int64_t n16 = (a.T - a.nq) * a.d * 2 / 16;  // 16-byte chunks per unit
    for (int64_t u = blockIdx.y; u < a.units; u += gridDim.y) {
        const uint4* src;
        uint4* dst;
        if (a.to_residual) {
            src = reinterpret_cast<const uint4*>(a.src + (u * a.T + a.nq) * a.d);
            dst = reinterpret_cast<uint4*>(a.dst + u * (a.T - a.nq) * a.d);
        } else {
            src = reinterpret_cast<const uint4*>(a.src + u * (a.T - a.nq) * a.d);
            dst = reinterpret_cast<uint4*>(a.dst + (u * a.T + a.nq) * a.d);
        }
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n16; i += (int64_t)gridDim.x * blockDim.x)
            dst[i] = src[i];
    }
}

__global__ void __launch_bounds__(256) row_move_kernel(MoveArgs a) {
    const int64_t c16 = a.d / 8;  // 16-byte chunks per token row
    const int64_t rows = a.t_hi - a.t_lo;
    const int64_t n = a.units * rows * c16;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t u = i / (rows * c16), rem = i - u * rows * c16;
        const int64_t t = a.t_lo + rem / c16, c = rem % c16;
        const uint16_t* src = t < a.src_split ? a.ring_src + (u * a.W + t % a.W) * a.d
                                              : a.x + (u * a.T_x + (t - a.x_t0)) * a.d;
        uint16_t* dst = a.dst_ring ? a.dst + (u * a.W + t % a.W) * a.d : a.dst + (u * a.dst_T + (t - a.dst_t0)) * a.d;
        reinterpret_cast<uint4*>(dst)[c] = reinterpret_cast<const uint4*>(src)[c];
    }
}

}  // namespace

cudaError_t launch_row_move(const MoveArgs& a, cudaStream_t st) {
    const int64_t n = a.units * (a.t_hi - a.t_lo) * (a.d / 8);
    if (n <= 0) return cudaSuccess;
    int64_t blocks = (n + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    row_move_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

// Warps per CTA of the tile encode kernel: as many as shared memory holds, at most 16.
static int tile_simt_warps(int d, int g) {
    if (!(d == 32 || d == 64 || d == 128 || d == 256)) return 0;
    const size_t gbytes = (size_t)d * g * 4;
    if (gbytes >= kSmemOptIn) return 0;
    const size_t n = (kSmemOptIn - gbytes) / tile_warp_bytes(d);
    return n < (size_t)kTileWarpsMax ? (int)n : kTileWarpsMax;
}

size_t tile_simt_smem(int d, int g) {
    const int nw = tile_simt_warps(d, g);
    return nw < 1 ? 0 : (size_t)d * g * 4 + (size_t)nw * tile_warp_bytes(d);
}

size_t row_simt_smem(int d, int g) {
    if (!(d == 32 || d == 64 || d == 128 || d == 256)) return 0;
    size_t enc = (size_t)d * g * 4 + (size_t)kRowWarps * d * 5 + (size_t)kRowWarps * 32 * 4;
    size_t dec = (size_t)d * g * 4 + (size_t)kRowWarps * d * 4 + (size_t)kRowWarps * (d / 4 + 4) * 4 +
                 (size_t)kRowWarps * 32 * 4;
    return enc > dec ? enc : dec;
}

size_t key_simt_smem(int d, int g, int Gt, int bits) {
    if (!(d == 32 || d == 64 || d == 128 || d == 256)) return 0;
    size_t pay = (size_t)Gt * bits / 8;
    size_t enc = (size_t)d * g * 4 + (size_t)Gt * d * 4 + (size_t)kRowWarps * d * 4 + (size_t)d * pay;
    return enc;
}

template <int NR>
static cudaError_t row_encode_nr(const RowArgs& a, cudaStream_t st) {
    size_t smem = row_simt_smem(a.d, a.g);
    cudaError_t e = cudaFuncSetAttribute(row_encode_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((a.B * a.t_count + kRowsPerCta - 1) / kRowsPerCta), (unsigned)(a.L * a.s_n * a.H));
    row_encode_kernel<NR><<<grid, kRowThreads, smem, st>>>(a);
    return cudaGetLastError();
}

template <int NR>
static cudaError_t tile_encode_nr(const RowArgs& a, cudaStream_t st) {
    const int nwarps = tile_simt_warps(a.d, a.g);
    const size_t smem = tile_simt_smem(a.d, a.g);
    if (nwarps < 1) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(tile_encode_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    // two tiles per warp per CTA; the tiles of one (l, s, h) spread over grid.x
    const int64_t tiles = (int64_t)a.B * ((a.t_count + kTileTokens - 1) / kTileTokens);
    int64_t gx = (tiles + 2 * nwarps - 1) / (2 * nwarps);
    if (gx > 65535) gx = 65535;
    dim3 grid((unsigned)gx, (unsigned)(a.L * a.s_n * a.H));
    tile_encode_kernel<NR><<<grid, nwarps * 32, smem, st>>>(a);
    return cudaGetLastError();
}

template <int NR>
static cudaError_t row_decode_nr(const RowArgs& a, cudaStream_t st) {
    size_t smem = row_simt_smem(a.d, a.g);
    cudaError_t e = cudaFuncSetAttribute(row_decode_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)((a.B * a.t_count + kRowsPerCta - 1) / kRowsPerCta), (unsigned)(a.L * a.s_n * a.H));
    row_decode_kernel<NR><<<grid, kRowThreads, smem, st>>>(a);
    return cudaGetLastError();
}

template <int NR>
static cudaError_t key_encode_nr(const KeyArgs& a, cudaStream_t st) {
    size_t smem = key_simt_smem(a.d, a.g, a.Gt, a.bits);
    cudaError_t e = cudaFuncSetAttribute(key_encode_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)(a.nq / a.Gt), (unsigned)(a.L * a.B * a.H));
    key_encode_kernel<NR><<<grid, kRowThreads, smem, st>>>(a);
    return cudaGetLastError();
}

template <int NR>
static cudaError_t key_decode_nr(const KeyArgs& a, cudaStream_t st) {
    size_t smem = key_simt_smem(a.d, a.g, a.Gt, a.bits);
    cudaError_t e = cudaFuncSetAttribute(key_decode_kernel<NR>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)(a.nq / a.Gt), (unsigned)(a.L * a.B * a.H));
    key_decode_kernel<NR><<<grid, kRowThreads, smem, st>>>(a);
    return cudaGetLastError();
}

#define CG_NR_SWITCH(FN, d, ...)                      \
    switch ((d) / 32) {                               \
        case 1: return FN<1>(__VA_ARGS__);            \
        case 2: return FN<2>(__VA_ARGS__);            \
        case 4: return FN<4>(__VA_ARGS__);            \
        case 8: return FN<8>(__VA_ARGS__);            \
        default: return cudaErrorInvalidValue;        \
    }

cudaError_t launch_row_encode_simt(const RowArgs& a, cudaStream_t st) { CG_NR_SWITCH(row_encode_nr, a.d, a, st) }
cudaError_t launch_row_decode_simt(const RowArgs& a, cudaStream_t st) { CG_NR_SWITCH(row_decode_nr, a.d, a, st) }
cudaError_t launch_tile_encode_simt(const RowArgs& a, cudaStream_t st) { CG_NR_SWITCH(tile_encode_nr, a.d, a, st) }

template <int CPL>
static cudaError_t hadamard_nr(const RowArgs& a, bool enc, cudaStream_t st) {
    const int64_t units = (int64_t)a.L * a.s_n * a.B * a.H;
    if (units < 1 || a.t_count < 1) return cudaSuccess;
    // token ranges per unit: about 8 rows per warp, at most 65535 ranges
    int64_t gy = (a.t_count + 8 * kRowWarps - 1) / (8 * kRowWarps);
    if (gy > 65535) gy = 65535;
    const dim3 grid((unsigned)units, (unsigned)gy);
    const float c = (float)(1.0 / sqrt((double)a.g));
    if (enc)
        hadamard_encode_kernel<CPL><<<grid, kRowThreads, 0, st>>>(a, c);
    else
        hadamard_decode_kernel<CPL><<<grid, kRowThreads, 0, st>>>(a, c);
    return cudaGetLastError();
}

cudaError_t launch_hadamard(const RowArgs& a, bool encode, cudaStream_t st) {
    switch (a.d / 32) {
        case 1: return hadamard_nr<1>(a, encode, st);
        case 2: return hadamard_nr<2>(a, encode, st);
        case 4: return hadamard_nr<4>(a, encode, st);
        case 8: return hadamard_nr<8>(a, encode, st);
        default: return cudaErrorInvalidValue;
    }
}
cudaError_t launch_key_encode_simt(const KeyArgs& a, cudaStream_t st) { CG_NR_SWITCH(key_encode_nr, a.d, a, st) }
cudaError_t launch_key_decode_simt(const KeyArgs& a, cudaStream_t st) { CG_NR_SWITCH(key_decode_nr, a.d, a, st) }

cudaError_t launch_residual_copy(const ResidArgs& a, cudaStream_t st) {
    const int64_t n16 = (a.T - a.nq) * a.d * 2 / 16;
    if (n16 <= 0 || a.units <= 0) return cudaSuccess;
    unsigned gx = (unsigned)((n16 + 255) / 256);
    if (gx > 1024) gx = 1024;
    dim3 grid(gx, (unsigned)(a.units < 65535 ? a.units : 65535));
    residual_copy_kernel<<<grid, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace cg
