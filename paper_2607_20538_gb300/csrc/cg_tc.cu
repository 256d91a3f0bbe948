// cg_tc.cu -- tensor-core (tcgen05) kernels of the row path, head dim d = 128.
//
// Encode (Sec. 3: Z = G X, then the block-uniform backend of Sec. 4.3) as one persistent,
// warp-specialized kernel per launch:
//   warp 0      TMA producer: 128-token x tiles (2 x [128 rows x 64 bf16], 128-byte swizzle)
//               into a ring of kStages shared-memory stages;
//   warp 1      MMA issuer: z~ = x G^T on tcgen05 (M = 128 tokens, N = K = gauge group, one
//               MMA chain per group block), with G split into npass bf16 terms (hi + lo
//               [+ lo2]) so that z~ is within a few fp32 ulps of the exact product; fp32
//               accumulators in tensor memory, double buffered;
//   warps 2..5  epilogue, one thread per token row (= TMEM lane): block min/max, fp16
//               scale/zero, codes, bit packing, stores.
// Exactness: the library defines z as a fixed-order fp32 sum (16-wide fma chains; see
// include/codecgauge.h). z~ differs from it by at most E = ||x_group||_2 * e_i, with e_i
// built per gauge row from the rounding bound of that order, the measured error model of
// the tensor-core accumulation and the exact residual of the bf16 split. The epilogue
// decides the fp16 scale/zero from the interval [z~ - E, z~ + E] when every value in it
// rounds to the same fp16 result; otherwise it recomputes the candidate extremes exactly.
// Codes whose pre-rounding value lies within E/s of a rounding boundary are recomputed
// exactly too. Recomputation uses the same fixed-order sum as the CUDA-core kernels,
// spread over the lanes of a warp through a small shared-memory job queue.
#include <cuda_bf16.h>

#include <cstdio>
#include <mutex>

#include "cg_sm100.cuh"
#include "cg_tc.h"
#include "cg_tmap.h"

namespace cg {
namespace {

using namespace sm100;

constexpr int kD = 128;                 // head dimension handled here
constexpr int kStages = 4;              // x tile ring
constexpr int kTileBytes = 128 * kD * 2;
constexpr int kThreads = 192;
constexpr int kQCap = 96;               // repair jobs per warp and round
constexpr uint64_t kWaitLimitNs = 4000000000ull;
constexpr float kU = 5.9604645e-08f;    // 2^-24

struct EncSmem {
    // byte offsets from the 1024-aligned base
    static constexpr uint32_t stages = 0;
    static constexpr uint32_t bsplit = stages + kStages * kTileBytes;  // npass x (16 or 32 KB)
    static constexpr uint32_t bsplit_max = 3 * 16384 > 2 * 32768 ? 3 * 16384 : 2 * 32768;
    static constexpr uint32_t codes_stage = bsplit + bsplit_max;       // 128 rows x (4*BITS+4) words
    static constexpr uint32_t codes_stage_max = 128 * (4 * 8 + 4) * 4;
    static constexpr uint32_t queue = codes_stage + codes_stage_max;   // 4 warps x kQCap x 8 B
    static constexpr uint32_t misc = queue + 4 * kQCap * 8;
    static constexpr uint32_t total = misc + 1024;
};

struct Misc {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint64_t g_ready;
    uint32_t tmem_slot;
    int abort_flag;
    int qcount[4];
    float emax[2][4][16];  // [conversion parity][epilogue warp][gauge group]: max_i e_i
};

struct EncParams {
    RowArgs a;
    int npass;
    int64_t n_units, tiles_per_unit, n_tiles;
};

__device__ __forceinline__ float bf_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf_hi(uint32_t w) { return __uint_as_float(w & 0xffff0000u); }

// unit index (b fastest, then h, s, l) -> (l, s, b, h); tiles of a unit are contiguous
__device__ __forceinline__ void unit_coords(const RowArgs& a, int64_t u, int& l, int& s, int& b, int& h) {
    b = (int)(u % a.B);
    int64_t r = u / a.B;
    h = (int)(r % a.H);
    r /= a.H;
    s = a.s_lo + (int)(r % a.s_n);
    l = (int)(r / a.s_n);
}

// Exact gauge-space value of (row, col) in the library's fixed order, x read from the
// swizzled stage tile and G from global memory (fp32, row `col` of the head's gauge set).
__device__ __noinline__ float exact_z(const unsigned char* stage, int row, int col, const float* Gf, int g) {
    const int r0 = (col / g) * g;
    const float* Grow = Gf + (size_t)col * g;
    const int nb = g >= 16 ? g / 16 : 1;
    const int w = g >= 16 ? 16 : g;
    float p[8];
#pragma unroll
    for (int b = 0; b < 8; b++) p[b] = 0.0f;
    for (int h8 = 0; h8 < w; h8 += 8) {
#pragma unroll
        for (int b = 0; b < 8; b++) {
            if (b < nb) {
                const int k = r0 + 16 * b + h8;
                const uint4 xv = *reinterpret_cast<const uint4*>(stage + (k >> 6) * 16384 + row * 128 +
                                                                 ((((k & 63) >> 3) ^ (row & 7)) << 4));
                const float4 g0 = __ldg(reinterpret_cast<const float4*>(Grow + 16 * b + h8));
                const float4 g1 = __ldg(reinterpret_cast<const float4*>(Grow + 16 * b + h8 + 4));
                float q = p[b];
                q = fmaf(g0.x, bf_lo(xv.x), q);
                q = fmaf(g0.y, bf_hi(xv.x), q);
                q = fmaf(g0.z, bf_lo(xv.y), q);
                q = fmaf(g0.w, bf_hi(xv.y), q);
                q = fmaf(g1.x, bf_lo(xv.z), q);
                q = fmaf(g1.y, bf_hi(xv.z), q);
                q = fmaf(g1.z, bf_lo(xv.w), q);
                q = fmaf(g1.w, bf_hi(xv.w), q);
                p[b] = q;
            }
        }
    }
    float acc = p[0];
#pragma unroll
    for (int b = 1; b < 8; b++)
        if (b < nb) acc = __fadd_rn(acc, p[b]);
    return acc;
}

// fp16 scale of a block with the given (max, min) in fp32, by the library's rule.
__device__ __forceinline__ uint32_t scale16(float mx, float mn, float qmax) {
    return f2h_bits(__fdiv_rn(__fsub_rn(mx, mn), qmax));
}

template <int BITS>
__global__ void __launch_bounds__(kThreads, 1) tc_encode_kernel(const __grid_constant__ CUtensorMap xmap,
                                                                 const EncParams P) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t base_u32 = (smem_u32(smem_raw) + 1023u) & ~1023u;
    unsigned char* sm = smem_raw + (base_u32 - smem_u32(smem_raw));
    Misc* M = reinterpret_cast<Misc*>(sm + EncSmem::misc);
    unsigned char* stages = sm + EncSmem::stages;
    unsigned char* bsplit = sm + EncSmem::bsplit;
    uint32_t* cstage = reinterpret_cast<uint32_t*>(sm + EncSmem::codes_stage);
    uint32_t* queue = reinterpret_cast<uint32_t*>(sm + EncSmem::queue);

    const RowArgs& a = P.a;
    const int g = a.g, blk = a.blk, npass = P.npass;
    const int gb = g < 16 ? 16 : g;
    const uint32_t bsz = (g == 128) ? 32768u : 16384u;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    // contiguous tile range of this CTA
    const int64_t t_begin = P.n_tiles * blockIdx.x / gridDim.x;
    const int64_t t_end = P.n_tiles * (blockIdx.x + 1) / gridDim.x;
    const int my_tiles = (int)(t_end - t_begin);

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&M->full[i], 1);
            mbar_init(&M->empty[i], 4);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&M->acc_full[i], 1);
            mbar_init(&M->acc_empty[i], 4);
        }
        mbar_init(&M->g_ready, 4);
        M->abort_flag = 0;
        for (int i = 0; i < 4; i++) M->qcount[i] = 0;
        fence_barrier_init();
    }
    // zero the B operand area once: off-diagonal gauge blocks stay zero
    for (uint32_t i = threadIdx.x; i < (uint32_t)npass * bsz / 16; i += kThreads)
        reinterpret_cast<uint4*>(bsplit)[i] = make_uint4(0, 0, 0, 0);
    if (warp == 1) {
        tmem_alloc(&M->tmem_slot, 256);
        tmem_relinquish();
        tc_fence_before();
    }
    fence_proxy_async_smem();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = M->tmem_slot;
    volatile int* abort_flag = &M->abort_flag;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0 && my_tiles > 0) {
            prefetch_tmap(&xmap);
            int issued = 0;
            for (int i = 0; i < my_tiles; i++) {
                const int st = i % kStages;
                if (!mbar_wait(&M->empty[st], ((i / kStages) & 1) ^ 1, abort_flag, kWaitLimitNs)) {
                    *abort_flag = 1;
                    break;
                }
                const int64_t tile = t_begin + i;
                const int64_t u = tile / P.tiles_per_unit;
                const int64_t t0 = (tile - u * P.tiles_per_unit) * 128;
                int l, s, b, h;
                unit_coords(a, u, l, s, b, h);
                const int64_t row0 = (((int64_t)(l * 2 + s) * a.B + b) * a.H + h) * a.T_x + t0;
                unsigned char* dst = stages + st * kTileBytes;
                mbar_arrive_expect_tx(&M->full[st], kTileBytes);
                tma_load_2d(dst, &xmap, &M->full[st], 0, (int)row0);
                tma_load_2d(dst + 16384, &xmap, &M->full[st], 64, (int)row0);
                issued = i + 1;
            }
            if (*abort_flag) {
                // let every load this thread issued land before the CTA can exit
                const int from = issued > kStages ? issued - kStages : 0;
                const int zero = 0;
                for (int i = from; i < issued; i++)
                    mbar_wait(&M->full[i % kStages], (i / kStages) & 1, &zero, kWaitLimitNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && my_tiles > 0) {
            const uint32_t idesc = idesc_bf16_f32(128, gb);
            int64_t cur_gid = -1;
            int g_phase = 0;
            int committed = 0;
            for (int i = 0; i < my_tiles; i++) {
                const int64_t tile = t_begin + i;
                const int64_t u = tile / P.tiles_per_unit;
                int l, s, b, h;
                unit_coords(a, u, l, s, b, h);
                const int64_t gid = (int64_t)(l * 2 + s) * a.H + h;
                bool ok = true;
                if (gid != cur_gid) {
                    ok = mbar_wait(&M->g_ready, g_phase, abort_flag, kWaitLimitNs);
                    g_phase ^= 1;
                    cur_gid = gid;
                }
                const int st = i % kStages, buf = i & 1;
                ok = ok && mbar_wait(&M->full[st], (i / kStages) & 1, abort_flag, kWaitLimitNs);
                ok = ok && mbar_wait(&M->acc_empty[buf], ((i >> 1) & 1) ^ 1, abort_flag, kWaitLimitNs);
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t a_base = smem_u32(stages + st * kTileBytes);
                const uint32_t d_base = tmem + buf * 128;
                for (int p = 0; p < npass; p++) {
                    const uint32_t b_base = smem_u32(bsplit) + p * bsz;
                    for (int r = 0; r < 128 / gb; r++) {
                        for (int ks = 0; ks < gb / 16; ks++) {
                            const int k0 = r * gb + ks * 16;
                            const uint32_t a_addr = a_base + (k0 >> 6) * 16384 + (k0 & 63) * 2;
                            const uint32_t b_addr =
                                b_base + (g == 128 ? (k0 >> 6) * 16384 : 0) + (r * gb) * 128 + (k0 & 63) * 2;
                            mma_bf16(d_base + r * gb, sdesc_sw128(a_addr), sdesc_sw128(b_addr), idesc,
                                     (p > 0 || ks > 0) ? 1u : 0u);
                        }
                    }
                }
                mma_commit(&M->acc_full[buf]);
                committed = i + 1;
            }
            if (*abort_flag && committed > 0) {
                const int zero = 0;
                const int i = committed - 1;
                mbar_wait(&M->acc_full[i & 1], (i >> 1) & 1, &zero, kWaitLimitNs);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int ew = warp & 3;              // TMEM lane quadrant of this warp
        const int row = ew * 32 + lane;       // tile row = TMEM lane
        const int etid = (warp - 2) * 32 + lane;  // B row this thread converts
        const int qw = warp - 2;
        uint32_t* qjob = queue + qw * kQCap * 2;       // (row | col << 8), result bits
        const int R = kD / g;
        const int nbk = kD / blk;
        const float qmaxf = (float)((1 << BITS) - 1);
        const int qmax = (1 << BITS) - 1;
        constexpr int kWords = 4 * BITS;               // packed words per row (128 codes)
        constexpr int kStride = kWords + 4;
        uint32_t* my_codes = cstage + row * kStride;
        // error coefficients of the fixed-order sum and of the tensor-core accumulation
        const int n_order = (g < 16 ? g : 16) + (g >= 16 ? g / 16 : 1) - 1;
        const float c_chain = (float)n_order * kU * 1.01f;
        const float c_tc = 2.0f * (float)(npass * (gb / 16) + 2) * kU;
        int32_t flag = 0;
        int64_t cur_gid = -1;
        int conv = 0;  // gauge conversions done by this warp
        const float* Gf = nullptr;
        bool ok = true;

        for (int i = 0; i < my_tiles && ok; i++) {
            const int64_t tile = t_begin + i;
            const int64_t u = tile / P.tiles_per_unit;
            const int64_t t0 = (tile - u * P.tiles_per_unit) * 128;
            int l, s, b, h;
            unit_coords(a, u, l, s, b, h);
            const int64_t gid = (int64_t)(l * 2 + s) * a.H + h;
            if (gid != cur_gid) {
                // ---- convert the gauge set of (l, s, h) into the bf16 split operand
                Gf = a.G + gid * (int64_t)kD * g;
                const int n = etid;  // B row = output channel
                const int r = n / g;
                const float* Gr = Gf + (size_t)n * g;
                float s_g2 = 0.0f, s_res2 = 0.0f;
                for (int j = 0; j < g; j += 8) {
                    const int k = r * g + j;
                    const float4 v0 = __ldg(reinterpret_cast<const float4*>(Gr + j));
                    const float4 v1 = __ldg(reinterpret_cast<const float4*>(Gr + j + 4));
                    const float v[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
                    // term t = 0 is the leading bf16 part; pass p uses term npass - 1 - p
                    uint32_t term[3][4];
#pragma unroll
                    for (int e = 0; e < 8; e += 2) {
                        float rest0 = v[e], rest1 = v[e + 1];
                        s_g2 = fmaf(v[e], v[e], s_g2);
                        s_g2 = fmaf(v[e + 1], v[e + 1], s_g2);
#pragma unroll
                        for (int t = 0; t < 3; t++) {
                            if (t < npass) {
                                const __nv_bfloat16 h0 = __float2bfloat16_rn(rest0);
                                const __nv_bfloat16 h1 = __float2bfloat16_rn(rest1);
                                rest0 = __fsub_rn(rest0, __bfloat162float(h0));
                                rest1 = __fsub_rn(rest1, __bfloat162float(h1));
                                term[t][e >> 1] = (uint32_t)__bfloat16_as_ushort(h0) |
                                                  ((uint32_t)__bfloat16_as_ushort(h1) << 16);
                            }
                        }
                        s_res2 = fmaf(rest0, rest0, s_res2);
                        s_res2 = fmaf(rest1, rest1, s_res2);
                    }
#pragma unroll
                    for (int t = 0; t < 3; t++) {
                        if (t < npass) {
                            const int pp = npass - 1 - t;
                            unsigned char* region = bsplit + pp * bsz + (g == 128 ? (k >> 6) * 16384 : 0);
                            *reinterpret_cast<uint4*>(region + sw128_offset(n, k & 63)) =
                                make_uint4(term[t][0], term[t][1], term[t][2], term[t][3]);
                        }
                    }
                }
                // e_n bounds |z~ - z| / ||x_group||_2 for this output channel; each warp keeps
                // the maximum over the rows of each group it covers
                float e_n = ((c_chain + c_tc) * sqrtf(s_g2) + sqrtf(s_res2)) * 1.001f + 1e-30f;
                const int seg = g < 32 ? g : 32;
                for (int off = seg >> 1; off >= 1; off >>= 1) e_n = fmaxf(e_n, __shfl_xor_sync(0xffffffffu, e_n, off));
                if ((lane & (seg - 1)) == 0) M->emax[conv & 1][qw][r] = e_n;
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&M->g_ready);
                // every epilogue warp's part (B operand and bounds) is written once the phase completes
                const bool g_ok = mbar_wait(&M->g_ready, conv & 1, abort_flag, kWaitLimitNs);
                if (!__all_sync(0xffffffffu, g_ok)) {
                    *abort_flag = 1;
                    ok = false;
                    break;
                }
                cur_gid = gid;
                conv++;
            }
            const int st = i % kStages, buf = i & 1;
            // accumulator ready; the stage's TMA data is acquired through its own barrier
            // (already complete: this warp releases the stage only after the tile)
            bool w_ok = mbar_wait(&M->acc_full[buf], (i >> 1) & 1, abort_flag, kWaitLimitNs);
            w_ok = w_ok && mbar_wait(&M->full[st], (i / kStages) & 1, abort_flag, kWaitLimitNs);
            if (!__all_sync(0xffffffffu, w_ok)) {
                *abort_flag = 1;
                ok = false;
                break;
            }
            tc_fence_after();
            const unsigned char* stg = stages + st * kTileBytes;
            const int rows_valid = (int)((a.t_count - t0) < 128 ? (a.t_count - t0) : 128);
            const bool valid = row < rows_valid;
            const uint32_t tacc = tmem + ((uint32_t)(ew * 32) << 16) + buf * 128;

            // ---- 1. per-group norms of x from the stage (bf16 exact -> fp32)
            float nrm2[16];
#pragma unroll
            for (int r = 0; r < 16; r++) nrm2[r] = 0.0f;
            bool nonfinite = false;
#pragma unroll
            for (int c = 0; c < 16; c++) {
                const uint4 xv = *reinterpret_cast<const uint4*>(stg + (c >> 3) * 16384 + row * 128 +
                                                                 (((c & 7) ^ (row & 7)) << 4));
                const uint32_t wv[4] = {xv.x, xv.y, xv.z, xv.w};
                float acc = 0.0f;
#pragma unroll
                for (int q = 0; q < 4; q++) {
                    const float lo = bf_lo(wv[q]), hi = bf_hi(wv[q]);
                    acc = fmaf(lo, lo, acc);
                    acc = fmaf(hi, hi, acc);
                    nonfinite |= ((wv[q] >> 7) & 0xffu) == 0xffu || ((wv[q] >> 23) & 0xffu) == 0xffu;
                }
                // chunk c holds channels 8c..8c+7, inside group (8c)/g
#pragma unroll
                for (int r = 0; r < 16; r++)
                    if (r == (8 * c) / g) nrm2[r] += acc;
            }
            if (valid && nonfinite) flag |= CG_FLAG_NONFINITE_INPUT;

            // ---- 2. approximate block ranges and their error bound
            float mnv[4], mxv[4], Eb[4];
#pragma unroll
            for (int bk = 0; bk < 4; bk++) {
                mnv[bk] = INFINITY;
                mxv[bk] = -INFINITY;
                Eb[bk] = 0.0f;
            }
#pragma unroll
            for (int c = 0; c < 4; c++) {
                uint32_t v[32];
                tmem_ld32(tacc + c * 32, v);
                tmem_wait_ld();
                const int bk = (c * 32) / blk;
                float lo = __uint_as_float(v[0]), hi = lo;
#pragma unroll
                for (int k = 1; k < 32; k++) {
                    lo = fminf(lo, __uint_as_float(v[k]));
                    hi = fmaxf(hi, __uint_as_float(v[k]));
                }
#pragma unroll
                for (int q = 0; q < 4; q++)
                    if (q == bk) {
                        mnv[q] = fminf(mnv[q], lo);
                        mxv[q] = fmaxf(mxv[q], hi);
                    }
            }
            // E per block: max over the gauge groups it overlaps (group bound = ||x_r|| * max_w emax)
            {
                const float (*em)[16] = M->emax[(conv - 1) & 1];
#pragma unroll
                for (int r = 0; r < 16; r++) {
                    if (r < R) {
                        float e = 0.0f;
                        // warps whose 32 rows intersect group r
                        const int w0 = (r * g) >> 5, w1 = ((r + 1) * g - 1) >> 5;
                        for (int w = w0; w <= w1; w++) e = fmaxf(e, em[w][r]);
                        const float er = sqrtf(nrm2[r]) * 1.0001f * e;
#pragma unroll
                        for (int bk = 0; bk < 4; bk++)
                            if (bk < nbk && r * g < (bk + 1) * blk && (r + 1) * g > bk * blk) Eb[bk] = fmaxf(Eb[bk], er);
                    }
                }
#pragma unroll
                for (int bk = 0; bk < 4; bk++) Eb[bk] += (fabsf(mnv[bk]) + fabsf(mxv[bk])) * 2.4e-7f;
            }

            // ---- 3. decide scale/zero from the intervals; flag ambiguous blocks
            uint32_t s16[4], m16[4];
            int amb = 0;  // bit 2*bk: scale ambiguous, bit 2*bk+1: zero ambiguous
#pragma unroll
            for (int bk = 0; bk < 4; bk++) {
                s16[bk] = m16[bk] = 0;
                if (bk < nbk) {
                    const float E = Eb[bk];
                    const float mn_lo = __fsub_rn(mnv[bk], E), mn_hi = __fadd_rn(mnv[bk], E);
                    const float mx_lo = __fsub_rn(mxv[bk], E), mx_hi = __fadd_rn(mxv[bk], E);
                    const float dlo = fmaxf(__fsub_rn(mx_lo, mn_hi), 0.0f);
                    const uint32_t slo = f2h_bits(__fdiv_rn(dlo, qmaxf));
                    const uint32_t shi = scale16(mx_hi, mn_lo, qmaxf);
                    const uint32_t mlo = f2h_bits(mn_lo), mhi = f2h_bits(mn_hi);
                    s16[bk] = slo;
                    m16[bk] = mlo;
                    if (valid && slo != shi) amb |= 1 << (2 * bk);
                    if (valid && mlo != mhi) amb |= 2 << (2 * bk);
                }
            }
            // ---- 4. exact recompute of the candidate extremes of ambiguous blocks
            float ex_mn[4], ex_mx[4];
#pragma unroll
            for (int bk = 0; bk < 4; bk++) {
                ex_mn[bk] = INFINITY;
                ex_mx[bk] = -INFINITY;
            }
            int myslot[8], mytag[8];
            int nmine = 0;
            if (__any_sync(0xffffffffu, amb != 0)) {
                if (lane == 0) M->qcount[qw] = 0;
                __syncwarp();
#pragma unroll
                for (int c = 0; c < 4; c++) {
                    const int bk = (c * 32) / blk;
                    const int need = (amb >> (2 * bk)) & 3;  // any side ambiguous -> need min; scale -> max too
                    if (!__any_sync(0xffffffffu, need != 0)) continue;
                    uint32_t v[32];
                    tmem_ld32(tacc + c * 32, v);
                    tmem_wait_ld();
                    if (need) {
                        float E = 0.0f, mnb = 0.0f, mxb = 0.0f;
#pragma unroll
                        for (int q = 0; q < 4; q++)
                            if (q == bk) {
                                E = Eb[q];
                                mnb = mnv[q];
                                mxb = mxv[q];
                            }
                        const float thr_lo = __fadd_rn(mnb, 2.0f * E), thr_hi = __fsub_rn(mxb, 2.0f * E);
                        uint32_t mmin = 0, mmax = 0;
#pragma unroll
                        for (int k = 0; k < 32; k++) {
                            const float z = __uint_as_float(v[k]);
                            if (z <= thr_lo) mmin |= 1u << k;
                            if ((need & 1) && z >= thr_hi) mmax |= 1u << k;
                        }
                        uint32_t mall = mmin | mmax;
                        while (mall) {
                            const int k = __ffs(mall) - 1;
                            mall &= mall - 1;
                            const bool cmin = (mmin >> k) & 1, cmax = (mmax >> k) & 1;
                            const int col = c * 32 + k;
                            const int slot = atomicAdd(&M->qcount[qw], 1);
                            const int tag = bk | (cmin ? 4 : 0) | (cmax ? 8 : 0);
                            if (slot < kQCap) qjob[2 * slot] = (uint32_t)row | ((uint32_t)col << 8);
                            if (slot < kQCap && nmine < 8) {
                                myslot[nmine] = slot;
                                mytag[nmine] = tag;
                                nmine++;
                            } else {
                                // no room to track the job: recompute in place
                                const float ze = exact_z(stg, row, col, Gf, g);
#pragma unroll
                                for (int q = 0; q < 4; q++)
                                    if (q == bk) {
                                        if (cmin) ex_mn[q] = fminf(ex_mn[q], ze);
                                        if (cmax) ex_mx[q] = fmaxf(ex_mx[q], ze);
                                    }
                            }
                        }
                    }
                }
                __syncwarp();
                const int nq = min(M->qcount[qw], kQCap);
                for (int j = lane; j < nq; j += 32) {
                    const uint32_t jb = qjob[2 * j];
                    qjob[2 * j + 1] = __float_as_uint(exact_z(stg, (int)(jb & 0xffu), (int)(jb >> 8), Gf, g));
                }
                __syncwarp();
                for (int m = 0; m < nmine; m++) {
                    const float ze = __uint_as_float(qjob[2 * myslot[m] + 1]);
                    const int tag = mytag[m];
#pragma unroll
                    for (int q = 0; q < 4; q++)
                        if (q == (tag & 3)) {
                            if (tag & 4) ex_mn[q] = fminf(ex_mn[q], ze);
                            if (tag & 8) ex_mx[q] = fmaxf(ex_mx[q], ze);
                        }
                }
                __syncwarp();
#pragma unroll
                for (int bk = 0; bk < 4; bk++) {
                    const int need = (amb >> (2 * bk)) & 3;
                    if (need) {
                        m16[bk] = f2h_bits(ex_mn[bk]);
                        if (need & 1) s16[bk] = scale16(ex_mx[bk], ex_mn[bk], qmaxf);
                    }
                }
            }
#pragma unroll
            for (int bk = 0; bk < 4; bk++)
                if (bk < nbk && valid && (h_is_inf(s16[bk]) || h_is_inf(m16[bk]))) flag |= CG_FLAG_FP16_OVERFLOW;

            // ---- 5. codes (fast path) with boundary check, packed into the row stage
            if (lane == 0) M->qcount[qw] = 0;
            __syncwarp();
            nmine = 0;
#pragma unroll
            for (int c = 0; c < 4; c++) {
                uint32_t v[32];
                tmem_ld32(tacc + c * 32, v);
                tmem_wait_ld();
                const int bk = (c * 32) / blk;
                float sc = 0.0f, mz = 0.0f, E = 0.0f;
                uint32_t s16b = 0;
#pragma unroll
                for (int q = 0; q < 4; q++)
                    if (q == bk) {
                        s16b = s16[q];
                        mz = h2f_bits(m16[q]);
                        E = Eb[q];
                    }
                sc = h2f_bits(s16b);
                const bool zero_scale = (sc == 0.0f);
                const float rinv = zero_scale ? 0.0f : __frcp_rn(sc);
                const float mu = zero_scale ? 0.0f : E * rinv * 1.0001f + (qmaxf + 1.0f) * 4.8e-7f;
                const float lim = 0.5f - mu;
                uint32_t words[BITS];
#pragma unroll
                for (int w = 0; w < BITS; w++) words[w] = 0;
                uint32_t ambmask = 0;
#pragma unroll
                for (int k = 0; k < 32; k++) {
                    const float z = __uint_as_float(v[k]);
                    float t = __fmul_rn(__fsub_rn(z, mz), rinv);
                    t = fminf(fmaxf(t, 0.0f), qmaxf);
                    const float rt = rintf(t);
                    const uint32_t q = zero_scale ? 0u : (uint32_t)(int)rt;
                    if (fabsf(t - rt) > lim && !zero_scale) ambmask |= 1u << k;
                    const int bit = k * BITS;
                    words[bit >> 5] |= q << (bit & 31);
                    if ((bit & 31) + BITS > 32) words[(bit >> 5) + 1] |= q >> (32 - (bit & 31));
                }
#pragma unroll
                for (int w = 0; w < BITS; w++) my_codes[c * BITS + w] = words[w];
                if (!valid) ambmask = 0;
                while (ambmask) {
                    const int k = __ffs(ambmask) - 1;
                    ambmask &= ambmask - 1;
                    const int col = c * 32 + k;
                    const int slot = atomicAdd(&M->qcount[qw], 1);
                    if (slot < kQCap) qjob[2 * slot] = (uint32_t)row | ((uint32_t)col << 8);
                    if (slot < kQCap && nmine < 8) {
                        myslot[nmine] = slot;
                        mytag[nmine] = col | ((int)s16b << 8);
                        nmine++;
                    } else {
                        const float ze = exact_z(stg, row, col, Gf, g);
                        const uint32_t q = quant_code(ze, sc, mz, qmax);
                        const int bit = col * BITS;
                        uint32_t* wp = my_codes + (bit >> 5);
                        const uint32_t msk = (uint32_t)qmax;
                        wp[0] = (wp[0] & ~(msk << (bit & 31))) | (q << (bit & 31));
                        if ((bit & 31) + BITS > 32) {
                            const int sh = 32 - (bit & 31);
                            wp[1] = (wp[1] & ~(msk >> sh)) | (q >> sh);
                        }
                    }
                }
            }
            if (__any_sync(0xffffffffu, nmine > 0)) {
                __syncwarp();
                const int nq = min(M->qcount[qw], kQCap);
                for (int j = lane; j < nq; j += 32) {
                    const uint32_t jb = qjob[2 * j];
                    qjob[2 * j + 1] = __float_as_uint(exact_z(stg, (int)(jb & 0xffu), (int)(jb >> 8), Gf, g));
                }
                __syncwarp();
                for (int m = 0; m < nmine; m++) {
                    const float ze = __uint_as_float(qjob[2 * myslot[m] + 1]);
                    const int col = mytag[m] & 0xff;
                    const uint32_t s16b = (uint32_t)mytag[m] >> 8;
                    const int bk = col / blk;
                    float mz = 0.0f;
#pragma unroll
                    for (int q = 0; q < 4; q++)
                        if (q == bk) mz = h2f_bits(m16[q]);
                    const uint32_t q = quant_code(ze, h2f_bits(s16b), mz, qmax);
                    const int bit = col * BITS;
                    uint32_t* wp = my_codes + (bit >> 5);
                    const uint32_t msk = (uint32_t)qmax;
                    wp[0] = (wp[0] & ~(msk << (bit & 31))) | (q << (bit & 31));
                    if ((bit & 31) + BITS > 32) {
                        const int sh = 32 - (bit & 31);
                        wp[1] = (wp[1] & ~(msk >> sh)) | (q >> sh);
                    }
                }
            }
            __syncwarp();

            // ---- 6. stores
            if (valid) {
                const int64_t t = t0 + row;
                uint4* dstc = reinterpret_cast<uint4*>(a.codes + a.cmap.at(l, s, b, h, t));
#pragma unroll
                for (int w = 0; w < kWords / 4; w++)
                    dstc[w] = make_uint4(my_codes[4 * w], my_codes[4 * w + 1], my_codes[4 * w + 2], my_codes[4 * w + 3]);
                uint32_t* dsts = a.scales + a.smap.at(l, s, b, h, t);
#pragma unroll
                for (int bk = 0; bk < 4; bk++)
                    if (bk < nbk) dsts[bk] = s16[bk] | (m16[bk] << 16);
            }
            // ---- 7. release the accumulator buffer and the stage
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&M->acc_empty[buf]);
                mbar_arrive(&M->empty[st]);
            }
        }
        if (flag) raise_flag(a.status, flag);
    }
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) raise_flag(a.status, CG_FLAG_PIPE_TIMEOUT);
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

int num_sms() {
    static int n[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) return 148;
    if (!n[dev]) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        n[dev] = v > 0 ? v : 148;
    }
    return n[dev];
}

template <int BITS>
cudaError_t launch_encode_bits(const EncParams& P, const CUtensorMap& map, cudaStream_t st) {
    const size_t smem = EncSmem::total + 1024;
    cudaError_t e = cudaFuncSetAttribute(tc_encode_kernel<BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = P.n_tiles < num_sms() ? P.n_tiles : num_sms();
    tc_encode_kernel<BITS><<<(unsigned)grid, kThreads, smem, st>>>(map, P);
    return cudaGetLastError();
}

}  // namespace

bool tc_row_encode_eligible(const RowArgs& a) {
    if (a.d != kD || a.none_mode) return false;
    if (!(a.blk == 32 || a.blk == 64 || a.blk == 128)) return false;
    if (a.t_count < 64) return false;
    const int64_t rows = (int64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (rows + 128 >= (int64_t)1 << 31) return false;
    if (reinterpret_cast<uintptr_t>(a.x) & 15u) return false;
    return tmap_encode_fn() != nullptr;
}

cudaError_t tc_launch_row_encode(const RowArgs& a, cudaStream_t st) {
    EncParams P;
    P.a = a;
    P.npass = a.g == 128 ? 2 : 3;
    P.n_units = (int64_t)a.L * a.s_n * a.B * a.H;
    P.tiles_per_unit = (a.t_count + 127) / 128;
    P.n_tiles = P.n_units * P.tiles_per_unit;
    if (P.n_tiles == 0) return cudaSuccess;
    CUtensorMap map;
    const uint64_t rows = (uint64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (!make_tmap_bf16_sw128(&map, a.x, rows, kD, kD * 2, 128)) return cudaErrorInvalidValue;
    switch (a.bits) {
        case 2: return launch_encode_bits<2>(P, map, st);
        case 3: return launch_encode_bits<3>(P, map, st);
        case 4: return launch_encode_bits<4>(P, map, st);
        case 6: return launch_encode_bits<6>(P, map, st);
        case 8: return launch_encode_bits<8>(P, map, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace cg
