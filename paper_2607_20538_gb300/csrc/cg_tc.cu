// cg_tc.cu -- tensor-core (tcgen05) encode of the row path, head dim d = 128: gauge
// rotation (Sec. 3, Z = G X) fused with the block-uniform quantizer of Sec. 4.3 (one range
// per block of `block` channels of a token), also used for KIVI value rows.
//
// Persistent warp-specialized kernel, one CTA per SM, 15 warps:
//   warp 0      TMA producer: 128-token x tiles (2 x [128 rows x 64 bf16], 128-byte
//               swizzle) into a 4-stage ring;
//   warp 1      MMA issuer: z~ = x G^T on tcgen05 (M = 128 tokens, N = K = gauge group,
//               one MMA chain per group block), G split into three bf16 terms (hi + lo +
//               lo2, exact for normal fp32 values); fp32 accumulators in tensor memory,
//               four buffers (the MMA runs one tile ahead of the three warpgroups);
//   warp 2      gauge converter: at each gauge change builds the bf16 split operand and
//               the per-block error coefficients of the new gauge set;
//   warps 3..14 three epilogue warpgroups; warpgroup k takes tiles i = k (mod 3); one
//               thread per token row (= TMEM lane): block min/max, fp16 scale/zero, codes,
//               packing, stores. The number of quantization blocks per row is a template
//               parameter, so the per-block state of a row takes only the registers it
//               needs (128 per thread for 15 warps); codes are packed into the output
//               words as they are produced.
//
// Exactness. The library defines z as a fixed-order fp32 sum (pairwise summation of the
// products; include/codecgauge.h). For every output channel i the converter bounds
// |z~_i - z_i| / ||x_group||_2 by
//     e_i = (c_order + c_tc) ||G_i||_2 + ||G_i - sum of split terms||_2,
// c_order = (1 + log2 g) u the rounding bound of the fixed order, c_tc a bound on the
// tensor-core fp32 accumulation, and the exact residual of the split. The MMAs accumulate
// the split's two small terms first (partial sums below 2^-8 of ||G_i|| ||x||, 2 n_hi
// K-steps) and the leading term last (n_hi = K / 16 steps), so c_tc = (n_hi + 4 + 2 n_hi /
// 128) u, 4 u covering the rounding inside each MMA and of the result; the measured
// |z~ - Gx| stays below 2.4 u ||G_i|| ||x|| (g = 32 and 128; random, Hadamard and DCT gauges). The epilogue
// turns it into E per block. A block's fp16 scale and zero are monotone functions of its
// (max, min); when every (max, min) within E of the approximate ones gives the same fp16
// results they are taken directly, otherwise the candidate extremes are recomputed
// exactly, so scales and zeros are bit-identical to the definition.
// Codes: a code taken from z~ can differ from the definition's only if the exact
// pre-rounding value t lies within mu = E/s (+ rounding slack) of a rounding boundary.
// The accepted tolerance lets a code differ by one where t lies within 1e-4 steps of a
// boundary, so blocks with mu < 1e-4 keep the z~ codes; in blocks with a larger mu the
// codes within mu of a boundary are recomputed exactly. Recomputation uses the library's
// order (as the CUDA-core kernels do): candidates go into a per-warp shared-memory job
// queue and teams of lanes compute them together.
#include <cuda_bf16.h>

#include "cg_sm100.cuh"
#include "cg_tc.h"
#include "cg_tc_common.cuh"
#include "cg_tc_enc.cuh"
#include "cg_tmap.h"

namespace cg {
namespace {

using namespace sm100;
using tc::kD;
using tc::kWaitLimitNs;

constexpr int kStages = 4;
constexpr int kTileBytes = 128 * kD * 2;
constexpr int kThreads = 480;
constexpr int kEpiWarp0 = 3;
constexpr int kQCap = 20;             // repair jobs per warp and round
constexpr int kAcc = 4;               // accumulator buffers in tensor memory
constexpr int kNPass = 3;             // bf16 terms of the gauge split
constexpr int kSegBufs = 4;
constexpr float kMagic = 12582912.0f; // 1.5 * 2^23: adding it rounds to an integer (RNE)

struct EncSmem {
    static constexpr uint32_t stages = 0;
    static constexpr uint32_t bsplit = stages + kStages * kTileBytes;  // 3 x (16 or 32 KB)
    static constexpr uint32_t queue = bsplit + kNPass * 32768;         // 12 warps x kQCap x 8 B
    static constexpr uint32_t xch = queue + 12 * kQCap * 8;  // keys: 3 warpgroups x 2 x 4 warps x 4 floats
    static constexpr uint32_t misc = xch + 3 * 2 * 4 * 4 * 4;
    static constexpr uint32_t total = misc + 384;  // base is 1024-aligned (checked in-kernel)
};

struct Misc {
    uint64_t full[kStages], empty[kStages];
    uint64_t accfull[kAcc], accempty[kAcc];
    uint64_t gready[kSegBufs];
    uint64_t bfree;
    uint32_t tmem_slot;
    int abort_flag;
    float emaxb[kSegBufs][4];  // per gauge set and quantization block: max_i e_i
    float gmaxb[kSegBufs][4];  // and max_i ||G_i||
    uint64_t xbar[3][2];       // keys: per warpgroup, exchange of the group-norm maxima
};

static_assert(sizeof(Misc) <= 384, "Misc outgrew its shared-memory slot");
static_assert(EncSmem::total <= 232448, "encode kernel exceeds 227 KB of shared memory");

struct EncParams {
    RowArgs a;
    tc::Sched S;
};

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

template <typename T>
__device__ __forceinline__ T pick4(const T (&v)[4], int i) {
    return i == 0 ? v[0] : i == 1 ? v[1] : i == 2 ? v[2] : v[3];
}
template <typename T>
__device__ __forceinline__ void set4(T (&v)[4], int i, T x) {
    v[0] = i == 0 ? x : v[0];
    v[1] = i == 1 ? x : v[1];
    v[2] = i == 2 ? x : v[2];
    v[3] = i == 3 ? x : v[3];
}

// Rows of the gauge channels whose error bounds block bk's values: the whole gauge group
// when the group spans the block, else the block's own channels.
__device__ __forceinline__ void bound_range(int bk, int g, int blk, int& lo, int& hi) {
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
// arithmetic, so one memory round trip serves kSlots x (32 / T) values.
template <int kSlots>
__device__ __noinline__ void run_jobs(uint32_t* qjob, int nq, const unsigned char* stage, const float* Gf, int g,
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
            gv[k] = __ldg(reinterpret_cast<const float4*>(Gf + (size_t)col * g + 4 * j));
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

// KEYS = false: block-uniform rows and KIVI value rows (thread = token, block = channels).
// KEYS = true: KIVI keys (Sec. 4.3, per-channel ranges over a 128-token group): the MMA
// operands are swapped, D[channel][token] = G x^T, so a thread owns one channel's 128
// tokens, which form its block and its packed code stream.
template <int BITS, bool KEYS, int NBK>
__global__ void __launch_bounds__(kThreads, 1) tc_encode_kernel(const __grid_constant__ CUtensorMap xmap,
                                                                 const EncParams P) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    if (smem_u32(smem_raw) & 1023u) {
        // the swizzled tiles need a 1024-byte aligned base; the layout leaves no slack
        if (threadIdx.x == 0) raise_flag(P.a.status, CG_FLAG_PIPE_TIMEOUT);
        return;
    }
    unsigned char* sm = smem_raw;
    Misc* M = reinterpret_cast<Misc*>(sm + EncSmem::misc);
    unsigned char* stages = sm + EncSmem::stages;
    unsigned char* bsplit = sm + EncSmem::bsplit;
    uint32_t* queue = reinterpret_cast<uint32_t*>(sm + EncSmem::queue);
    float* xch = reinterpret_cast<float*>(sm + EncSmem::xch);

    const RowArgs& a = P.a;
    const tc::Sched& S = P.S;
    const int g = a.g, npass = kNPass;
    constexpr int blk = kD / NBK;  // quantization block: NBK blocks per row
    const int gb = g < 16 ? 16 : g;
    constexpr int nbk = NBK;
    // values per lane and memory round trip in the exact recompute (measured: 4 with two
    // blocks per row, the 8B-shaped cache; 2 with one or four)
    constexpr int kJobSlots = NBK == 2 ? 4 : 2;
    // gauge operand layout: full K = 128 (block-diagonal for g < 128) for keys and g = 128,
    // else one g-wide K block per group in a 64-column tile
    const bool fullk = KEYS || g == 128;
    const uint32_t bsz = fullk ? 32768u : 16384u;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int64_t t_begin = S.n_tiles * blockIdx.x / gridDim.x;
    const int64_t t_end = S.n_tiles * (blockIdx.x + 1) / gridDim.x;
    const int my_tiles = (int)(t_end - t_begin);
    const int64_t seg0 = my_tiles > 0 ? tc::tile_info(a, S, t_begin).seg : 0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kStages; i++) {
            mbar_init(&M->full[i], 1);
            mbar_init(&M->empty[i], 4);
        }
        for (int i = 0; i < kAcc; i++) {
            mbar_init(&M->accfull[i], 1);
            mbar_init(&M->accempty[i], 4);
        }
        for (int i = 0; i < kSegBufs; i++) mbar_init(&M->gready[i], 1);
        for (int w = 0; w < 3; w++) {
            mbar_init(&M->xbar[w][0], 4);
            mbar_init(&M->xbar[w][1], 4);
        }
        mbar_init(&M->bfree, 1);
        M->abort_flag = 0;
        fence_barrier_init();
    }
    for (uint32_t i = threadIdx.x; i < (uint32_t)npass * bsz / 16; i += kThreads)
        reinterpret_cast<uint4*>(bsplit)[i] = make_uint4(0, 0, 0, 0);
    if (warp == 1) {
        tmem_alloc(&M->tmem_slot, kAcc * 128);
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
            tc::TileIter it;
            it.init(a, S, t_begin);
            for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
                const int st = i % kStages;
                if (!mbar_wait(&M->empty[st], ((i / kStages) & 1) ^ 1, abort_flag, a.wait_ns)) {
                    *abort_flag = 1;
                    break;
                }
                const tc::TileInfo ti = it.info(a);
                const int64_t row0 = tc::dense_row(a, ti);
                unsigned char* dst = stages + st * kTileBytes;
                mbar_arrive_expect_tx(&M->full[st], kTileBytes);
                tma_load_2d(dst, &xmap, &M->full[st], 0, (int)row0);
                tma_load_2d(dst + 16384, &xmap, &M->full[st], 64, (int)row0);
                issued = i + 1;
            }
            if (*abort_flag) {
                const int zero = 0;
                const int from = issued > kStages ? issued - kStages : 0;
                for (int i = from; i < issued; i++)
                    mbar_wait(&M->full[i % kStages], (i / kStages) & 1, &zero, kWaitLimitNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && my_tiles > 0) {
            const uint32_t idesc = idesc_bf16_f32(128, KEYS ? 128 : gb);
            const int kg = KEYS ? 128 : gb;  // keys: one chain over the full K
            int64_t cur = -1;
            int committed = 0;
            tc::TileIter it;
            it.init(a, S, t_begin);
            for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
                const tc::TileInfo ti = it.info(a);
                const int64_t ls = ti.seg - seg0;
                bool ok = true;
                if (ti.seg != cur) {
                    ok = mbar_wait(&M->gready[ls & 3], (ls >> 2) & 1, abort_flag, a.wait_ns);
                    cur = ti.seg;
                }
                const int st = i % kStages, buf = i % kAcc;
                ok = ok && mbar_wait(&M->full[st], (i / kStages) & 1, abort_flag, a.wait_ns);
                ok = ok && mbar_wait(&M->accempty[buf], ((i / kAcc) & 1) ^ 1, abort_flag, a.wait_ns);
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
                tc_fence_after();
                const uint32_t a_base = smem_u32(stages + st * kTileBytes);
                const uint32_t d_base = tmem + buf * 128;
                for (int p = 0; p < npass; p++) {
                    const uint32_t b_base = smem_u32(bsplit) + p * bsz;
                    for (int r = 0; r < 128 / kg; r++) {
                        for (int ks = 0; ks < kg / 16; ks++) {
                            const int k0 = r * kg + ks * 16;
                            const uint32_t a_addr = a_base + (k0 >> 6) * 16384 + (k0 & 63) * 2;
                            const uint32_t b_addr = b_base + (fullk ? (k0 >> 6) * 16384 : 0) +
                                                    (KEYS ? 0 : (r * gb) * 128) + (k0 & 63) * 2;
                            if (KEYS)  // D[channel][token] = G x^T
                                mma_bf16(d_base, sdesc_sw128(b_addr), sdesc_sw128(a_addr), idesc,
                                         (p > 0 || ks > 0) ? 1u : 0u);
                            else  // D[token][channel] = x G^T, one chain per gauge group
                                mma_bf16(d_base + r * gb, sdesc_sw128(a_addr), sdesc_sw128(b_addr), idesc,
                                         (p > 0 || ks > 0) ? 1u : 0u);
                        }
                    }
                }
                mma_commit(&M->accfull[buf]);
                const bool last_of_seg = (i + 1 == my_tiles) || it.seg_last(a);
                if (last_of_seg) mma_commit(&M->bfree);
                committed = i + 1;
            }
            if (*abort_flag && committed > 0) {
                const int zero = 0;
                const int i = committed - 1;
                mbar_wait(&M->accfull[i % kAcc], (i / kAcc) & 1, &zero, kWaitLimitNs);
            }
        }
    } else if (warp == 2) {
        // ------------------------------------------------------------ gauge converter
        int64_t cur = -1;
        int nconv = 0;
        tc::TileIter it;
        it.init(a, S, t_begin);
        for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
            const tc::TileInfo ti = it.info(a);
            if (ti.seg == cur) continue;
            const int64_t ls = ti.seg - seg0;
            if (nconv > 0) {
                const bool ok = mbar_wait(&M->bfree, (nconv - 1) & 1, abort_flag, a.wait_ns);
                if (!__all_sync(0xffffffffu, ok)) {
                    *abort_flag = 1;
                    break;
                }
            }
            const float* Gf = a.G + tc::gauge_set(a, ti) * (int64_t)kD * g;
            tce::prefetch_next_gauges(a, ti, g, lane);
            tce::convert_gauge_set<KEYS, 4>(Gf, g, blk, nbk, fullk, bsz, bsplit, M->emaxb[ls & 3], M->gmaxb[ls & 3], 0, lane);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&M->gready[ls & 3]);
            cur = ti.seg;
            nconv++;
        }
    } else {
        // ------------------------------------------------------------ epilogue warpgroups
        const int wg = (warp - kEpiWarp0) >> 2;       // warpgroup: tiles i = wg (mod 3)
        const int q4 = warp & 3;                      // TMEM lane quadrant of this warp
        const int row = q4 * 32 + lane;               // TMEM lane: token (rows) or channel (keys)
        const int qw = warp - kEpiWarp0;              // job queue of this warp
        uint32_t* qjob = queue + qw * kQCap * 2;
        const float qmaxf = (float)((1 << BITS) - 1);
        const int qmax = (1 << BITS) - 1;
        int lo8[4], hi8[4];
#pragma unroll
        for (int bk = 0; bk < 4; bk++) {
            int lo = 0, hi = 0;
            if (bk < nbk) bound_range(bk, g, blk, lo, hi);
            lo8[bk] = lo >> 3;
            hi8[bk] = hi >> 3;
        }
        int32_t flag = 0;
        tc::TileIter it;
        it.init(a, S, t_begin + wg);
        for (int i = wg; i < my_tiles; i += 3, it.step(a, 3)) {
            const tc::TileInfo ti = it.info(a);
            const int64_t ls = ti.seg - seg0;
            const int st = i % kStages, buf = i % kAcc;
            bool ok = mbar_wait(&M->accfull[buf], (i / kAcc) & 1, abort_flag, a.wait_ns);
            ok = ok && mbar_wait(&M->full[st], (i / kStages) & 1, abort_flag, a.wait_ns);
            ok = ok && mbar_wait(&M->gready[ls & 3], (ls >> 2) & 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            const unsigned char* stg = stages + st * kTileBytes;
            const bool valid = KEYS || row < ti.rows_valid;  // key tiles are whole token groups
            const uint32_t tacc = tmem + ((uint32_t)(q4 * 32) << 16) + buf * 128;
            const float* Gf = a.G + tc::gauge_set(a, ti) * (int64_t)kD * g;

            // ---- 1. ||x||^2 over the bound range of every block (bf16 -> fp32 exact)
            float bs[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            if (KEYS) {
                // a key block is one channel over the tile's 128 tokens: its bound uses the
                // largest group norm among those tokens. Each warp takes its own 32 token rows
                // (one per lane); the four warps of the warpgroup then exchange their per-group
                // maxima in shared memory (two buffers, alternating by tile)
                float gs[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll 4
                for (int c8 = 0; c8 < 16; c8++) {
                    const uint4 xv = *reinterpret_cast<const uint4*>(stg + (c8 >> 3) * 16384 + row * 128 +
                                                                     (((c8 & 7) ^ (row & 7)) << 4));
                    float s0 = bf_lo(xv.x) * bf_lo(xv.x);
                    s0 = fmaf(bf_hi(xv.x), bf_hi(xv.x), s0);
                    s0 = fmaf(bf_lo(xv.y), bf_lo(xv.y), s0);
                    s0 = fmaf(bf_hi(xv.y), bf_hi(xv.y), s0);
                    s0 = fmaf(bf_lo(xv.z), bf_lo(xv.z), s0);
                    s0 = fmaf(bf_hi(xv.z), bf_hi(xv.z), s0);
                    s0 = fmaf(bf_lo(xv.w), bf_lo(xv.w), s0);
                    s0 = fmaf(bf_hi(xv.w), bf_hi(xv.w), s0);
                    const int r = (c8 * 8) / g;  // g >= 32: at most 4 groups
#pragma unroll
                    for (int rr = 0; rr < 4; rr++)
                        if (rr == r) gs[rr] += s0;
                }
                if (!(isfinite(gs[0]) && isfinite(gs[1]) && isfinite(gs[2]) && isfinite(gs[3]))) {
                    for (int c8 = 0; c8 < 16; c8++) {
                        const uint4 xv = *reinterpret_cast<const uint4*>(stg + (c8 >> 3) * 16384 + row * 128 +
                                                                         (((c8 & 7) ^ (row & 7)) << 4));
                        const uint32_t wv[4] = {xv.x, xv.y, xv.z, xv.w};
                        for (int k = 0; k < 4; k++)
                            if (bf16_nonfinite(wv[k] & 0xffffu) || bf16_nonfinite(wv[k] >> 16))
                                flag |= CG_FLAG_NONFINITE_INPUT;
                    }
                }
#pragma unroll
                for (int rr = 0; rr < 4; rr++)
                    for (int off = 16; off >= 1; off >>= 1)
                        gs[rr] = fmaxf(gs[rr], __shfl_xor_sync(0xffffffffu, gs[rr], off));
                const int kx = (i - wg) / 3;  // this warpgroup's tile count
                float* xb = xch + (wg * 2 + (kx & 1)) * 16;
                if (lane == 0) {
#pragma unroll
                    for (int rr = 0; rr < 4; rr++) xb[q4 * 4 + rr] = gs[rr];
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&M->xbar[wg][kx & 1]);
                const bool okx = mbar_wait(&M->xbar[wg][kx & 1], (kx >> 1) & 1, abort_flag, a.wait_ns);
                if (!__all_sync(0xffffffffu, okx)) {
                    *abort_flag = 1;
                    break;
                }
                float gm[4];
#pragma unroll
                for (int rr = 0; rr < 4; rr++)
                    gm[rr] = fmaxf(fmaxf(xb[rr], xb[4 + rr]), fmaxf(xb[8 + rr], xb[12 + rr]));
                bs[0] = pick4(gm, row / g);  // fmaxf keeps a NaN out; non-finite input is flagged above
            }
            // unroll depth measured per block count (code size against load parallelism)
            constexpr int kNormUnroll = NBK == 2 ? 8 : (NBK == 4 ? 2 : 4);
#pragma unroll kNormUnroll
            for (int c8 = 0; c8 < (KEYS ? 0 : 16); c8++) {
                const uint4 xv = *reinterpret_cast<const uint4*>(stg + (c8 >> 3) * 16384 + row * 128 +
                                                                 (((c8 & 7) ^ (row & 7)) << 4));
                float s0 = bf_lo(xv.x) * bf_lo(xv.x);
                s0 = fmaf(bf_hi(xv.x), bf_hi(xv.x), s0);
                s0 = fmaf(bf_lo(xv.y), bf_lo(xv.y), s0);
                s0 = fmaf(bf_hi(xv.y), bf_hi(xv.y), s0);
                s0 = fmaf(bf_lo(xv.z), bf_lo(xv.z), s0);
                s0 = fmaf(bf_hi(xv.z), bf_hi(xv.z), s0);
                s0 = fmaf(bf_lo(xv.w), bf_lo(xv.w), s0);
                s0 = fmaf(bf_hi(xv.w), bf_hi(xv.w), s0);
#pragma unroll
                for (int bk = 0; bk < 4; bk++)
                    if (c8 >= lo8[bk] && c8 < hi8[bk]) bs[bk] += s0;
            }
            if (!KEYS && valid && !(isfinite(bs[0]) && isfinite(bs[1]) && isfinite(bs[2]) && isfinite(bs[3]))) {
                // a non-finite sum of squares: look for an Inf/NaN input (huge finite values
                // can also overflow the square)
                for (int c8 = 0; c8 < 16; c8++) {
                    const uint4 xv = *reinterpret_cast<const uint4*>(stg + (c8 >> 3) * 16384 + row * 128 +
                                                                     (((c8 & 7) ^ (row & 7)) << 4));
                    const uint32_t wv[4] = {xv.x, xv.y, xv.z, xv.w};
                    for (int q = 0; q < 4; q++)
                        if (bf16_nonfinite(wv[q] & 0xffffu) || bf16_nonfinite(wv[q] >> 16)) flag |= CG_FLAG_NONFINITE_INPUT;
                }
            }

            // ---- 2. approximate block ranges from the accumulator. With two blocks per row the
            // candidate masks are built here for every chunk (measured faster there): the values
            // within 2 Ep of the chunk's own min / max, Ep >= E (item 3) being known before the
            // ranges are. Otherwise they are built in the exact-extreme round, only where needed.
            constexpr bool kEagerMasks = NBK == 2;
            float mn[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
            float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            float clo[4], chi[4];           // chunk min / max (eager masks)
            uint32_t pm[4], px[4];          // chunk candidate masks (bit k = column 32c + k)
#pragma unroll 1
            for (int c = 0; c < 4; c++) {
                uint32_t v[32];
                tmem_ld32(tacc + c * 32, v);
                tmem_wait_ld();
                float lo = __uint_as_float(v[0]), hi = lo;
#pragma unroll
                for (int k = 1; k < 31; k += 2) {
                    lo = min3f(lo, __uint_as_float(v[k]), __uint_as_float(v[k + 1]));
                    hi = max3f(hi, __uint_as_float(v[k]), __uint_as_float(v[k + 1]));
                }
                lo = fminf(lo, __uint_as_float(v[31]));
                hi = fmaxf(hi, __uint_as_float(v[31]));
                const int bk = (c * 32) / blk;
                set4(mn, bk, fminf(pick4(mn, bk), lo));
                set4(mx, bk, fmaxf(pick4(mx, bk), hi));
                if constexpr (!kEagerMasks) continue;
                // |z~| <= ||G_i|| ||x|| + E, so Ep bounds the E of item 3 from above
                const float xn = sqrtf(pick4(bs, bk)) * 1.0001f;
                const float ep = xn * M->emaxb[ls & 3][bk] + 2.0f * xn * M->gmaxb[ls & 3][bk] * 2.41e-7f;
                const float tl = __fadd_rn(lo, 2.0f * ep), th = __fsub_rn(hi, 2.0f * ep);
                // sign bits of (threshold - z) and (z - threshold), shifted in from column 31 down
                uint32_t a0 = 0, a1 = 0;
#pragma unroll
                for (int k = 31; k >= 0; k--) {
                    const float z = __uint_as_float(v[k]);
                    a0 = __funnelshift_l(__float_as_uint(__fsub_rn(tl, z)), a0, 1);
                    a1 = __funnelshift_l(__float_as_uint(__fsub_rn(z, th)), a1, 1);
                }
                set4(clo, c, lo);
                set4(chi, c, hi);
                set4(pm, c, ~a0);  // z <= tl
                set4(px, c, ~a1);  // z >= th
            }

            // ---- 3. error bound per block; scale/zero from the intervals when they agree
            float E[4];
            uint32_t s16[4], m16[4];
            int amb = 0;  // bit 2bk: scale needs the exact extremes; bit 2bk+1: zero needs the exact min
#pragma unroll
            for (int bk = 0; bk < 4; bk++) {
                E[bk] = 0.0f;
                s16[bk] = m16[bk] = 0;
                if (bk < nbk) {
                    E[bk] = sqrtf(bs[bk]) * 1.0001f * M->emaxb[ls & 3][bk] + (fabsf(mn[bk]) + fabsf(mx[bk])) * 2.4e-7f;
                    const float e = E[bk];
                    const float mn_lo = __fsub_rn(mn[bk], e), mn_hi = __fadd_rn(mn[bk], e);
                    const float mx_lo = __fsub_rn(mx[bk], e), mx_hi = __fadd_rn(mx[bk], e);
                    const uint32_t slo = f2h_bits(__fdiv_rn(fmaxf(__fsub_rn(mx_lo, mn_hi), 0.0f), qmaxf));
                    const uint32_t shi = scale16(mx_hi, mn_lo, qmaxf);
                    const uint32_t mlo = f2h_bits(mn_lo), mhi = f2h_bits(mn_hi);
                    s16[bk] = slo;
                    m16[bk] = mlo;
                    if (valid && slo != shi) amb |= 1 << (2 * bk);
                    if (valid && mlo != mhi) amb |= 2 << (2 * bk);
                }
            }

            // ---- 4. exact extremes of ambiguous blocks (warp-cooperative rounds)
            if (__any_sync(0xffffffffu, amb != 0)) {
                if constexpr (kEagerMasks) {
                    // candidates: a chunk's values near its own min (max) are candidates of the
                    // block min (max) when the chunk min lies within 2E of the block min
#pragma unroll 1
                    for (int c = 0; c < 4; c++) {
                        const int bk = (c * 32) / blk;
                        const int need = (amb >> (2 * bk)) & 3;
                        const float e2 = 2.0f * pick4(E, bk);
                        const bool nl = need && pick4(clo, c) <= __fadd_rn(pick4(mn, bk), e2);
                        const bool nh = (need & 1) && pick4(chi, c) >= __fsub_rn(pick4(mx, bk), e2);
                        set4(pm, c, nl ? pick4(pm, c) : 0u);
                        set4(px, c, nh ? pick4(px, c) : 0u);
                    }
                } else {
                    // candidates of an ambiguous block's min (max): its values within 2E of the
                    // approximate min (max); the chunks some lane needs are reloaded from TMEM
#pragma unroll 1
                    for (int c = 0; c < 4; c++) {
                        const int bk = (c * 32) / blk;
                        const int need = (amb >> (2 * bk)) & 3;
                        uint32_t m0 = 0, m1 = 0;
                        if (__any_sync(0xffffffffu, need != 0)) {
                            uint32_t v[32];
                            tmem_ld32(tacc + c * 32, v);
                            tmem_wait_ld();
                            const float e2 = 2.0f * pick4(E, bk);
                            const float tl = __fadd_rn(pick4(mn, bk), e2), th = __fsub_rn(pick4(mx, bk), e2);
                            uint32_t a0 = 0, a1 = 0;
#pragma unroll
                            for (int k = 31; k >= 0; k--) {
                                const float z = __uint_as_float(v[k]);
                                a0 = __funnelshift_l(__float_as_uint(__fsub_rn(tl, z)), a0, 1);
                                a1 = __funnelshift_l(__float_as_uint(__fsub_rn(z, th)), a1, 1);
                            }
                            m0 = need ? ~a0 : 0u;        // z <= tl
                            m1 = (need & 1) ? ~a1 : 0u;  // z >= th
                        }
                        set4(pm, c, m0);
                        set4(px, c, m1);
                    }
                }
                float ex_mn[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
                float ex_mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                bool pend = (pm[0] | pm[1] | pm[2] | pm[3] | px[0] | px[1] | px[2] | px[3]) != 0;
                while (__any_sync(0xffffffffu, pend)) {
                    // every lane's candidates take consecutive slots (warp prefix sum of the
                    // counts); one cooperative round serves up to kQCap of them
                    const int cnt = __popc(pm[0] | px[0]) + __popc(pm[1] | px[1]) + __popc(pm[2] | px[2]) +
                                    __popc(pm[3] | px[3]);
                    int inc = cnt;
#pragma unroll
                    for (int off = 1; off < 32; off <<= 1) {
                        const int t = __shfl_up_sync(0xffffffffu, inc, off);
                        if (lane >= off) inc += t;
                    }
                    const int base = inc - cnt;
                    const int total = __shfl_sync(0xffffffffu, inc, 31);
                    int slot = base;
#pragma unroll 1
                    for (int c = 0; c < 4 && slot < kQCap; c++) {
                        uint32_t m = pick4(pm, c) | pick4(px, c);
                        while (m && slot < kQCap) {
                            const uint32_t col = (uint32_t)(c * 32 + __ffs(m) - 1);
                            qjob[2 * slot] = KEYS ? col | ((uint32_t)row << 8) : (uint32_t)row | (col << 8);
                            m &= m - 1;
                            slot++;
                        }
                    }
                    __syncwarp();
                    run_jobs<kJobSlots>(qjob, min(total, kQCap), stg, Gf, g, lane);
                    __syncwarp();
                    // the same candidates in the same order: fold the exact values in
                    slot = base;
#pragma unroll 1
                    for (int c = 0; c < 4 && slot < kQCap; c++) {
                        uint32_t cm = pick4(pm, c), cx = pick4(px, c);
                        uint32_t m = cm | cx;
                        const int bk = (c * 32) / blk;
                        float emn = pick4(ex_mn, bk), emx = pick4(ex_mx, bk);
                        while (m && slot < kQCap) {
                            const uint32_t bit = m & (0u - m);
                            const float ze = __uint_as_float(qjob[2 * slot + 1]);
                            if (cm & bit) emn = fminf(emn, ze);
                            if (cx & bit) emx = fmaxf(emx, ze);
                            cm &= ~bit;
                            cx &= ~bit;
                            m &= m - 1;
                            slot++;
                        }
                        set4(ex_mn, bk, emn);
                        set4(ex_mx, bk, emx);
                        set4(pm, c, cm);
                        set4(px, c, cx);
                    }
                    __syncwarp();
                    pend = (pm[0] | pm[1] | pm[2] | pm[3] | px[0] | px[1] | px[2] | px[3]) != 0;
                }
#pragma unroll
                for (int bk = 0; bk < 4; bk++) {
                    const int need = (amb >> (2 * bk)) & 3;
                    if (need) {
                        m16[bk] = f2h_bits(ex_mn[bk]);
                        if (need & 1) s16[bk] = scale16(ex_mx[bk], ex_mn[bk], qmaxf);
                    }
                }
            }

            // ---- 5. code parameters per block
            float rinv[4], c0[4], lim[4];
            int fast = 0;  // bit bk: no value of the block can leave [0, qmax]
            int live = 0;  // bit bk: finite, non-zero scale (else every code is 0)
#pragma unroll
            for (int bk = 0; bk < 4; bk++) {
                rinv[bk] = c0[bk] = 0.0f;
                lim[bk] = 0.5f;
                if (bk < nbk) {
                    if (valid && (h_is_inf(s16[bk]) || h_is_inf(m16[bk]))) flag |= CG_FLAG_FP16_OVERFLOW;
                    const float sc = h2f_bits(s16[bk]), mz = h2f_bits(m16[bk]);
                    if (sc != 0.0f && !h_is_inf(s16[bk]) && !h_is_inf(m16[bk])) {
                        const float r = __frcp_rn(sc);
                        const float cc = -mz * r;
                        rinv[bk] = r;
                        c0[bk] = cc;
                        // |t~ - t| <= E/s plus roundings: the fma and its inputs r and c0 (u|z r|,
                        // 2u|c0|, u|t|) and the definition's subtract and divide (2u|t|)
                        const float zr = fmaxf(fabsf(mn[bk]), fabsf(mx[bk])) * r;
                        const float mu = E[bk] * r * 1.0001f + (zr + 2.0f * fabsf(cc) + 3.0f * (qmaxf + 1.0f)) * 6.6e-8f;
                        // mu < 1e-4: a code from z~ can only differ where the tolerance allows it
                        lim[bk] = mu < 0.99e-4f ? 2.0f : 0.5f - mu;
                        const float tlo = (mn[bk] - E[bk]) * r + cc, thi = (mx[bk] + E[bk]) * r + cc;
                        if (tlo > -0.49f + mu && thi < qmaxf + 0.49f - mu) fast |= 1 << bk;
                        live |= 1 << bk;
                    }
                }
            }

            // ---- 6. codes from z~, stored straight from registers; near-boundary values repaired
            // rows: the token's codes; keys: the channel's 128-token stream (16 * BITS bytes)
            uint8_t* crow = KEYS ? a.codes + a.cmap.at(ti.l, ti.s, ti.b, ti.h, ti.t0) + (size_t)row * (16 * BITS)
                                 : a.codes + a.cmap.at(ti.l, ti.s, ti.b, ti.h, ti.t0 + row);
            uint32_t am[4] = {0, 0, 0, 0};  // values within mu of a rounding boundary
#pragma unroll 1
            for (int c = 0; c < 4; c++) {
                uint32_t v[32];
                tmem_ld32(tacc + c * 32, v);
                tmem_wait_ld();
                const int bk = (c * 32) / blk;
                const float r = pick4(rinv, bk), cc = pick4(c0, bk), lm = pick4(lim, bk);
                const bool fst = (fast >> bk) & 1;
                const bool lv = (live >> bk) & 1;
                uint32_t words[BITS];
#pragma unroll
                for (int w = 0; w < BITS; w++) words[w] = 0;
                // code k into the packed little-endian stream of this 32-code chunk
                // y = kMagic + q has the bit pattern 0x4B400000 + q. Widths that straddle words
                // (3, 6 bits) measure faster with a wrapping sum of y << s per word, less the
                // constant sum of 0x4B400000 << s; the others mask and OR the codes in.
                constexpr bool kBiasPack = BITS == 3 || BITS == 6;
                auto put = [&](int k, uint32_t y) {
                    const int bit = k * BITS;
                    if constexpr (kBiasPack) {
                        words[bit >> 5] += y << (bit & 31);
                        if ((bit & 31) + BITS > 32) words[(bit >> 5) + 1] += (y & (uint32_t)qmax) >> (32 - (bit & 31));
                    } else {
                        const uint32_t q = y & (uint32_t)qmax;
                        words[bit >> 5] |= q << (bit & 31);
                        if ((bit & 31) + BITS > 32) words[(bit >> 5) + 1] |= q >> (32 - (bit & 31));
                    }
                };
                uint32_t mk = 0;  // values within mu of a rounding boundary (bit k: column 32c + k)
                if (fst && lm > 1.0f) {
#pragma unroll
                    for (int k = 0; k < 32; k++) put(k, __float_as_uint(fmaf(__uint_as_float(v[k]), r, cc) + kMagic));
                } else {
                    // clamping before the rounding gives the same code as clamping after it
#pragma unroll
                    for (int k = 31; k >= 0; k--) {
                        float t = fmaf(__uint_as_float(v[k]), r, cc);
                        t = fminf(fmaxf(t, 0.0f), qmaxf);
                        const float y = t + kMagic;
                        mk = __funnelshift_l(__float_as_uint(__fsub_rn(lm, fabsf(t - (y - kMagic)))), mk, 1);
                        put(k, lv ? __float_as_uint(y) : 0x4B400000u);  // dead block: q = 0
                    }
                }
                if constexpr (kBiasPack) {
#pragma unroll
                    for (int w = 0; w < BITS; w++) words[w] -= pack_bias<BITS>(w);
                }
                if (valid) {
                    uint32_t* dst = reinterpret_cast<uint32_t*>(crow) + c * BITS;
                    if (BITS % 4 == 0) {
#pragma unroll
                        for (int w = 0; w < BITS; w += 4)
                            *reinterpret_cast<uint4*>(dst + w) = make_uint4(words[w], words[w + 1], words[w + 2], words[w + 3]);
                    } else if (BITS % 2 == 0) {
#pragma unroll
                        for (int w = 0; w < BITS; w += 2) *reinterpret_cast<uint2*>(dst + w) = make_uint2(words[w], words[w + 1]);
                    } else {
#pragma unroll
                        for (int w = 0; w < BITS; w++) dst[w] = words[w];
                    }
                }
                if (valid && lv) set4(am, c, mk);
            }
            bool pend = (am[0] | am[1] | am[2] | am[3]) != 0;
            while (__any_sync(0xffffffffu, pend)) {
                const int cnt = __popc(am[0]) + __popc(am[1]) + __popc(am[2]) + __popc(am[3]);
                int inc = cnt;
#pragma unroll
                for (int off = 1; off < 32; off <<= 1) {
                    const int t = __shfl_up_sync(0xffffffffu, inc, off);
                    if (lane >= off) inc += t;
                }
                const int base = inc - cnt;
                const int total = __shfl_sync(0xffffffffu, inc, 31);
                int slot = base;
#pragma unroll 1
                for (int c = 0; c < 4 && slot < kQCap; c++) {
                    uint32_t m = pick4(am, c);
                    while (m && slot < kQCap) {
                        const uint32_t col = (uint32_t)(c * 32 + __ffs(m) - 1);
                        qjob[2 * slot] = KEYS ? col | ((uint32_t)row << 8) : (uint32_t)row | (col << 8);
                        m &= m - 1;
                        slot++;
                    }
                }
                __syncwarp();
                run_jobs<kJobSlots>(qjob, min(total, kQCap), stg, Gf, g, lane);
                __syncwarp();
                slot = base;
#pragma unroll 1
                for (int c = 0; c < 4 && slot < kQCap; c++) {
                    uint32_t m = pick4(am, c);
                    while (m && slot < kQCap) {
                        const int col = c * 32 + __ffs(m) - 1;
                        const float ze = __uint_as_float(qjob[2 * slot + 1]);
                        const int bk = col / blk;
                        const uint32_t q = quant_code(ze, h2f_bits(pick4(s16, bk)), h2f_bits(pick4(m16, bk)), qmax);
                        patch_code<BITS>(crow, col * BITS, q);
                        m &= m - 1;
                        slot++;
                    }
                    set4(am, c, m);
                }
                __syncwarp();
                pend = (am[0] | am[1] | am[2] | am[3]) != 0;
            }

            // ---- 7. scales; release the stage and the accumulator buffer
            if (valid) {
                uint32_t* sp = KEYS ? a.scales + a.smap.at(ti.l, ti.s, ti.b, ti.h, ti.t0) + row
                                    : a.scales + a.smap.at(ti.l, ti.s, ti.b, ti.h, ti.t0 + row);
#pragma unroll
                for (int bk = 0; bk < 4; bk++)
                    if (bk < nbk) sp[bk] = s16[bk] | (m16[bk] << 16);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&M->accempty[buf]);
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
        tmem_dealloc(tmem, kAcc * 128);
    }
}

template <int BITS, bool KEYS, int NBK>
cudaError_t launch_encode_nbk(const EncParams& P, const CUtensorMap& map, cudaStream_t st) {
    const size_t smem = EncSmem::total;
    cudaError_t e =
        cudaFuncSetAttribute(tc_encode_kernel<BITS, KEYS, NBK>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = P.S.n_tiles < tc::num_sms() ? P.S.n_tiles : tc::num_sms();
    tc_encode_kernel<BITS, KEYS, NBK><<<(unsigned)grid, kThreads, smem, st>>>(map, P);
    return cudaGetLastError();
}

// keys: one block (the 128-token group) per channel (block-uniform and KIVI value rows are
// encoded by cg_tc_rows.cu)
template <int BITS, bool KEYS>
cudaError_t launch_encode_bits(const EncParams& P, const CUtensorMap& map, cudaStream_t st) {
    static_assert(KEYS, "rows are encoded by tc_rows_encode_kernel");
    return launch_encode_nbk<BITS, KEYS, 1>(P, map, st);
}

template <bool KEYS>
cudaError_t launch_encode(const RowArgs& a, cudaStream_t st) {
    EncParams P;
    P.a = a;
    P.S = tc::make_sched(a);
    if (P.S.n_tiles == 0) return cudaSuccess;
    CUtensorMap map;
    const uint64_t rows = (uint64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (!make_tmap_bf16_sw128(&map, a.x, rows, kD, kD * 2, 128)) return cudaErrorInvalidValue;
    switch (a.bits) {
        case 2: return launch_encode_bits<2, KEYS>(P, map, st);
        case 3: return launch_encode_bits<3, KEYS>(P, map, st);
        case 4: return launch_encode_bits<4, KEYS>(P, map, st);
        case 6: return launch_encode_bits<6, KEYS>(P, map, st);
        case 8: return launch_encode_bits<8, KEYS>(P, map, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

// KIVI keys as rows of the key tensor: s = 0 only, block = the 128-token key group, t_count
// = the quantized tokens (whole groups); cmap/smap address a group's first token (the
// kernel adds the channel's stream). Groups of g >= 32 channels (at most 4 per head).
bool tc_key_encode_eligible(const RowArgs& a) {
    if (a.d != kD || a.blk != 128 || a.g < 32) return false;
    if (a.t_count < 128 || a.t_count % 128) return false;
    const int64_t rows = (int64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (rows + 128 >= (int64_t)1 << 31) return false;
    if ((reinterpret_cast<uintptr_t>(a.x) & 15u) || (reinterpret_cast<uintptr_t>(a.codes) & 15u)) return false;
    return tmap_encode_fn() != nullptr;
}

cudaError_t tc_launch_key_encode(const RowArgs& a, cudaStream_t st) { return launch_encode<true>(a, st); }

}  // namespace cg
