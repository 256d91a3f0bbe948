// cg_tc_rows.cu -- tensor-core (tcgen05) encode of the row path, head dim d = 128: gauge
// rotation (Sec. 3, Z = G X) fused with the block-uniform quantizer of Sec. 4.3 (one range
// per block of `block` channels of a token), also used for KIVI value rows.
//
// Persistent warp-specialized kernel, one CTA per SM, 20 warps:
//   warp 0      TMA producer: 128-token x tiles (2 x [128 rows x 64 bf16], 128-byte
//               swizzle) into a 4-stage ring;
//   warp 1      MMA issuer: z~ = x G^T on tcgen05 (M = 128 tokens, N = K = gauge group, one
//               MMA chain per group block), G split into three bf16 terms (cg_tc_enc.cuh);
//               fp32 accumulators in tensor memory, four buffers;
//   warps 2, 19 gauge converters: at each gauge change they build the split operand and
//               the per-block error coefficients of the new gauge set (half of its rows each;
//               the MMAs wait for it, so it is kept short);
//   warps 3..18 four epilogue warpgroups; warpgroup k takes tiles i = k (mod 4); one
//               thread per token row (= TMEM lane). Four warps per SMSP hide more of the
//               epilogue's latencies than three; the kernel fits in 96 registers a thread.
//
// Epilogue of a tile, per row:
//   1. the group norms ||x_R||_2 that scale the error bound, from the staged tile with
//      bf16x2 fused multiply-adds (products exact, each partial sum rounded to bf16; at
//      most eight steps per accumulator, so the sum is at least (1 - 2^-8)^8 of the true
//      one and the inflated result bounds it from above); R is the gauge group, or the
//      block when blocks span several groups;
//   2. block min / max of z~ from tensor memory (two 32-column loads per wait, 3-input
//      min / max trees), the per-chunk extremes kept for step 4;
//   3. per block the bound E and the fp16 scale / zero decided from the error intervals
//      (both are monotone in the extremes, so equal interval ends decide them exactly);
//   4. blocks the intervals leave undecided: candidate extremes (values within 2E of the
//      approximate extreme, only in chunks whose own extreme qualifies) are recomputed
//      exactly in the library's order by the warp together (run_jobs);
//   5. codes straight from tensor memory: t = z~ * (1/s) - m/s, y = t + 1.5 * 2^23 (round to
//      nearest even in the add; y's bit pattern is 0x4B400000 + q), packed by wrapping sums
//      of y << (bit offset) less a compile-time constant. A chunk takes the short loop when
//      every lane's block needs no clamp and no boundary check (the usual case), else the
//      checked loop, which clamps and marks values within mu of a rounding boundary;
//   6. marked values (only when mu >= 1e-4, e.g. 8-bit codes) are recomputed and patched.
// The block count is a template parameter, so the per-block state of a row takes only the
// registers it needs; the chunk loops are not unrolled (the epilogue's code size sets its
// instruction-fetch stalls) and pick a chunk's block values with selects.
#include "cg_tc.h"
#include "cg_tc_enc.cuh"
#include "cg_tmap.h"

namespace cg {
namespace {

using namespace sm100;
using namespace tce;
using tc::kWaitLimitNs;

constexpr int kStages = 4;
constexpr int kTileBytes = 128 * kD * 2;
constexpr int kThreads = 640;
constexpr int kEpiWG = 4;  // epilogue warpgroups
constexpr int kConvWarp1 = 19;  // second gauge-converter warp (the first is warp 2)
constexpr int kEpiWarp0 = 3;
constexpr int kQCap = 20;  // repair jobs per warp and round
constexpr int kAcc = 4;    // accumulator buffers in tensor memory

struct RowSmem {
    static constexpr uint32_t stages = 0;
    static constexpr uint32_t bsplit = stages + kStages * kTileBytes;  // 3 x (16 or 32 KB)
    static constexpr uint32_t queue = bsplit + kNPass * 32768;         // 16 warps x kQCap x 8 B
    static constexpr uint32_t misc = queue + 4 * kEpiWG * kQCap * 8;
    static constexpr uint32_t total = misc + 512;  // base is 1024-aligned (checked in-kernel)
};

struct RowMisc {
    uint64_t full[kStages], empty[kStages];
    uint64_t accfull[kAcc], accempty[kAcc];
    uint64_t gready[kSegBufs];
    uint64_t bfree;
    uint32_t tmem_slot;
    int abort_flag;
    float emaxb[kSegBufs][2][4];  // per gauge set, converter warp and quantization block: max_i e_i
    float gmaxb[kSegBufs][2][4];  // and max_i ||G_i||
};

static_assert(sizeof(RowMisc) <= 512, "RowMisc outgrew its shared-memory slot");
static_assert(RowSmem::total <= 232448, "row encode kernel exceeds 227 KB of shared memory");

struct RowEncParams {
    RowArgs a;
    tc::Sched S;
    int nr;  // norm ranges per row: 128 / max(group, block)
};

// min and max of 32 fp32 values (bit patterns) by 3-input trees: 16 + 16 instructions
__device__ __forceinline__ void minmax32(const uint32_t (&v)[32], float& lo, float& hi) {
    float l[11], h[11];
#pragma unroll
    for (int k = 0; k < 10; k++) {
        l[k] = min3f(__uint_as_float(v[3 * k]), __uint_as_float(v[3 * k + 1]), __uint_as_float(v[3 * k + 2]));
        h[k] = max3f(__uint_as_float(v[3 * k]), __uint_as_float(v[3 * k + 1]), __uint_as_float(v[3 * k + 2]));
    }
    l[10] = fminf(__uint_as_float(v[30]), __uint_as_float(v[31]));
    h[10] = fmaxf(__uint_as_float(v[30]), __uint_as_float(v[31]));
    const float l0 = min3f(l[0], l[1], l[2]), l1 = min3f(l[3], l[4], l[5]), l2 = min3f(l[6], l[7], l[8]);
    const float h0 = max3f(h[0], h[1], h[2]), h1 = max3f(h[3], h[4], h[5]), h2 = max3f(h[6], h[7], h[8]);
    lo = fminf(min3f(l0, l1, l2), fminf(l[9], l[10]));
    hi = fmaxf(max3f(h0, h1, h2), fmaxf(h[9], h[10]));
}

// Element i (runtime) of a small register array, by selects (no local memory).
template <typename T, int N>
__device__ __forceinline__ T pickn(const T (&v)[N], int i) {
    T r = v[0];
#pragma unroll
    for (int k = 1; k < N; k++) r = i == k ? v[k] : r;
    return r;
}
template <typename T, int N>
__device__ __forceinline__ void setn(T (&v)[N], int i, T x) {
#pragma unroll
    for (int k = 0; k < N; k++) v[k] = i == k ? x : v[k];
}

__device__ __forceinline__ __nv_bfloat162 as_bf2(uint32_t w) {
    __nv_bfloat162 r;
    *reinterpret_cast<uint32_t*>(&r) = w;
    return r;
}

// Upper bound of the sum of squares of row `row`'s bf16 values over each of its NR norm
// ranges (128 / NR channels each), for block bk (range bk * NR / NBK) in nb[bk]. bf16x2
// fused multiply-adds square exactly and round each partial sum to bf16 (relative error at
// most 2^-8 per step, all terms non-negative); at most eight steps per accumulator, so the
// true sum is at most 1 / (1 - 2^-8)^8 < 1.0318 times the computed one; the fp32 combine adds
// at most 16 u; a floor of 128 x 2^-126 covers squares that underflow.
template <int NR, int NBK>
__device__ __forceinline__ void row_norms(const unsigned char* stg, int row, float (&nb)[NBK]) {
    constexpr int A = NR == 1 ? 2 : 1;  // accumulator sets per range
    __nv_bfloat162 acc[NR][A][4];
    const __nv_bfloat162 zero = as_bf2(0u);
#pragma unroll
    for (int r = 0; r < NR; r++)
#pragma unroll
        for (int s = 0; s < A; s++)
#pragma unroll
            for (int w = 0; w < 4; w++) acc[r][s][w] = zero;
#pragma unroll
    for (int c8 = 0; c8 < 16; c8++) {
        const uint4 xv = *reinterpret_cast<const uint4*>(stg + (c8 >> 3) * 16384 + row * 128 + (((c8 & 7) ^ (row & 7)) << 4));
        const int r = (c8 * NR) / 16, s = c8 % A;
        acc[r][s][0] = __hfma2(as_bf2(xv.x), as_bf2(xv.x), acc[r][s][0]);
        acc[r][s][1] = __hfma2(as_bf2(xv.y), as_bf2(xv.y), acc[r][s][1]);
        acc[r][s][2] = __hfma2(as_bf2(xv.z), as_bf2(xv.z), acc[r][s][2]);
        acc[r][s][3] = __hfma2(as_bf2(xv.w), as_bf2(xv.w), acc[r][s][3]);
    }
    float n2[NR];
#pragma unroll
    for (int r = 0; r < NR; r++) {
        float t = 0.0f;
#pragma unroll
        for (int s = 0; s < A; s++)
#pragma unroll
            for (int w = 0; w < 4; w++) t += __low2float(acc[r][s][w]) + __high2float(acc[r][s][w]);
        n2[r] = fmaf(t, 1.0325f, 1.5e-36f);
    }
#pragma unroll
    for (int bk = 0; bk < NBK; bk++) nb[bk] = n2[(bk * NR) / NBK];
}

// BITS-bit code of z~ in the packed word set of a 32-code chunk: y = 0x4B400000 + q is added
// shifted to its bit offset (wrapping sums; the constant part is removed at the end), the
// high bits of a code that straddles two words go to the next word.
template <int BITS>
__device__ __forceinline__ void put_code(uint32_t (&words)[BITS], int k, uint32_t y) {
    constexpr uint32_t qmask = (1u << BITS) - 1u;
    const int bit = k * BITS;
    words[bit >> 5] += y << (bit & 31);
    if ((bit & 31) + BITS > 32) words[(bit >> 5) + 1] += (y & qmask) >> (32 - (bit & 31));
}

template <int BITS, int NBK>
__global__ void __launch_bounds__(kThreads, 1) tc_rows_encode_kernel(const __grid_constant__ CUtensorMap xmap,
                                                                      const RowEncParams P) {
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    if (smem_u32(smem_raw) & 1023u) {
        // the swizzled tiles need a 1024-byte aligned base; the layout leaves no slack
        if (threadIdx.x == 0) raise_flag(P.a.status, CG_FLAG_PIPE_TIMEOUT);
        return;
    }
    unsigned char* sm = smem_raw;
    RowMisc* M = reinterpret_cast<RowMisc*>(sm + RowSmem::misc);
    unsigned char* stages = sm + RowSmem::stages;
    unsigned char* bsplit = sm + RowSmem::bsplit;
    uint32_t* queue = reinterpret_cast<uint32_t*>(sm + RowSmem::queue);

    const RowArgs& a = P.a;
    const tc::Sched& S = P.S;
    const int g = a.g;
    constexpr int blk = kD / NBK;  // quantization block: NBK blocks per row
    constexpr int CPB = 4 / NBK;   // 32-column chunks per block
    const int gb = g < 16 ? 16 : g;
    // gauge operand layout: full K = 128 for g = 128, else one g-wide K block per group
    const bool fullk = g == 128;
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
        for (int i = 0; i < kSegBufs; i++) mbar_init(&M->gready[i], 2);
        mbar_init(&M->bfree, 1);
        M->abort_flag = 0;
        fence_barrier_init();
    }
    for (uint32_t i = threadIdx.x; i < (uint32_t)kNPass * bsz / 16; i += kThreads)
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
                // the cache tiles are read once: first out of L2, so that the gauge sets the
                // exact recomputes read stay there
                const uint64_t pol = policy_evict_first();
                tma_load_2d_hint(dst, &xmap, &M->full[st], 0, (int)row0, pol);
                tma_load_2d_hint(dst + 16384, &xmap, &M->full[st], 64, (int)row0, pol);
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
        // A tile is always 24 MMAs (3 split terms x 128 / 16 K-steps, in one chain per gauge
        // group). Their B descriptors, A offsets and accumulator columns are laid out once,
        // so per tile the single issuing thread only adds the stage's A base: descriptor
        // arithmetic in that thread would otherwise set the pace of the whole pipeline.
        if (lane == 0 && my_tiles > 0) {
            constexpr int kMma = kNPass * (kD / 16);
            const uint32_t idesc = idesc_bf16_f32(128, gb);
            uint64_t bdesc[kMma];
            uint32_t aoff[kMma], doff[kMma], accb = 0;
#pragma unroll
            for (int q = 0; q < kMma; q++) {
                const int p = q / (kD / 16), kk = q % (kD / 16);  // pass, K-step over the row
                const int r = (kk * 16) / gb, ks = kk - r * (gb / 16);
                const int k0 = kk * 16;
                aoff[q] = (uint32_t)(((k0 >> 6) * 16384 + (k0 & 63) * 2) >> 4);
                bdesc[q] = sdesc_sw128(smem_u32(bsplit) + p * bsz + (fullk ? (k0 >> 6) * 16384 : 0) + (r * gb) * 128 +
                                       (k0 & 63) * 2);
                doff[q] = (uint32_t)(r * gb);
                accb |= (uint32_t)(p > 0 || ks > 0) << q;
            }
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
                const uint64_t adesc = sdesc_sw128(smem_u32(stages + st * kTileBytes));
                const uint32_t d_base = tmem + buf * 128;
                // D[token][channel] = x G^T, one chain per gauge group
#pragma unroll
                for (int q = 0; q < kMma; q++) mma_bf16(d_base + doff[q], adesc + aoff[q], bdesc[q], idesc, (accb >> q) & 1u);
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
    } else if (warp == 2 || warp == kConvWarp1) {
        // ------------------------------------------------------------ gauge converters
        // (two warps, 64 of the 128 gauge rows each)
        const int cw = warp == 2 ? 0 : 1;
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
            if (cw == 0) prefetch_next_gauges(a, ti, g, lane);
            (void)convert_gauge_set<false, 2>(Gf, g, blk, NBK, fullk, bsz, bsplit, M->emaxb[ls & 3][cw],
                                              M->gmaxb[ls & 3][cw], 2 * cw, lane);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(&M->gready[ls & 3]);
            cur = ti.seg;
            nconv++;
        }
    } else {
        // ------------------------------------------------------------ epilogue warpgroups
        const int wg = (warp - kEpiWarp0) >> 2;  // warpgroup: tiles i = wg (mod kEpiWG)
        const int q4 = warp & 3;                 // TMEM lane quadrant of this warp
        const int row = q4 * 32 + lane;          // TMEM lane = token row of the tile
        const int qw = warp - kEpiWarp0;         // job queue of this warp
        uint32_t* qjob = queue + qw * kQCap * 2;
        constexpr float qmaxf = (float)((1 << BITS) - 1);
        constexpr float kRq = 1.0f / qmaxf;        // fl(1 / qmax)
        constexpr float kBelow1 = 1.0f - 8.0f * kU;  // 1 - 2^-21 and 1 + 2^-21, both exact in fp32
        constexpr float kAbove1 = 1.0f + 8.0f * kU;
        constexpr int qmax = (1 << BITS) - 1;
        constexpr int kJobSlots = NBK == 2 ? 4 : 2;  // values per lane and memory round trip
        int32_t flag = 0;
        tc::TileIter it;
        it.init(a, S, t_begin + wg);
        for (int i = wg; i < my_tiles; i += kEpiWG, it.step(a, kEpiWG)) {
            const tc::TileInfo ti = it.info(a);
            const int64_t ls = ti.seg - seg0;
            const int st = i % kStages, buf = i % kAcc;
            bool ok = mbar_wait(&M->full[st], (i / kStages) & 1, abort_flag, a.wait_ns);
            ok = ok && mbar_wait(&M->gready[ls & 3], (ls >> 2) & 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            const unsigned char* stg = stages + st * kTileBytes;
            const bool valid = row < ti.rows_valid;
            const float* Gf = a.G + tc::gauge_set(a, ti) * (int64_t)kD * g;

            // ---- 1. sums of squares of the norm range of every block
            float nb[NBK];
            if (P.nr == 1) {
                row_norms<1, NBK>(stg, row, nb);
            } else if (P.nr == 2) {
                if constexpr (NBK >= 2) row_norms<2, NBK>(stg, row, nb);
            } else {
                if constexpr (NBK >= 4) row_norms<4, NBK>(stg, row, nb);
            }
            bool fin = true;
#pragma unroll
            for (int bk = 0; bk < NBK; bk++) fin = fin && isfinite(nb[bk]);
            if (valid && !fin) {
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

            // ---- 2. block ranges of z~ from the accumulator
            ok = mbar_wait(&M->accfull[buf], (i / kAcc) & 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            const uint32_t tacc = tmem + ((uint32_t)(q4 * 32) << 16) + buf * 128;
            float cmn[4], cmx[4];  // per 32-column chunk
#pragma unroll 1
            for (int h = 0; h < 2; h++) {
                uint32_t va[32], vb[32];
                tmem_ld32(tacc + (2 * h) * 32, va);
                tmem_ld32(tacc + (2 * h + 1) * 32, vb);
                tmem_wait_ld();
                float l0, h0, l1, h1;
                minmax32(va, l0, h0);
                minmax32(vb, l1, h1);
                setn(cmn, 2 * h, l0);
                setn(cmx, 2 * h, h0);
                setn(cmn, 2 * h + 1, l1);
                setn(cmx, 2 * h + 1, h1);
            }
            float mn[NBK], mx[NBK];
#pragma unroll
            for (int bk = 0; bk < NBK; bk++) {
                mn[bk] = cmn[bk * CPB];
                mx[bk] = cmx[bk * CPB];
#pragma unroll
                for (int c = 1; c < CPB; c++) {
                    mn[bk] = fminf(mn[bk], cmn[bk * CPB + c]);
                    mx[bk] = fmaxf(mx[bk], cmx[bk * CPB + c]);
                }
            }

            // ---- 3. error bound per block; scale/zero from the intervals when they agree
            float E[NBK], Ec[NBK];  // Ec bounds |z~ - z|; E adds the rounding of the interval ends
            uint32_t s16[NBK], m16[NBK];
            int amb = 0;  // bit 2bk: scale needs the exact extremes; bit 2bk+1: zero needs the exact min
#pragma unroll
            for (int bk = 0; bk < NBK; bk++) {
                const float emax = fmaxf(M->emaxb[ls & 3][0][bk], M->emaxb[ls & 3][1][bk]);
                Ec[bk] = sqrtf(nb[bk]) * 1.0001f * emax;
                E[bk] = Ec[bk] + (fabsf(mn[bk]) + fabsf(mx[bk])) * 2.4e-7f;
                const float e = E[bk];
                const float mn_lo = __fsub_rn(mn[bk], e), mn_hi = __fadd_rn(mn[bk], e);
                const float mx_lo = __fsub_rn(mx[bk], e), mx_hi = __fadd_rn(mx[bk], e);
                // fp16 scales of the smallest and largest possible ranges. fl(d * fl(1/qmax))
                // is within (1 +- u)^2 of d / qmax and the widening product adds one more
                // rounding, so the products widened by 8u bracket the IEEE quotients of both
                // ends (which are within u of d / qmax); fp16 rounding is monotone, so equal
                // roundings of the bracket decide the scale exactly (no division on this path)
                const float dlo = fmaxf(__fsub_rn(mx_lo, mn_hi), 0.0f), dhi = __fsub_rn(mx_hi, mn_lo);
                const uint32_t slo = f2h_bits(__fmul_rn(__fmul_rn(dlo, kRq), kBelow1));
                const uint32_t shi = f2h_bits(__fmul_rn(__fmul_rn(dhi, kRq), kAbove1));
                const uint32_t mlo = f2h_bits(mn_lo), mhi = f2h_bits(mn_hi);
                s16[bk] = slo;
                m16[bk] = mlo;
                if (valid && slo != shi) amb |= 1 << (2 * bk);
                if (valid && mlo != mhi) amb |= 2 << (2 * bk);
            }

            // ---- 4. exact extremes of undecided blocks (warp-cooperative rounds)
            if (__any_sync(0xffffffffu, amb != 0)) {
                // candidates of an undecided block's min (max): its values within 2E of the
                // approximate min (max), only in chunks whose own min (max) lies that close
                uint32_t pm[4] = {0, 0, 0, 0}, px[4] = {0, 0, 0, 0};
#pragma unroll 1
                for (int c = 0; c < 4; c++) {
                    const int bk = c / CPB;
                    const int need = (amb >> (2 * bk)) & 3;
                    const float e2 = 2.0f * pickn(E, bk);
                    const float tl = __fadd_rn(pickn(mn, bk), e2), th = __fsub_rn(pickn(mx, bk), e2);
                    const bool nl = need != 0 && pickn(cmn, c) <= tl;
                    const bool nh = (need & 1) && pickn(cmx, c) >= th;
                    uint32_t m0 = 0, m1 = 0;
                    const bool anyl = __any_sync(0xffffffffu, nl), anyh = __any_sync(0xffffffffu, nh);
                    if (anyl || anyh) {
                        uint32_t v[32];
                        tmem_ld32(tacc + c * 32, v);
                        tmem_wait_ld();
                        // sign bits of tl - z (z > tl) and z - th (z < th), one bit per column;
                        // each side only when some lane of the warp needs it (with four blocks
                        // per row, one loop for both keeps the row's state in registers)
                        uint32_t a0 = 0, a1 = 0;
                        if constexpr (NBK == 4) {
#pragma unroll
                            for (int k = 31; k >= 0; k--) {
                                const float z = __uint_as_float(v[k]);
                                a0 = __funnelshift_l(__float_as_uint(__fsub_rn(tl, z)), a0, 1);
                                a1 = __funnelshift_l(__float_as_uint(__fsub_rn(z, th)), a1, 1);
                            }
                        } else {
                            if (anyl) {
#pragma unroll
                                for (int k = 31; k >= 0; k--)
                                    a0 = __funnelshift_l(__float_as_uint(__fsub_rn(tl, __uint_as_float(v[k]))), a0, 1);
                            }
                            if (anyh) {
#pragma unroll
                                for (int k = 31; k >= 0; k--)
                                    a1 = __funnelshift_l(__float_as_uint(__fsub_rn(__uint_as_float(v[k]), th)), a1, 1);
                            }
                        }
                        m0 = nl ? ~a0 : 0u;  // z <= tl
                        m1 = nh ? ~a1 : 0u;  // z >= th
                    }
                    setn(pm, c, m0);
                    setn(px, c, m1);
                }
                float ex_mn[NBK], ex_mx[NBK];
#pragma unroll
                for (int bk = 0; bk < NBK; bk++) {
                    ex_mn[bk] = INFINITY;
                    ex_mx[bk] = -INFINITY;
                }
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
                        uint32_t m = pickn(pm, c) | pickn(px, c);
                        while (m && slot < kQCap) {
                            const uint32_t col = (uint32_t)(c * 32 + __ffs(m) - 1);
                            qjob[2 * slot] = (uint32_t)row | (col << 8);
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
                        const int bk = c / CPB;
                        uint32_t cm = pickn(pm, c), cx = pickn(px, c);
                        uint32_t m = cm | cx;
                        float emn = pickn(ex_mn, bk), emx = pickn(ex_mx, bk);
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
                        setn(ex_mn, bk, emn);
                        setn(ex_mx, bk, emx);
                        setn(pm, c, cm);
                        setn(px, c, cx);
                    }
                    __syncwarp();
                    pend = (pm[0] | pm[1] | pm[2] | pm[3] | px[0] | px[1] | px[2] | px[3]) != 0;
                }
#pragma unroll
                for (int bk = 0; bk < NBK; bk++) {
                    const int need = (amb >> (2 * bk)) & 3;
                    if (need) {
                        m16[bk] = f2h_bits(ex_mn[bk]);
                        if (need & 1) s16[bk] = scale16(ex_mx[bk], ex_mn[bk], qmaxf);
                    }
                }
            }

            // ---- 5. code parameters per block
            float rinv[NBK], c0[NBK], lim[NBK];
            bool fast[NBK];  // no value of the block can leave [0, qmax] and mu < 1e-4
#pragma unroll
            for (int bk = 0; bk < NBK; bk++) {
                rinv[bk] = c0[bk] = 0.0f;
                lim[bk] = 0.5f;
                fast[bk] = true;  // a dead block (zero or overflowing scale) codes to 0 with r = c0 = 0
                if (valid && (h_is_inf(s16[bk]) || h_is_inf(m16[bk]))) flag |= CG_FLAG_FP16_OVERFLOW;
                const float sc = h2f_bits(s16[bk]), mz = h2f_bits(m16[bk]);
                if (sc != 0.0f && !h_is_inf(s16[bk]) && !h_is_inf(m16[bk])) {
                    const float r = __frcp_rn(sc);
                    const float cc = -mz * r;
                    rinv[bk] = r;
                    c0[bk] = cc;
                    // |t~ - t| <= |z~ - z| / s plus roundings: the fma and its inputs r and c0 (u|z r|,
                    // 2u|c0|, u|t|) and the definition's subtract and divide (2u|t|)
                    const float zr = fmaxf(fabsf(mn[bk]), fabsf(mx[bk])) * r;
                    const float mu = Ec[bk] * r * 1.0001f + (zr + 2.0f * fabsf(cc) + 3.0f * (qmaxf + 1.0f)) * 6.6e-8f;
                    // mu < 1e-4: a code from z~ can only differ where the tolerance allows it
                    lim[bk] = mu < 0.99e-4f ? 2.0f : 0.5f - mu;
                    const float tlo = (mn[bk] - E[bk]) * r + cc, thi = (mx[bk] + E[bk]) * r + cc;
                    fast[bk] = tlo > -0.49f + mu && thi < qmaxf + 0.49f - mu && lim[bk] > 1.0f;
                }
            }

            // ---- 6. codes from z~, stored straight from registers
            uint8_t* crow = a.codes + a.cmap.at(ti.l, ti.s, ti.b, ti.h, ti.t0 + row);
            uint32_t am[4] = {0, 0, 0, 0};  // values within mu of a rounding boundary
#pragma unroll 1
            for (int c = 0; c < 4; c++) {
                uint32_t v[32];
                tmem_ld32(tacc + c * 32, v);
                tmem_wait_ld();
                const int bk = c / CPB;
                const float r = pickn(rinv, bk), cz = pickn(c0, bk);
                const bool fst = pickn(fast, bk);
                uint32_t words[BITS];
#pragma unroll
                for (int w = 0; w < BITS; w++) words[w] = 0;
                uint32_t mk = 0;
                if (__all_sync(0xffffffffu, fst)) {
                    // the same fma and add per value, two values per instruction
                    const float2 r2 = make_float2(r, r), c2 = make_float2(cz, cz), m2 = make_float2(kMagic, kMagic);
#pragma unroll
                    for (int k = 0; k < 32; k += 2) {
                        const float2 y = __fadd2_rn(
                            __ffma2_rn(make_float2(__uint_as_float(v[k]), __uint_as_float(v[k + 1])), r2, c2), m2);
                        put_code<BITS>(words, k, __float_as_uint(y.x));
                        put_code<BITS>(words, k + 1, __float_as_uint(y.y));
                    }
                } else {
                    // clamping before the rounding gives the same code as clamping after it
                    const float lm = pickn(lim, bk);
#pragma unroll
                    for (int k = 31; k >= 0; k--) {
                        float t = fmaf(__uint_as_float(v[k]), r, cz);
                        t = fminf(fmaxf(t, 0.0f), qmaxf);
                        const float y = t + kMagic;
                        mk = __funnelshift_l(__float_as_uint(__fsub_rn(lm, fabsf(t - (y - kMagic)))), mk, 1);
                        put_code<BITS>(words, k, __float_as_uint(y));
                    }
                    if (fst) mk = 0;
                }
#pragma unroll
                for (int w = 0; w < BITS; w++) words[w] -= pack_bias<BITS>(w);
                if (valid) {
                    uint32_t* dst = reinterpret_cast<uint32_t*>(crow) + c * BITS;
                    if constexpr (BITS % 4 == 0) {
#pragma unroll
                        for (int w = 0; w < BITS; w += 4)  // written once: first out of L2
                            stg_hint_u4(dst + w, make_uint4(words[w], words[w + 1], words[w + 2], words[w + 3]),
                                        policy_evict_first());
                    } else if constexpr (BITS % 2 == 0) {
#pragma unroll
                        for (int w = 0; w < BITS; w += 2) *reinterpret_cast<uint2*>(dst + w) = make_uint2(words[w], words[w + 1]);
                    } else {
#pragma unroll
                        for (int w = 0; w < BITS; w++) dst[w] = words[w];
                    }
                    setn(am, c, mk);
                }
            }

            // ---- 7. values within mu of a rounding boundary: exact recompute and patch
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
                    uint32_t m = pickn(am, c);
                    while (m && slot < kQCap) {
                        const uint32_t col = (uint32_t)(c * 32 + __ffs(m) - 1);
                        qjob[2 * slot] = (uint32_t)row | (col << 8);
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
                    const int bk = c / CPB;
                    uint32_t m = pickn(am, c);
                    const float sb = h2f_bits(pickn(s16, bk)), mb = h2f_bits(pickn(m16, bk));
                    while (m && slot < kQCap) {
                        const int col = c * 32 + __ffs(m) - 1;
                        const float ze = __uint_as_float(qjob[2 * slot + 1]);
                        patch_code<BITS>(crow, col * BITS, quant_code(ze, sb, mb, qmax));
                        m &= m - 1;
                        slot++;
                    }
                    setn(am, c, m);
                }
                __syncwarp();
                pend = (am[0] | am[1] | am[2] | am[3]) != 0;
            }

            // ---- 8. scales; release the stage and the accumulator buffer
            if (valid) {
                uint32_t* sp = a.scales + a.smap.at(ti.l, ti.s, ti.b, ti.h, ti.t0 + row);
                const bool vec = (reinterpret_cast<uintptr_t>(sp) & (NBK * 4 - 1)) == 0;
                if (NBK == 4 && vec) {
                    *reinterpret_cast<uint4*>(sp) = make_uint4(s16[0] | (m16[0] << 16), s16[1] | (m16[1] << 16),
                                                               s16[NBK > 2 ? 2 : 0] | (m16[NBK > 2 ? 2 : 0] << 16),
                                                               s16[NBK > 3 ? 3 : 0] | (m16[NBK > 3 ? 3 : 0] << 16));
                } else if (NBK == 2 && vec) {
                    *reinterpret_cast<uint2*>(sp) = make_uint2(s16[0] | (m16[0] << 16), s16[NBK > 1 ? 1 : 0] | (m16[NBK > 1 ? 1 : 0] << 16));
                } else {
#pragma unroll
                    for (int bk = 0; bk < NBK; bk++) sp[bk] = s16[bk] | (m16[bk] << 16);
                }
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

template <int BITS, int NBK>
cudaError_t launch_rows(const RowEncParams& P, const CUtensorMap& map, cudaStream_t st) {
    const size_t smem = RowSmem::total;
    cudaError_t e = cudaFuncSetAttribute(tc_rows_encode_kernel<BITS, NBK>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = P.S.n_tiles < tc::num_sms() ? P.S.n_tiles : tc::num_sms();
    tc_rows_encode_kernel<BITS, NBK><<<(unsigned)grid, kThreads, smem, st>>>(map, P);
    return cudaGetLastError();
}

template <int BITS>
cudaError_t launch_rows_bits(const RowEncParams& P, const CUtensorMap& map, cudaStream_t st) {
    if (P.a.blk == 128) return launch_rows<BITS, 1>(P, map, st);
    if (P.a.blk == 64) return launch_rows<BITS, 2>(P, map, st);
    return launch_rows<BITS, 4>(P, map, st);
}

}  // namespace

bool tc_row_encode_eligible(const RowArgs& a) {
    if (a.d != kD || a.none_mode) return false;
    if (!(a.blk == 32 || a.blk == 64 || a.blk == 128)) return false;
    if (a.t_count < 64) return false;
    const int64_t rows = (int64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (rows + 128 >= (int64_t)1 << 31) return false;
    if ((reinterpret_cast<uintptr_t>(a.x) & 15u) || (reinterpret_cast<uintptr_t>(a.codes) & 15u)) return false;
    return tmap_encode_fn() != nullptr;
}

cudaError_t tc_launch_row_encode(const RowArgs& a, cudaStream_t st) {
    RowEncParams P;
    P.a = a;
    P.S = tc::make_sched(a);
    P.nr = kD / (a.g > a.blk ? a.g : a.blk);
    if (P.S.n_tiles == 0) return cudaSuccess;
    CUtensorMap map;
    const uint64_t rows = (uint64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (!make_tmap_bf16_sw128(&map, a.x, rows, kD, kD * 2, 128)) return cudaErrorInvalidValue;
    switch (a.bits) {
        case 2: return launch_rows_bits<2>(P, map, st);
        case 3: return launch_rows_bits<3>(P, map, st);
        case 4: return launch_rows_bits<4>(P, map, st);
        case 6: return launch_rows_bits<6>(P, map, st);
        case 8: return launch_rows_bits<8>(P, map, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace cg
