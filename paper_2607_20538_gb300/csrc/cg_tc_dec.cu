// cg_tc_dec.cu -- tensor-core decode of the row path (Sec. 3: Zhat = D(B_c), Xhat = G^T Zhat),
// head dim d = 128, block-uniform rows and KIVI value rows.
//
// Persistent warp-specialized kernel, one CTA per SM, 14 warps:
//   warp 0      bulk-copy producer: the packed codes of a 128-token tile are contiguous
//               (rows of 16*bits bytes); one cp.async.bulk per tile into a ring of stages;
//   warp 1      MMA issuer: D_k = A_k B^T on tcgen05, A = codes as bf16 (2^b + q, exact;
//               8-bit codes as q),
//               B = G^T of the gauge group split into two bf16 terms; one fp32
//               accumulator per quantization sub-block k of a group (block < group gives
//               two), double buffered in tensor memory (tile i uses buffer i mod 2);
//   warps 2..5  unpackers, one token row each: codes -> bf16 A tile (128-byte swizzle);
//               at a gauge change they also build B and the per-column sums c_k[i] =
//               sum_{j in sub-block k} G[j][i] of the split;
//   warps 6..13 epilogue: both warpgroups work on every tile, warpgroup h on output
//               columns 64h..64h+63, one token row (TMEM lane) per thread:
//               xhat_i = sum_k s_k * D_k[i] + (m_k - 2^b s_k) * c_k[i]. The accumulator
//               buffer is released as soon as it is in registers, so the MMAs of tile i+2
//               overlap the arithmetic of tile i; each warp stages its 32 x 64 bf16 block
//               in shared memory (128-byte swizzle) and writes it with one TMA tile store.
//               Each thread loads the next tile's block scales one tile ahead.
// With the scale and zero of a block constant along the token, dequantization commutes
// with the rotation, so the integer codes go through the tensor cores unscaled. In real
// arithmetic s_k D_k + (m_k - 2^b s_k) c_k = sum_j (hi + lo)_ji zhat_j, so the split residual
// of G is not amplified by the offset; the offset only scales the fp32 rounding of D_k and of
// the zero-point term, which is why it is the smallest power of two that keeps 2^b + q a
// plain bit pattern (2^b + q has b significant bits below its leading one), and why c_k is
// a compensated sum. The number of sub-block accumulators is a template parameter, so each
// kernel holds only its own epilogue.
#include <cuda_bf16.h>

#include "cg_sm100.cuh"
#include "cg_tc.h"
#include "cg_tc_common.cuh"
#include "cg_tmap.h"

namespace cg {
namespace {

using namespace sm100;
using tc::kD;
using tc::kWaitLimitNs;

constexpr int kThreads = 448;
constexpr int kEpiWarp0 = 6;
constexpr int kATile = 128 * kD * 2;
constexpr int kSegBufs = 4;
constexpr int kMaxCStages = 4;
constexpr uint32_t kOutWarpBytes = 32 * 128;  // 32 rows x 64 bf16 per epilogue warp
constexpr int kMmaPerTile = 16;  // 2 split terms x 128 / 16 K steps, for every group and block

template <int BITS>
struct DecSmem {
    static constexpr int cstages_n = BITS == 8 ? 3 : 4;
    static constexpr uint32_t cstage_bytes = 128u * 16u * BITS;  // 128 rows of packed codes
    static constexpr uint32_t a_tiles = 0;                        // 2 x 32 KB
    static constexpr uint32_t bsplit = a_tiles + 2 * kATile;      // 2 x (16 or 32 KB)
    static constexpr uint32_t ostage = bsplit + 2 * 32768;        // 8 warps x 4 KB
    static constexpr uint32_t cstages = ostage + 8 * kOutWarpBytes;
    static constexpr uint32_t csum = cstages + cstages_n * cstage_bytes;  // [4][2][128] fp32
    static constexpr uint32_t misc = csum + kSegBufs * 2 * kD * 4;
    static constexpr uint32_t total = misc + 512;
    static_assert(ostage % 1024 == 0 && cstages % 1024 == 0, "swizzled tiles need 1024-byte alignment");
    static_assert(total + 1024 <= 232448, "shared memory budget");
};

struct DecMisc {
    uint64_t cfull[kMaxCStages], cempty[kMaxCStages];
    uint64_t afull[2], aempty[2];
    uint64_t accfull[2], accempty[2];
    uint64_t gready[kSegBufs];
    uint64_t bfree;
    uint32_t mseq[16][4];  // the MMA sequence of a tile
    uint32_t tmem_slot;
    int abort_flag;
};

static_assert(sizeof(DecMisc) <= 512, "misc block");

struct DecParams {
    RowArgs a;
    tc::Sched S;
    int nsub;  // accumulators per gauge group: group / block when block < group, else 1
};

// bf16 bit pattern of 2^BITS + q (q < 2^BITS): exponent of 2^BITS, q in the top BITS of the
// 7 mantissa bits
template <int BITS>
__host__ __device__ constexpr uint32_t code_bf16_base() {
    return (uint32_t)(127 + BITS) << 7;
}

// codes of one row (128 codes, little-endian bit stream) -> 16 chunks of 8 bf16 (2^b + q; 8-bit
// codes as q)
template <int BITS>
__device__ __forceinline__ void unpack_row(const uint32_t* w, uint4 (&out)[16]) {
    if constexpr (BITS == 4) {
        // eight nibbles per word: place the low/high nibbles at mantissa bits 3..6 of their
        // bytes (with the exponent's low bit 0x80), interleave them back into code order
        // with byte permutes, then pair each byte with the 0x41 exponent byte (16 + q)
#pragma unroll
        for (int c = 0; c < 16; c++) {
            const uint32_t lo_n = ((w[c] << 3) & 0x78787878u) | 0x80808080u;  // codes 0, 2, 4, 6
            const uint32_t hi_n = ((w[c] >> 1) & 0x78787878u) | 0x80808080u;  // codes 1, 3, 5, 7
            const uint32_t q03 = __byte_perm(lo_n, hi_n, 0x5140);  // codes 0..3 as bytes
            const uint32_t q47 = __byte_perm(lo_n, hi_n, 0x7362);  // codes 4..7
            out[c] = make_uint4(__byte_perm(q03, 0x41u, 0x4140), __byte_perm(q03, 0x41u, 0x4342),
                                __byte_perm(q47, 0x41u, 0x4140), __byte_perm(q47, 0x41u, 0x4342));
        }
    } else {
#pragma unroll
        for (int c = 0; c < 16; c++) {
            uint32_t o[4];
#pragma unroll
            for (int e = 0; e < 4; e++) {
                uint32_t q[2];
#pragma unroll
                for (int h = 0; h < 2; h++) {
                    const int k = 8 * c + 2 * e + h;
                    const int p = k * BITS;
                    uint32_t v = w[p >> 5] >> (p & 31);
                    if ((p & 31) + BITS > 32) v |= w[(p >> 5) + 1] << (32 - (p & 31));
                    q[h] = v & ((1u << BITS) - 1u);
                }
                if (BITS < 8) {
                    constexpr uint32_t base = code_bf16_base<BITS>() * 0x10001u;
                    o[e] = base | (q[0] << (7 - BITS)) | (q[1] << (23 - BITS));
                } else {
                    const __nv_bfloat162 b2 = __floats2bfloat162_rn((float)q[0], (float)q[1]);
                    o[e] = *reinterpret_cast<const uint32_t*>(&b2);
                }
            }
            out[c] = make_uint4(o[0], o[1], o[2], o[3]);
        }
    }
}

template <int BITS, int NSUB>
__global__ void __launch_bounds__(kThreads, 1) tc_decode_kernel(const __grid_constant__ CUtensorMap omap,
                                                                 const DecParams P) {
    using SL = DecSmem<BITS>;
    constexpr int kCStages = SL::cstages_n;
    constexpr uint32_t kCStageBytes = SL::cstage_bytes;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t base_u32 = (smem_u32(smem_raw) + 1023u) & ~1023u;
    unsigned char* sm = smem_raw + (base_u32 - smem_u32(smem_raw));
    DecMisc* M = reinterpret_cast<DecMisc*>(sm + SL::misc);
    unsigned char* atiles = sm + SL::a_tiles;
    unsigned char* bsplit = sm + SL::bsplit;
    unsigned char* cst = sm + SL::cstages;
    float* csum = reinterpret_cast<float*>(sm + SL::csum);

    const RowArgs& a = P.a;
    const tc::Sched& S = P.S;
    const int g = a.g, blk = a.blk;
    constexpr int nsub = NSUB;  // accumulators per gauge group
    const int gb = g < 16 ? 16 : g;
    const uint32_t bsz = (g == 128) ? 32768u : 16384u;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr int kRowBytes = 16 * BITS;
    constexpr float kOff = BITS < 8 ? (float)(1 << BITS) : 0.0f;

    const int64_t t_begin = S.n_tiles * blockIdx.x / gridDim.x;
    const int64_t t_end = S.n_tiles * (blockIdx.x + 1) / gridDim.x;
    const int my_tiles = (int)(t_end - t_begin);
    const int64_t seg0 = my_tiles > 0 ? tc::tile_info(a, S, t_begin).seg : 0;
    const uint32_t acc_cols = (uint32_t)nsub * 128u;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kCStages; i++) {
            mbar_init(&M->cfull[i], 1);
            mbar_init(&M->cempty[i], 4);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&M->afull[i], 4);
            mbar_init(&M->aempty[i], 1);
            mbar_init(&M->accfull[i], 1);
            mbar_init(&M->accempty[i], 8);
        }
        for (int i = 0; i < kSegBufs; i++) mbar_init(&M->gready[i], 4);
        mbar_init(&M->bfree, 1);
        M->abort_flag = 0;
        fence_barrier_init();
    }
    for (uint32_t i = threadIdx.x; i < 2u * bsz / 16u; i += kThreads)
        reinterpret_cast<uint4*>(bsplit)[i] = make_uint4(0, 0, 0, 0);
    if (warp == 1) {
        tmem_alloc(&M->tmem_slot, 2 * acc_cols);
        tmem_relinquish();
        tc_fence_before();
    }
    fence_proxy_async_smem();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = M->tmem_slot;
    volatile int* abort_flag = &M->abort_flag;

    if (warp == 0) {
        // ------------------------------------------------------------ codes producer
        if (lane == 0 && my_tiles > 0) {
            int issued = 0;
            tc::TileIter it;
            it.init(a, S, t_begin);
            for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
                const int st = i % kCStages;
                if (!mbar_wait(&M->cempty[st], ((i / kCStages) & 1) ^ 1, abort_flag, a.wait_ns)) {
                    *abort_flag = 1;
                    break;
                }
                const tc::TileInfo ti = it.info(a);
                const uint32_t bytes = (uint32_t)ti.rows_valid * kRowBytes;
                mbar_arrive_expect_tx(&M->cfull[st], bytes);
                bulk_load(cst + st * kCStageBytes, a.codes + a.cmap.at(ti.l, ti.s, ti.b, ti.h, ti.t0), bytes,
                          &M->cfull[st]);
                issued = i + 1;
            }
            if (*abort_flag) {
                const int zero = 0;
                const int from = issued > kCStages ? issued - kCStages : 0;
                for (int i = from; i < issued; i++)
                    mbar_wait(&M->cfull[i % kCStages], (i / kCStages) & 1, &zero, kWaitLimitNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && my_tiles > 0) {
            const uint32_t idesc = idesc_bf16_f32(128, gb);
            // The MMAs of a tile form a fixed sequence (16 for every supported group and
            // block): D column offset, A and B byte offsets, accumulate flag. It is laid out
            // once; per tile only the stage bases change.
            int nseq = 0;
            {
                int& n = nseq;
                for (int p = 0; p < 2; p++)
                    for (int r = 0; r < 128 / gb; r++)
                        for (int k = 0; k < nsub; k++) {
                            const int kw = nsub > 1 ? blk : gb;  // K width of this sub-block
                            const int kbeg = r * gb + k * (nsub > 1 ? blk : 0);
                            for (int ks = 0; ks < kw / 16 && n < kMmaPerTile; ks++, n++) {
                                const int k0 = kbeg + ks * 16;
                                M->mseq[n][0] = (uint32_t)(k * 128 + r * gb);
                                M->mseq[n][1] = (uint32_t)((k0 >> 6) * 16384 + (k0 & 63) * 2);
                                M->mseq[n][2] = (uint32_t)(p * bsz + (g == 128 ? (k0 >> 6) * 16384 : 0) +
                                                           (r * gb) * 128 + (k0 & 63) * 2);
                                M->mseq[n][3] = (p > 0 || ks > 0) ? 1u : 0u;
                            }
                        }
            }
            uint32_t q_d[kMmaPerTile], q_a[kMmaPerTile], q_b[kMmaPerTile], q_acc = 0;
#pragma unroll
            for (int q = 0; q < kMmaPerTile; q++) {
                q_d[q] = M->mseq[q][0];
                q_a[q] = M->mseq[q][1] >> 4;
                q_b[q] = M->mseq[q][2] >> 4;
                q_acc |= M->mseq[q][3] << q;
            }
            const uint64_t bdesc = sdesc_sw128(smem_u32(bsplit));
            int64_t cur = -1;
            int committed = 0;
            tc::TileIter it;
            it.init(a, S, t_begin);
            if (nseq != kMmaPerTile) *abort_flag = 1;  // unreachable for the eligible shapes
            for (int i = 0; i < my_tiles && nseq == kMmaPerTile; i++, it.step(a, 1)) {
                const tc::TileInfo ti = it.info(a);
                const int64_t ls = ti.seg - seg0;
                bool ok = true;
                if (ti.seg != cur) {
                    ok = mbar_wait(&M->gready[ls & 3], (ls >> 2) & 1, abort_flag, a.wait_ns);
                    cur = ti.seg;
                }
                const int ab = i & 1, buf = i & 1;
                ok = ok && mbar_wait(&M->afull[ab], (i >> 1) & 1, abort_flag, a.wait_ns);
                ok = ok && mbar_wait(&M->accempty[buf], ((i >> 1) & 1) ^ 1, abort_flag, a.wait_ns);
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
                tc_fence_after();
                const uint64_t adesc = sdesc_sw128(smem_u32(atiles + ab * kATile));
                const uint32_t d_base = tmem + buf * acc_cols;
#pragma unroll
                for (int q = 0; q < kMmaPerTile; q++)
                    mma_bf16(d_base + q_d[q], adesc + q_a[q], bdesc + q_b[q], idesc, (q_acc >> q) & 1u);
                mma_commit(&M->accfull[buf]);
                mma_commit(&M->aempty[ab]);
                const bool last_of_seg = (i + 1 == my_tiles) || it.seg_last(a);
                if (last_of_seg) mma_commit(&M->bfree);
                committed = i + 1;
            }
            if (*abort_flag && committed > 0) {
                const int zero = 0;
                const int i = committed - 1;
                mbar_wait(&M->accfull[i & 1], (i >> 1) & 1, &zero, kWaitLimitNs);
            }
        }
    } else if (warp < 6) {
        // ------------------------------------------------------------ unpackers / gauge
        const int uw = warp - 2;
        const int row = uw * 32 + lane;
        int64_t cur = -1;
        int nconv = 0;
        tc::TileIter it;
        it.init(a, S, t_begin);
        for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
            const tc::TileInfo ti = it.info(a);
            if (ti.seg != cur) {
                const int64_t ls = ti.seg - seg0;
                if (nconv > 0) {
                    // the MMAs of the previous gauge set must be done with B
                    const bool ok = mbar_wait(&M->bfree, (nconv - 1) & 1, abort_flag, a.wait_ns);
                    if (!__all_sync(0xffffffffu, ok)) {
                        *abort_flag = 1;
                        break;
                    }
                }
                // B[n][k] = G_r[k - r g][n - r g]: thread `row` builds output channel n = row
                const int n = row, r = n / g, i_in = n - r * g;
                const float* Gc = a.G + tc::gauge_set(a, ti) * (int64_t)kD * g + (int64_t)r * g * g + i_in;
                // c_k: the split's (hi + lo) values summed by a pairwise tree over each step's
                // eight, the step sums accumulated with compensation (Neumaier), so c_k is within
                // a few u of its value (fp64 arithmetic is far slower on this part)
                float cs0 = 0.0f, ce0 = 0.0f, cs1 = 0.0f, ce1 = 0.0f;
                auto kadd = [](float& sum, float& comp, float v) {
                    const float t = sum + v;
                    comp += fabsf(sum) >= fabsf(v) ? (sum - t) + v : (v - t) + sum;
                    sum = t;
                };
                float tv[8];
                // eight gauge values per step; the next step's loads are in flight while this
                // step converts (a gauge change stalls the MMAs until it is done)
                float nv[8];
#pragma unroll
                for (int e = 0; e < 8; e++) nv[e] = __ldg(Gc + (int64_t)e * g);
                for (int j = 0; j < g; j += 8) {
                    float cv[8];
#pragma unroll
                    for (int e = 0; e < 8; e++) cv[e] = nv[e];
                    if (j + 8 < g) {
#pragma unroll
                        for (int e = 0; e < 8; e++) nv[e] = __ldg(Gc + (int64_t)(j + 8 + e) * g);
                    }
                    uint32_t hi[4], lo[4];
#pragma unroll
                    for (int e = 0; e < 8; e += 2) {
                        // both values to bf16 in one conversion (round to nearest even)
                        const __nv_bfloat162 h = __float22bfloat162_rn(make_float2(cv[e], cv[e + 1]));
                        const float2 hf = __bfloat1622float2(h);
                        const __nv_bfloat162 l = __float22bfloat162_rn(make_float2(cv[e] - hf.x, cv[e + 1] - hf.y));
                        const float2 lf = __bfloat1622float2(l);
                        hi[e >> 1] = *reinterpret_cast<const uint32_t*>(&h);
                        lo[e >> 1] = *reinterpret_cast<const uint32_t*>(&l);
                        tv[e] = hf.x + lf.x;  // exact
                        tv[e + 1] = hf.y + lf.y;
                    }
                    const float t8 = ((tv[0] + tv[1]) + (tv[2] + tv[3])) + ((tv[4] + tv[5]) + (tv[6] + tv[7]));
                    // blk is a multiple of 8, so the eight values of a step share a sub-block
                    if (nsub > 1 && j >= blk) kadd(cs1, ce1, t8);
                    else kadd(cs0, ce0, t8);
                    const int k = r * g + j;
                    unsigned char* reg1 = bsplit + 1 * bsz + (g == 128 ? (k >> 6) * 16384 : 0);
                    unsigned char* reg0 = bsplit + 0 * bsz + (g == 128 ? (k >> 6) * 16384 : 0);
                    *reinterpret_cast<uint4*>(reg1 + sw128_offset(n, k & 63)) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                    *reinterpret_cast<uint4*>(reg0 + sw128_offset(n, k & 63)) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
                }
                float* cb = csum + (ls & 3) * 2 * kD;
                cb[n] = cs0 + ce0;
                cb[kD + n] = cs1 + ce1;
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&M->gready[ls & 3]);
                cur = ti.seg;
                nconv++;
            }
            const int st = i % kCStages, ab = i & 1;
            bool ok = mbar_wait(&M->cfull[st], (i / kCStages) & 1, abort_flag, a.wait_ns);
            ok = ok && mbar_wait(&M->aempty[ab], ((i >> 1) & 1) ^ 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            const uint4* src = reinterpret_cast<const uint4*>(cst + st * kCStageBytes + row * kRowBytes);
            uint32_t w[4 * BITS + 1];
#pragma unroll
            for (int q = 0; q < BITS; q++) {
                const uint4 v = src[q];
                w[4 * q] = v.x;
                w[4 * q + 1] = v.y;
                w[4 * q + 2] = v.z;
                w[4 * q + 3] = v.w;
            }
            w[4 * BITS] = 0;
            uint4 outc[16];
            unpack_row<BITS>(w, outc);
            unsigned char* at = atiles + ab * kATile;
#pragma unroll
            for (int c = 0; c < 16; c++)
                *reinterpret_cast<uint4*>(at + (c >> 3) * 16384 + row * 128 + (((c & 7) ^ (row & 7)) << 4)) = outc[c];
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&M->afull[ab]);
                mbar_arrive(&M->cempty[st]);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int ew = warp - kEpiWarp0;  // 0..7
        const int half = ew >> 2;         // output columns 64*half .. 64*half + 63
        const int q4 = warp & 3;          // TMEM lane quadrant of this warp
        const int row = q4 * 32 + lane;
        const int nbk = kD / blk;
        unsigned char* ost = sm + SL::ostage + ew * kOutWarpBytes;
        tc::TileIter it;
        it.init(a, S, t_begin);
        // block scales of this thread's row, loaded one tile ahead
        uint32_t sz_next[4] = {0, 0, 0, 0};
        auto load_scales = [&](const tc::TileInfo& t, uint32_t (&dst)[4]) {
            if (row < t.rows_valid) {
                const uint32_t* sp = a.scales + a.smap.at(t.l, t.s, t.b, t.h, t.t0 + row);
#pragma unroll
                for (int bk = 0; bk < 4; bk++)
                    if (bk < nbk) dst[bk] = __ldg(sp + bk);
            }
        };
        if (my_tiles > 0) load_scales(it.info(a), sz_next);
        for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
            const tc::TileInfo ti = it.info(a);
            const int64_t ls = ti.seg - seg0;
            const int buf = i & 1;
            uint32_t sz[4];
#pragma unroll
            for (int q = 0; q < 4; q++) sz[q] = sz_next[q];
            if (i + 1 < my_tiles) {
                tc::TileIter nx = it;
                nx.step(a, 1);
                load_scales(nx.info(a), sz_next);
            }
            bool ok = mbar_wait(&M->accfull[buf], (i >> 1) & 1, abort_flag, a.wait_ns);
            ok = ok && mbar_wait(&M->gready[ls & 3], (ls >> 2) & 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            const bool valid = row < ti.rows_valid;
            // the warp's 32 rows all exist: staged and written by one TMA store; else the
            // valid rows are stored directly
            const bool whole = q4 * 32 + 32 <= ti.rows_valid;
            const float* cb = csum + (ls & 3) * 2 * kD;
            const uint32_t tacc = tmem + ((uint32_t)(q4 * 32) << 16) + buf * acc_cols;
            const int64_t row0 = tc::dense_row(a, ti) + q4 * 32;  // first row of this warp
            uint4* orow = reinterpret_cast<uint4*>(a.out + (row0 + lane) * kD);
            // the previous TMA store of this warp has finished reading the staging block
            if (lane == 0) bulk_wait_read<0>();
            __syncwarp();
            auto chunk = [&](int cc, const uint32_t (&d0)[32], const uint32_t (&d1)[32]) {
                const int c = 2 * half + cc;  // 32-column chunk of the tile
                // gauge group r = 32c / g (g >= 32) or several (g < 32, then nsub = 1)
                const int r = (c * 32) / g;
                float sk[2], ak[2];
#pragma unroll
                for (int k = 0; k < 2; k++) {
                    const int bk = nsub > 1 ? (r * g + k * blk) / blk : (c * 32) / blk;
                    uint32_t v = 0;
#pragma unroll
                    for (int q = 0; q < 4; q++)
                        if (q == bk) v = sz[q];
                    const float s = __half2float(__ushort_as_half((unsigned short)(v & 0xffffu)));
                    const float m = __half2float(__ushort_as_half((unsigned short)(v >> 16)));
                    sk[k] = s;
                    ak[k] = m - kOff * s;
                }
                uint32_t o[16];
                // the same multiply and fused multiply-adds per value, two columns per instruction
                const float2 s0 = make_float2(sk[0], sk[0]), a0 = make_float2(ak[0], ak[0]);
                const float2 s1 = make_float2(sk[1], sk[1]), a1 = make_float2(ak[1], ak[1]);
#pragma unroll
                for (int e = 0; e < 32; e += 4) {
                    const float4 c0 = *reinterpret_cast<const float4*>(cb + c * 32 + e);
                    float2 x01 = __ffma2_rn(s0, make_float2(__uint_as_float(d0[e]), __uint_as_float(d0[e + 1])),
                                            __fmul2_rn(a0, make_float2(c0.x, c0.y)));
                    float2 x23 = __ffma2_rn(s0, make_float2(__uint_as_float(d0[e + 2]), __uint_as_float(d0[e + 3])),
                                            __fmul2_rn(a0, make_float2(c0.z, c0.w)));
                    if (nsub > 1) {
                        const float4 c1 = *reinterpret_cast<const float4*>(cb + kD + c * 32 + e);
                        x01 = __ffma2_rn(s1, make_float2(__uint_as_float(d1[e]), __uint_as_float(d1[e + 1])),
                                         __ffma2_rn(a1, make_float2(c1.x, c1.y), x01));
                        x23 = __ffma2_rn(s1, make_float2(__uint_as_float(d1[e + 2]), __uint_as_float(d1[e + 3])),
                                         __ffma2_rn(a1, make_float2(c1.z, c1.w), x23));
                    }
                    const __nv_bfloat162 b0 = __floats2bfloat162_rn(x01.x, x01.y);
                    const __nv_bfloat162 b1 = __floats2bfloat162_rn(x23.x, x23.y);
                    o[e >> 1] = *reinterpret_cast<const uint32_t*>(&b0);
                    o[(e >> 1) + 1] = *reinterpret_cast<const uint32_t*>(&b1);
                }
                if (whole) {
                    // row `lane` of the warp's 32 x 128 B block; 16-byte unit u at u ^ (lane & 7)
#pragma unroll
                    for (int q = 0; q < 4; q++) {
                        const int u = cc * 4 + q;
                        *reinterpret_cast<uint4*>(ost + lane * 128 + ((u ^ (lane & 7)) << 4)) =
                            make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                    }
                } else if (valid) {
#pragma unroll
                    for (int q = 0; q < 4; q++)
                        orow[c * 4 + q] = make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
                }
            };
            auto release = [&]() {
                // everything this warp needs from the buffer is in registers
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&M->accempty[buf]);
            };
            if (nsub == 1) {
                // both chunks in flight before the single wait
                uint32_t da[32], db[32];
                tmem_ld32(tacc + (2 * half) * 32, da);
                tmem_ld32(tacc + (2 * half + 1) * 32, db);
                tmem_wait_ld();
                release();
                chunk(0, da, da);
                chunk(1, db, db);
            } else {
#pragma unroll
                for (int cc = 0; cc < 2; cc++) {
                    uint32_t d0[32], d1[32];
                    tmem_ld32(tacc + (2 * half + cc) * 32, d0);
                    tmem_ld32(tacc + 128 + (2 * half + cc) * 32, d1);
                    tmem_wait_ld();
                    if (cc == 1) release();
                    chunk(cc, d0, d1);
                }
            }
            if (whole) {
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&omap, ost, 64 * half, (int)row0);
                    bulk_commit();
                }
            }
        }
        if (lane == 0) bulk_wait<0>();
    }
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) raise_flag(a.status, CG_FLAG_PIPE_TIMEOUT);
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, 2 * acc_cols);
    }
}

template <int BITS, int NSUB>
cudaError_t launch_dec_ns(const DecParams& P, const CUtensorMap& omap, cudaStream_t st) {
    const size_t smem = DecSmem<BITS>::total + 1024;
    cudaError_t e =
        cudaFuncSetAttribute(tc_decode_kernel<BITS, NSUB>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = P.S.n_tiles < tc::num_sms() ? P.S.n_tiles : tc::num_sms();
    tc_decode_kernel<BITS, NSUB><<<(unsigned)grid, kThreads, smem, st>>>(omap, P);
    return cudaGetLastError();
}

template <int BITS>
cudaError_t launch_dec(const DecParams& P, const CUtensorMap& omap, cudaStream_t st) {
    return P.nsub > 1 ? launch_dec_ns<BITS, 2>(P, omap, st) : launch_dec_ns<BITS, 1>(P, omap, st);
}

}  // namespace

bool tc_row_decode_eligible(const RowArgs& a) {
    if (a.d != kD || a.none_mode) return false;
    if (!(a.blk == 32 || a.blk == 64 || a.blk == 128)) return false;
    if (a.blk < a.g && a.g / a.blk > 2) return false;
    if (a.t_count < 64) return false;
    if ((reinterpret_cast<uintptr_t>(a.codes) & 15u) || (reinterpret_cast<uintptr_t>(a.out) & 15u)) return false;
    const int64_t rows = (int64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (rows + 128 >= (int64_t)1 << 31) return false;
    return tmap_encode_fn() != nullptr;
}

cudaError_t tc_launch_row_decode(const RowArgs& a, cudaStream_t st) {
    DecParams P;
    P.a = a;
    P.S = tc::make_sched(a);
    P.nsub = a.blk < a.g ? a.g / a.blk : 1;
    if (P.S.n_tiles == 0) return cudaSuccess;
    // output rows [L][2][B][H][T_x] of 128 bf16, written in 32-row x 64-column boxes
    CUtensorMap omap;
    const uint64_t rows = (uint64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (!make_tmap_bf16_sw128(&omap, a.out, rows, kD, kD * 2, 32)) return cudaErrorInvalidValue;
    switch (a.bits) {
        case 2: return launch_dec<2>(P, omap, st);
        case 3: return launch_dec<3>(P, omap, st);
        case 4: return launch_dec<4>(P, omap, st);
        case 6: return launch_dec<6>(P, omap, st);
        case 8: return launch_dec<8>(P, omap, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace cg
