// cg_tc_keydec.cu -- tensor-core decode of KIVI keys (Sec. 4.3: per-channel key ranges over
// a token group; Sec. 3: Xhat = G^T Zhat), head dim d = 128, key groups of 128 tokens.
//
// A key group stores, per gauge-space channel, a stream of 128 token codes with one scale
// and zero, so the scale varies along the contraction index of Xhat = G^T Zhat and cannot
// be applied after the MMA. The unpackers therefore dequantize, zhat = q s + m in fp32, and
// write zhat as two bf16 terms (hi + lo, 16 significant bits) into an A tile that the MMA
// reads MN-major (tokens contiguous per channel, as the code streams are), so a thread
// stores 8 tokens of its channel at a time;
// D[token][i] = sum_j A[token][j] B[i][j] with B = G^T (two bf16 terms) takes three MMA
// passes (hi·hi, hi·lo, lo·hi; the lo·lo term is below 2^-16 relative).
//
// Persistent warp-specialized kernel, one CTA per SM, 14 warps:
//   warp 0      bulk copy of a group's code streams (128 x 16*bits bytes) and its 128 scales;
//   warp 1      MMA issuer (24 MMAs per tile, each one gauge group wide, fp32 accumulators,
//               two TMEM buffers);
//   warps 2..9  one gauge-space channel and 64 of its tokens per thread (warps 2..5 the
//               first 64 tokens, 6..9 the others): unpack, dequantize, split, store that
//               part of the channel's K-row of the A tile; at a gauge change warps 2..5
//               build G^T's split (full K for g = 128; for smaller groups the diagonal
//               blocks packed into one 64-column tile, one MMA chain per group);
//   warps 10..13 one token row per thread: accumulator -> bf16 -> global.
#include <cuda_bf16.h>

#include "cg_sm100.cuh"
#include "cg_tc.h"
#include "cg_tc_common.cuh"

namespace cg {
namespace {

using namespace sm100;
using tc::kD;
using tc::kWaitLimitNs;

constexpr int kThreads = 448;
constexpr int kEpiWarp0 = 10;
constexpr int kATerm = 128 * kD * 2;  // one bf16 term of a 128 x 128 tile
constexpr int kAStages = 2;
constexpr int kSegBufs = 4;
constexpr int kMma = 3 * 8;           // 3 term pairs x K = 128 in steps of 16

template <int BITS>
struct KdSmem {
    static constexpr int cstages_n = BITS >= 4 ? 2 : 4;
    static constexpr uint32_t cstage_bytes = 128u * 16u * BITS + 512u;  // streams + scales
    static constexpr uint32_t a_tiles = 0;                              // kAStages x 2 terms
    static constexpr uint32_t bsplit = a_tiles + kAStages * 2 * kATerm;  // 2 terms x 32 KB
    static constexpr uint32_t cstages = bsplit + 2 * 32768;
    static constexpr uint32_t misc = cstages + cstages_n * cstage_bytes;
    static constexpr uint32_t total = misc + 512;
    static_assert(cstage_bytes % 16 == 0, "bulk copy sizes are multiples of 16 bytes");
    static_assert(total + 1024 <= 232448, "shared memory budget");
};

struct KdMisc {
    uint64_t cfull[4], cempty[4];
    uint64_t afull[kAStages], aempty[kAStages];
    uint64_t accfull[2], accempty[2];
    uint64_t gready[kSegBufs];
    uint64_t bfree;
    uint32_t tmem_slot;
    int abort_flag;
};
static_assert(sizeof(KdMisc) <= 512, "misc block");

struct KdParams {
    RowArgs a;
    tc::Sched S;
};

template <int BITS>
__global__ void __launch_bounds__(kThreads, 1) tc_key_decode_kernel(const KdParams P) {
    using SL = KdSmem<BITS>;
    constexpr int kCStages = SL::cstages_n;
    constexpr uint32_t kCStageBytes = SL::cstage_bytes;
    constexpr uint32_t kStreamBytes = 16u * BITS;  // one channel's 128 codes
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const uint32_t base_u32 = (smem_u32(smem_raw) + 1023u) & ~1023u;
    unsigned char* sm = smem_raw + (base_u32 - smem_u32(smem_raw));
    KdMisc* M = reinterpret_cast<KdMisc*>(sm + SL::misc);
    unsigned char* atiles = sm + SL::a_tiles;
    unsigned char* bsplit = sm + SL::bsplit;
    unsigned char* cst = sm + SL::cstages;

    const RowArgs& a = P.a;
    const tc::Sched& S = P.S;
    const int g = a.g;
    const int gb = g < 16 ? 16 : g;  // MMA width: one gauge group (two for g = 8)
    // G^T split: full K for g = 128, else the groups' diagonal blocks packed into one
    // 64-column tile per term (rows of a group at its own channels)
    const uint32_t bsz = g == 128 ? 32768u : 16384u;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int64_t t_begin = S.n_tiles * blockIdx.x / gridDim.x;
    const int64_t t_end = S.n_tiles * (blockIdx.x + 1) / gridDim.x;
    const int my_tiles = (int)(t_end - t_begin);
    const int64_t seg0 = my_tiles > 0 ? tc::tile_info(a, S, t_begin).seg : 0;

    if (threadIdx.x == 0) {
        for (int i = 0; i < kCStages; i++) {
            mbar_init(&M->cfull[i], 1);
            mbar_init(&M->cempty[i], 8);
        }
        for (int i = 0; i < kAStages; i++) {
            mbar_init(&M->afull[i], 8);
            mbar_init(&M->aempty[i], 1);
        }
        for (int i = 0; i < 2; i++) {
            mbar_init(&M->accfull[i], 1);
            mbar_init(&M->accempty[i], 4);
        }
        for (int i = 0; i < kSegBufs; i++) mbar_init(&M->gready[i], 4);
        mbar_init(&M->bfree, 1);
        M->abort_flag = 0;
        fence_barrier_init();
    }
    // G^T's split: off-diagonal blocks stay zero for the whole launch
    for (uint32_t i = threadIdx.x; i < 2u * 32768u / 16u; i += kThreads)
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
        // ------------------------------------------------------------ code/scale producer
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
                unsigned char* dst = cst + st * kCStageBytes;
                mbar_arrive_expect_tx(&M->cfull[st], 128u * kStreamBytes + 512u);
                bulk_load(dst, a.codes + a.cmap.at(ti.l, ti.s, ti.b, ti.h, ti.t0), 128u * kStreamBytes, &M->cfull[st]);
                bulk_load(dst + 128u * kStreamBytes, a.scales + a.smap.at(ti.l, ti.s, ti.b, ti.h, ti.t0), 512u,
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
            const uint32_t idesc = idesc_bf16_f32(128, gb) | kIdescAMnMajor;  // A read MN-major
            const uint64_t bdesc = sdesc_sw128(smem_u32(bsplit));
            // the tile's 24 MMAs (3 term pairs x 8 K-steps of 16 over the groups): D column,
            // A and B byte offsets (in 16-byte units), accumulate bits
            uint32_t q_d[kMma], q_a[kMma], q_b[kMma], q_acc = 0;
#pragma unroll
            for (int q = 0; q < kMma; q++) {
                const int pair = q >> 3, qq = q & 7;  // pairs: (A hi, B hi), (A hi, B lo), (A lo, B hi)
                const uint32_t ta = pair == 2 ? 1u : 0u, tb = pair == 1 ? 1u : 0u;
                const int per = gb >> 4;  // K-steps per group
                const int r = qq / per, ks = qq - r * per;
                const int k0 = r * gb + ks * 16;
                q_d[q] = (uint32_t)(r * gb);
                q_a[q] = (ta * kATerm + (uint32_t)((k0 >> 3) * 1024)) >> 4;  // K-step: two 8-channel atoms
                q_b[q] = (tb * bsz + (uint32_t)((g == 128 ? (k0 >> 6) * 16384 : r * gb * 128) + (k0 & 63) * 2)) >> 4;
                q_acc |= (pair > 0 || ks > 0 ? 1u : 0u) << q;
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
                const int ab = i % kAStages, buf = i & 1;
                ok = ok && mbar_wait(&M->afull[ab], (i / kAStages) & 1, abort_flag, a.wait_ns);
                ok = ok && mbar_wait(&M->accempty[buf], ((i >> 1) & 1) ^ 1, abort_flag, a.wait_ns);
                if (!ok) {
                    *abort_flag = 1;
                    break;
                }
                tc_fence_after();
                const uint64_t adesc = sdesc_sw128_mn(smem_u32(atiles + ab * 2 * kATerm), 16384u, 1024u);
                const uint32_t d_base = tmem + buf * 128;
#pragma unroll
                for (int q = 0; q < kMma; q++)
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
    } else if (warp < kEpiWarp0) {
        // ------------------------------------------------------------ unpack + dequantize
        const int ch = ((warp - 2) & 3) * 32 + lane;  // gauge-space channel of this thread
        const int half = (warp - 2) >> 2;             // its tokens: 64 half .. 64 half + 63
        int64_t cur = -1;
        int nconv = 0;
        tc::TileIter it;
        it.init(a, S, t_begin);
        for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
            const tc::TileInfo ti = it.info(a);
            if (ti.seg != cur && half == 0) {
                const int64_t ls = ti.seg - seg0;
                if (nconv > 0) {
                    const bool ok = mbar_wait(&M->bfree, (nconv - 1) & 1, abort_flag, a.wait_ns);
                    if (!__all_sync(0xffffffffu, ok)) {
                        *abort_flag = 1;
                        break;
                    }
                }
                // B[n][k] = G_r[k - r g][n - r g] (n, k in group r): thread builds row n = ch
                const int n = ch, r = n / g, i_in = n - r * g;
                const float* Gc = a.G + tc::gauge_set(a, ti) * (int64_t)kD * g + (int64_t)r * g * g + i_in;
                for (int j = 0; j < g; j += 8) {
                    uint32_t hi[4], lo[4];
#pragma unroll
                    for (int e = 0; e < 8; e += 2) {
                        const float v0 = __ldg(Gc + (int64_t)(j + e) * g);
                        const float v1 = __ldg(Gc + (int64_t)(j + e + 1) * g);
                        const __nv_bfloat16 h0 = __float2bfloat16_rn(v0), h1 = __float2bfloat16_rn(v1);
                        const __nv_bfloat16 l0 = __float2bfloat16_rn(v0 - __bfloat162float(h0));
                        const __nv_bfloat16 l1 = __float2bfloat16_rn(v1 - __bfloat162float(h1));
                        hi[e >> 1] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
                        lo[e >> 1] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
                    }
                    const int k = r * g + j;
                    const uint32_t off = (g == 128 ? (k >> 6) * 16384 : 0) + sw128_offset(n, k & 63);
                    *reinterpret_cast<uint4*>(bsplit + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                    *reinterpret_cast<uint4*>(bsplit + bsz + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&M->gready[ls & 3]);
                cur = ti.seg;
                nconv++;
            }
            const int st = i % kCStages, ab = i % kAStages;
            bool ok = mbar_wait(&M->cfull[st], (i / kCStages) & 1, abort_flag, a.wait_ns);
            ok = ok && mbar_wait(&M->aempty[ab], ((i / kAStages) & 1) ^ 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            const unsigned char* stage = cst + st * kCStageBytes;
            // this thread's 64 codes: 8 * BITS bytes of the channel stream
            uint32_t w[2 * BITS + 1];
#pragma unroll
            for (int q = 0; q < BITS; q++) {
                const uint2 v = reinterpret_cast<const uint2*>(stage + ch * kStreamBytes + half * 8 * BITS)[q];
                w[2 * q] = v.x;
                w[2 * q + 1] = v.y;
            }
            w[2 * BITS] = 0;
            const uint32_t sz = reinterpret_cast<const uint32_t*>(stage + 128u * kStreamBytes)[ch];
            const float s = __half2float(__ushort_as_half((unsigned short)(sz & 0xffffu)));
            const float m = __half2float(__ushort_as_half((unsigned short)(sz >> 16)));
            // MN-major A tile: channel ch is K-row (ch & 7) of atom (half, ch >> 3); its 64 tokens
            // are 8 chunks of 8 (16 bytes), chunk c stored at position c ^ (ch & 7)
            unsigned char* ahi = atiles + ab * 2 * kATerm + half * 16384 + (ch >> 3) * 1024 + (ch & 7) * 128;
            unsigned char* alo = ahi + kATerm;
#pragma unroll
            for (int c = 0; c < 8; c++) {
                uint32_t hi[4], lo[4];
#pragma unroll
                for (int e = 0; e < 4; e++) {
                    // q as fp32 without an integer conversion: 2^23 + q has q in its low
                    // mantissa bits, and subtracting 2^23 is exact
                    uint32_t qb[2];
#pragma unroll
                    for (int u = 0; u < 2; u++) {
                        const int t = 8 * c + 2 * e + u;
                        const int p = t * BITS;
                        uint32_t v = w[p >> 5] >> (p & 31);
                        if ((p & 31) + BITS > 32) v |= w[(p >> 5) + 1] << (32 - (p & 31));
                        qb[u] = (v & ((1u << BITS) - 1u)) | 0x4B000000u;
                    }
                    const float2 qf = __fadd2_rn(make_float2(__uint_as_float(qb[0]), __uint_as_float(qb[1])),
                                                 make_float2(-8388608.0f, -8388608.0f));
                    const float2 z2 = __ffma2_rn(qf, make_float2(s, s), make_float2(m, m));  // q s + m
                    const __nv_bfloat162 h2 = __floats2bfloat162_rn(z2.x, z2.y);
                    const float2 hf = __bfloat1622float2(h2);
                    const float2 r2 = __fadd2_rn(z2, make_float2(-hf.x, -hf.y));  // exact
                    const __nv_bfloat162 l2 = __floats2bfloat162_rn(r2.x, r2.y);
                    hi[e] = *reinterpret_cast<const uint32_t*>(&h2);
                    lo[e] = *reinterpret_cast<const uint32_t*>(&l2);
                }
                const uint32_t o = (uint32_t)((c ^ (ch & 7)) << 4);
                *reinterpret_cast<uint4*>(ahi + o) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4*>(alo + o) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(&M->afull[ab]);
                mbar_arrive(&M->cempty[st]);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int q4 = warp & 3;
        const int row = q4 * 32 + lane;  // token of the group
        tc::TileIter it;
        it.init(a, S, t_begin);
        for (int i = 0; i < my_tiles; i++, it.step(a, 1)) {
            const tc::TileInfo ti = it.info(a);
            const int buf = i & 1;
            const bool ok = mbar_wait(&M->accfull[buf], (i >> 1) & 1, abort_flag, a.wait_ns);
            if (!__all_sync(0xffffffffu, ok)) {
                *abort_flag = 1;
                break;
            }
            tc_fence_after();
            const uint32_t tacc = tmem + ((uint32_t)(q4 * 32) << 16) + buf * 128;
            uint4* orow = reinterpret_cast<uint4*>(a.out + (tc::dense_row(a, ti) + row) * kD);
#pragma unroll 1
            for (int c = 0; c < 4; c++) {
                uint32_t v[32];
                tmem_ld32(tacc + c * 32, v);
                tmem_wait_ld();
                if (c == 3) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&M->accempty[buf]);
                }
                uint32_t o[16];
#pragma unroll
                for (int e = 0; e < 16; e++) {
                    const __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(v[2 * e]), __uint_as_float(v[2 * e + 1]));
                    o[e] = *reinterpret_cast<const uint32_t*>(&b2);
                }
#pragma unroll
                for (int q = 0; q < 4; q++) orow[c * 4 + q] = make_uint4(o[4 * q], o[4 * q + 1], o[4 * q + 2], o[4 * q + 3]);
            }
        }
    }
    __syncthreads();
    if (*abort_flag && threadIdx.x == 0) raise_flag(a.status, CG_FLAG_PIPE_TIMEOUT);
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem, 256);
    }
}

template <int BITS>
cudaError_t launch_kd(const KdParams& P, cudaStream_t st) {
    const size_t smem = KdSmem<BITS>::total + 1024;
    cudaError_t e =
        cudaFuncSetAttribute(tc_key_decode_kernel<BITS>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int64_t grid = P.S.n_tiles < tc::num_sms() ? P.S.n_tiles : tc::num_sms();
    tc_key_decode_kernel<BITS><<<(unsigned)grid, kThreads, smem, st>>>(P);
    return cudaGetLastError();
}

}  // namespace

// KIVI keys as rows of the key tensor (s = 0, t_count = the quantized tokens, whole
// 128-token groups); cmap/smap address a group's first channel stream and scale.
bool tc_key_decode_eligible(const RowArgs& a) {
    if (a.d != kD || a.blk != 128) return false;
    if (a.t_count < 128 || a.t_count % 128) return false;
    const int64_t rows = (int64_t)a.L * 2 * a.B * a.H * a.T_x;
    if (rows + 128 >= (int64_t)1 << 31) return false;
    if ((reinterpret_cast<uintptr_t>(a.codes) & 15u) || (reinterpret_cast<uintptr_t>(a.scales) & 15u) ||
        (reinterpret_cast<uintptr_t>(a.out) & 15u))
        return false;
    return true;
}

cudaError_t tc_launch_key_decode(const RowArgs& a, cudaStream_t st) {
    KdParams P;
    P.a = a;
    P.S = tc::make_sched(a);
    if (P.S.n_tiles == 0) return cudaSuccess;
    switch (a.bits) {
        case 2: return launch_kd<2>(P, st);
        case 3: return launch_kd<3>(P, st);
        case 4: return launch_kd<4>(P, st);
        case 6: return launch_kd<6>(P, st);
        case 8: return launch_kd<8>(P, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace cg
