// cg_attn.cu -- attention of one decoding query per sequence, straight from the packed codes of
// a block-uniform cache: the recovered cache of Sec. 3 consumed by softmax attention (Fig. 1),
// with the inverse gauge folded out of the token loop (Sec. 3 notes that recovery can be folded
// into the surrounding computation).
//
// For KV head h and one of its n_rep query heads (grouped queries):
//   scores  q . khat_t = q . (G_K^T zhat_t) = (G_K q) . zhat_t: the query is rotated once into
//           gauge space and dotted with the dequantized codes;
//   values  sum_t p_t vhat_t = G_V^T (sum_t p_t zhat_t): the weighted sum stays in gauge space
//           and is rotated once per query at the end.
// The token loop reads only codes and scales (no bf16 cache is written or read).
//
// A b-bit code q enters the fp32 arithmetic as f = 1 + q 2^-b (bit pattern 0x3F800000 | q << (23-b),
// two integer operations, exact), so sum_c w_c q_c = 2^b (sum_c w_c f_c - sum_c w_c).
//
// Kernels: attn_query_kernel (q' = scale * G_K q); a chunk kernel that writes, per (l, b, h) and
// part, the part's softmax max, sum and gauge-space weighted value sum (attn_chunk_mma_kernel for
// 2- and 4-bit codes: many 128-token chunks per CTA, codes staged by bulk copies one chunk ahead,
// online softmax; attn_chunk_kernel for 3-, 6- and 8-bit codes: one chunk per CTA, all on CUDA
// cores); attn_combine_kernel (merges the parts, applies G_V^T).
#include "cg_launch.h"
#include "cg_sm100.cuh"
#include "cg_tc_common.cuh"

namespace cg {
namespace {

using namespace sm100;

constexpr int kAD = 128;           // head dim served
constexpr int kAThreads = 256;
constexpr int kASlices = kAThreads / 16;  // value phase: 16 channel octets x 16 token slices

// f = 1 + code * 2^-BITS for code c of a row held in registers (c known at compile time).
template <int BITS>
__device__ __forceinline__ float code_f(const uint32_t* w, int c) {
    const int bit = c * BITS, wi = bit >> 5, sh = bit & 31;
    uint32_t v = w[wi] >> sh;
    if (sh + BITS > 32) v |= w[wi + 1] << (32 - sh);
    return __uint_as_float(0x3F800000u | ((v & ((1u << BITS) - 1u)) << (23 - BITS)));
}

__device__ __forceinline__ float half_lo(uint32_t v) { return h2f_bits(v & 0xffffu); }
__device__ __forceinline__ float half_hi(uint32_t v) { return h2f_bits(v >> 16); }

constexpr int kQuerySeqs = 4;  // sequences per CTA of the query rotation

// q' = scale * G_K q for the query heads of kQuerySeqs sequences of one (l, h); G_K transposed
// in shared memory.
__global__ void __launch_bounds__(kAD) attn_query_kernel(AttnArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    const int g = a.g;
    float* Gt = reinterpret_cast<float*>(smem);  // Gt[r][j][i] = G_r[i][j]
    float* qs = Gt + kAD * g;                    // one query vector
    const int l = blockIdx.x / a.H, h = blockIdx.x % a.H, c = threadIdx.x;
    const float* Gsrc = a.G + ((int64_t)(l * 2 + 0) * a.H + h) * (int64_t)kAD * g;
    for (int e = threadIdx.x; e < kAD * g; e += blockDim.x) {
        const int r = e / (g * g), rem = e - r * g * g, i = rem / g, j = rem - i * g;
        Gt[r * g * g + j * g + i] = __ldg(Gsrc + e);
    }
    const int grp = c / g, i = c - grp * g;
    const int b_hi = (blockIdx.y + 1) * kQuerySeqs < a.B ? (blockIdx.y + 1) * kQuerySeqs : a.B;
    for (int b = blockIdx.y * kQuerySeqs; b < b_hi; b++)
        for (int rq = 0; rq < a.n_rep; rq++) {
            const int64_t qi = ((((int64_t)l * a.B + b) * a.H + h) * a.n_rep + rq) * kAD;
            __syncthreads();
            qs[c] = bf16_bits_to_float(a.q[qi + c]);
            __syncthreads();
            const float* Gc = Gt + grp * g * g + i;
            const float* xq = qs + grp * g;
            float acc = 0.0f;
            for (int j = 0; j < g; j++) acc = fmaf(Gc[j * g], xq[j], acc);
            a.qrot[qi + c] = a.scale * acc;
        }
}

// Deterministic block reduction of NV values per thread (sum or max) over NT threads, result
// in out[NV].
template <int NV, bool MAX, int NT>
__device__ __forceinline__ void block_reduce_n(float (&v)[NV], float* scratch, float* out) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int k = 0; k < NV; k++)
        for (int off = 16; off >= 1; off >>= 1) {
            const float o = __shfl_xor_sync(0xffffffffu, v[k], off);
            v[k] = MAX ? fmaxf(v[k], o) : v[k] + o;
        }
    if (lane == 0)
#pragma unroll
        for (int k = 0; k < NV; k++) scratch[warp * NV + k] = v[k];
    __syncthreads();
    if (threadIdx.x < NV) {
        float r = scratch[threadIdx.x];
        for (int w = 1; w < NT / 32; w++) {
            const float o = scratch[w * NV + threadIdx.x];
            r = MAX ? fmaxf(r, o) : r + o;
        }
        out[threadIdx.x] = r;
    }
    __syncthreads();
}

template <int NV, bool MAX>
__device__ __forceinline__ void block_reduce(float (&v)[NV], float* scratch, float* out) {
    block_reduce_n<NV, MAX, kAThreads>(v, scratch, out);
}

template <int BITS, int NREP>
__global__ void __launch_bounds__(kAThreads) attn_chunk_kernel(AttnArgs a) {
    extern __shared__ __align__(16) unsigned char smem[];
    float* qs = reinterpret_cast<float*>(smem);                  // [NREP][128] q'
    float* c32 = qs + NREP * kAD;                                // [NREP][4] sums of q' per 32 channels
    float* mx = c32 + NREP * 4;                                  // [NREP] chunk max
    float* sm = mx + NREP;                                       // [NREP] chunk sum of exp
    float* Wr = sm + NREP;                                       // [NREP][4] sum_t p s_V per block
    float* Zr = Wr + NREP * 4;                                   // [NREP][4] sum_t p m_V per block
    float* scratch = Zr + NREP * 4;                              // [8 warps][NREP * 4]
    uint32_t* SV = reinterpret_cast<uint32_t*>(scratch + 8 * NREP * 4);  // [chunk][4] value scales
    float* P = reinterpret_cast<float*>(SV + kAttnChunk * 4);    // [NREP][chunk] scores, then p;
                                                                 // later [16][NREP][128] partial sums
    const int tid = threadIdx.x;
    const int unit = blockIdx.y;
    const int l = unit / (a.B * a.H), bh = unit - l * a.B * a.H, b = bh / a.H, h = bh - (bh / a.H) * a.H;
    const int64_t c0 = (int64_t)blockIdx.x * kAttnChunk;
    const int n_tok = a.T - c0 < kAttnChunk ? (int)(a.T - c0) : kAttnChunk;
    const int blk = a.blk, nb = kAD / blk;
    constexpr float kTwoB = (float)(1 << BITS);

    for (int e = tid; e < NREP * kAD; e += kAThreads) qs[e] = a.qrot[(int64_t)unit * NREP * kAD + e];
    __syncthreads();
    if (tid < NREP * 4) {
        const float* src = qs + (tid >> 2) * kAD + (tid & 3) * 32;
        float s = 0.0f;
        for (int k = 0; k < 32; k++) s += src[k];
        c32[tid] = s;
    }
    __syncthreads();

    // scores: one token per thread, its packed key row in registers
    for (int tt = tid; tt < n_tok; tt += kAThreads) {
        const int64_t t = c0 + tt;
        const uint4* row = reinterpret_cast<const uint4*>(a.codes + a.cmap.at(l, 0, b, h, t));
        uint32_t w[4 * BITS + 1];
#pragma unroll
        for (int k = 0; k < BITS; k++) {
            const uint4 v = __ldg(row + k);
            w[4 * k] = v.x;
            w[4 * k + 1] = v.y;
            w[4 * k + 2] = v.z;
            w[4 * k + 3] = v.w;
        }
        w[4 * BITS] = 0u;
        const uint32_t* sk = a.scales + a.smap.at(l, 0, b, h, t);
        uint32_t sz[4];
#pragma unroll
        for (int k = 0; k < 4; k++) sz[k] = k < nb ? __ldg(sk + k) : 0u;
        float acc[NREP][4];
#pragma unroll
        for (int r = 0; r < NREP; r++)
#pragma unroll
            for (int k = 0; k < 4; k++) acc[r][k] = 0.0f;
#pragma unroll
        for (int c = 0; c < kAD; c++) {
            const float f = code_f<BITS>(w, c);
#pragma unroll
            for (int r = 0; r < NREP; r++) acc[r][c >> 5] = fmaf(qs[r * kAD + c], f, acc[r][c >> 5]);
        }
#pragma unroll
        for (int r = 0; r < NREP; r++) {
            float s = 0.0f;
#pragma unroll
            for (int k = 0; k < 4; k++) {
                const uint32_t z = sz[(32 * k) / blk];
                s += half_lo(z) * kTwoB * (acc[r][k] - c32[r * 4 + k]) + half_hi(z) * c32[r * 4 + k];
            }
            P[r * kAttnChunk + tt] = s;
        }
    }
    __syncthreads();

    // chunk softmax, and the per-block sums of p s_V and p m_V
    {
        float v[NREP];
#pragma unroll
        for (int r = 0; r < NREP; r++) {
            v[r] = -INFINITY;
            for (int tt = tid; tt < n_tok; tt += kAThreads) v[r] = fmaxf(v[r], P[r * kAttnChunk + tt]);
        }
        block_reduce<NREP, true>(v, scratch, mx);
        float ws[NREP * 4], zs[NREP * 4], es[NREP];
#pragma unroll
        for (int k = 0; k < NREP * 4; k++) ws[k] = zs[k] = 0.0f;
#pragma unroll
        for (int r = 0; r < NREP; r++) es[r] = 0.0f;
        for (int tt = tid; tt < n_tok; tt += kAThreads) {
            const int64_t t = c0 + tt;
            const uint32_t* sv = a.scales + a.smap.at(l, 1, b, h, t);
            uint32_t z[4];
#pragma unroll
            for (int k = 0; k < 4; k++) {
                z[k] = k < nb ? __ldg(sv + k) : 0u;
                SV[tt * 4 + k] = z[k];
            }
#pragma unroll
            for (int r = 0; r < NREP; r++) {
                const float p = __expf(P[r * kAttnChunk + tt] - mx[r]);
                P[r * kAttnChunk + tt] = p;
                es[r] += p;
#pragma unroll
                for (int k = 0; k < 4; k++) {
                    ws[r * 4 + k] = fmaf(p, half_lo(z[k]), ws[r * 4 + k]);
                    zs[r * 4 + k] = fmaf(p, half_hi(z[k]), zs[r * 4 + k]);
                }
            }
        }
        block_reduce<NREP, false>(es, scratch, sm);
        block_reduce<NREP * 4, false>(ws, scratch, Wr);
        block_reduce<NREP * 4, false>(zs, scratch, Zr);
    }

    // values: thread = (8 channels, token slice); sum_t (p s_V) f per channel
    const int oct = tid & 15, sl = tid >> 4;
    const int bk = (8 * oct) / blk;
    float acc[NREP][8];
#pragma unroll
    for (int r = 0; r < NREP; r++)
#pragma unroll
        for (int k = 0; k < 8; k++) acc[r][k] = 0.0f;
    {
        const int bit0 = 8 * oct * BITS, wi = bit0 >> 5, sh = bit0 & 31;
        const bool two = sh + 8 * BITS > 32;
        for (int tt = sl; tt < n_tok; tt += kASlices) {
            const uint32_t* row = reinterpret_cast<const uint32_t*>(a.codes + a.cmap.at(l, 1, b, h, c0 + tt));
            const uint32_t w0 = __ldg(row + wi);
            const uint32_t w1 = two ? __ldg(row + wi + 1) : 0u;
            const uint32_t w2 = (BITS == 8 && sh) ? __ldg(row + wi + 2) : 0u;
            const uint64_t v = ((((uint64_t)w1 << 32) | w0) >> sh) | (sh ? ((uint64_t)w2 << (64 - sh)) : 0ull);
            const float s_v = half_lo(SV[tt * 4 + bk]);
#pragma unroll
            for (int k = 0; k < 8; k++) {
                const uint32_t q = (uint32_t)(v >> (k * BITS)) & ((1u << BITS) - 1u);
                const float f = __uint_as_float(0x3F800000u | (q << (23 - BITS)));
#pragma unroll
                for (int r = 0; r < NREP; r++) acc[r][k] = fmaf(P[r * kAttnChunk + tt] * s_v, f, acc[r][k]);
            }
        }
    }
    __syncthreads();  // all reads of P done: its space now holds the slice sums
    float* red = P;   // [16][NREP][128]
#pragma unroll
    for (int r = 0; r < NREP; r++)
#pragma unroll
        for (int k = 0; k < 8; k++) red[(sl * NREP + r) * kAD + 8 * oct + k] = acc[r][k];
    __syncthreads();
    float* part = a.part + ((int64_t)unit * a.n_parts + blockIdx.x) * NREP * (kAD + 2);
    for (int e = tid; e < NREP * kAD; e += kAThreads) {
        const int r = e / kAD, c = e - r * kAD, k = c / blk;
        float s = 0.0f;
        for (int q = 0; q < kASlices; q++) s += red[(q * NREP + r) * kAD + c];
        part[r * (kAD + 2) + 2 + c] = kTwoB * (s - Wr[r * 4 + k]) + Zr[r * 4 + k];
    }
    if (tid < NREP) {
        part[tid * (kAD + 2)] = mx[tid];
        part[tid * (kAD + 2) + 1] = sm[tid];
    }
}

// Merge the chunks of one (l, b, h) and apply G_V^T (per gauge group): out fp32.
__global__ void __launch_bounds__(kAD) attn_combine_kernel(AttnArgs a) {
    __shared__ float zs[kAD];
    const int unit = blockIdx.x, c = threadIdx.x;
    const int l = unit / (a.B * a.H), h = unit % a.H;
    const int g = a.g, grp = c / g, i = c - grp * g;
    const float* Gv = a.G + ((int64_t)(l * 2 + 1) * a.H + h) * (int64_t)kAD * g + (int64_t)grp * g * g;
    for (int r = 0; r < a.n_rep; r++) {
        const float* part = a.part + ((int64_t)unit * a.n_parts * a.n_rep + r) * (kAD + 2);
        const int64_t stride = (int64_t)a.n_rep * (kAD + 2);
        float M = -INFINITY;
        for (int j = 0; j < a.n_parts; j++) M = fmaxf(M, part[j * stride]);
        float Ls = 0.0f, o = 0.0f;
        for (int j = 0; j < a.n_parts; j++) {
            const float e = __expf(part[j * stride] - M);
            Ls = fmaf(part[j * stride + 1], e, Ls);
            o = fmaf(part[j * stride + 2 + c], e, o);
        }
        __syncthreads();
        zs[c] = o / Ls;
        __syncthreads();
        float acc = 0.0f;
        for (int j = 0; j < g; j++) acc = fmaf(__ldg(Gv + (int64_t)j * g + i), zs[grp * g + j], acc);
        a.out[((int64_t)unit * a.n_rep + r) * kAD + c] = acc;
    }
}

// ------------------------------------------------------------------------------------
// Pipelined variant for 2- and 4-bit codes. Scores on tensor cores (mma.sync m16n8k16, bf16 in,
// fp32 accumulate): a code enters as bf16 2^b + q (exact for b <= 7, three integer operations
// per pair of codes) and q' as a bf16 hi + lo pair (two MMAs, 2^-16 relative):
//   D[token][query] = sum_c (2^b + q_tc) q'_c over each 32-channel chunk,
//   q' . zhat_t = sum_chunks s D + (m - 2^b s) C, C = sum_c q'_c over the chunk.
// Values on CUDA cores (their contraction runs over tokens, which would need the codes paired
// along tokens for an MMA): f = 1 + q 2^-b per code, sum_t p_t zhat_tc = 2^b (A - W) + Z with
// A = sum_t p s_V f, W = sum_t p s_V, Z = sum_t p m_V.
// ------------------------------------------------------------------------------------
constexpr int kMThreads = 128;  // 4 warps; each takes 16-token groups in turn

__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile("mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
                 "{%0,%1,%2,%3};\n"
                 : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
                 : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// bf16 pair (low half first) of (2^B + q0, 2^B + q1) from x = q0 | q1 << B (higher bits zero):
// x * (2^(7-B) + 2^(23-2B)) places q0 at bits 7-B.. and q1 at 23-B.. (the ranges do not overlap),
// the mask keeps those two fields, and the constant is the bf16 pattern of 2^B twice.
template <int B>
__device__ __forceinline__ uint32_t pair_bf16(uint32_t x) {
    constexpr uint32_t kM = (1u << B) - 1u;
    constexpr uint32_t kMul = (1u << (7 - B)) | (1u << (23 - 2 * B));
    constexpr uint32_t kMask = (kM << (7 - B)) | (kM << (23 - B));
    constexpr uint32_t kOne = ((127u + B) << 7) * 0x10001u;
    return ((x * kMul) & kMask) | kOne;
}

// (d0, d1) += a * (b0, b1): one packed fp32 fused multiply-add (each lane rounded once, as fmaf).
__device__ __forceinline__ void ffma2(float& d0, float& d1, float a, float b0, float b1) {
    asm("{\n\t.reg .b64 dd, aa, bb;\n\tmov.b64 dd, {%0, %1};\n\tmov.b64 aa, {%2, %2};\n\t"
        "mov.b64 bb, {%3, %4};\n\tfma.rn.f32x2 dd, aa, bb, dd;\n\tmov.b64 {%0, %1}, dd;\n\t}"
        : "+f"(d0), "+f"(d1)
        : "f"(a), "f"(b0), "f"(b1));
}

// v[i] for a runtime i < 4 without indexing a register array (no local memory).
template <typename T>
__device__ __forceinline__ T pick4(const T (&v)[4], int i) {
    return i == 0 ? v[0] : (i == 1 ? v[1] : (i == 2 ? v[2] : v[3]));
}

// bf16 hi + lo of two fp32 values, packed as (lo half = first value).
__device__ __forceinline__ void split2(float v0, float v1, uint32_t& hi, uint32_t& lo) {
    const __nv_bfloat16 h0 = __float2bfloat16_rn(v0), h1 = __float2bfloat16_rn(v1);
    const __nv_bfloat16 l0 = __float2bfloat16_rn(v0 - __bfloat162float(h0));
    const __nv_bfloat16 l1 = __float2bfloat16_rn(v1 - __bfloat162float(h1));
    hi = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    lo = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
}

// The 2B-bit field of channels (2j, 2j + 1) of a row, j = 4 * wsel + t within word w.
template <int B>
__device__ __forceinline__ uint32_t pair_field(uint32_t w, int t) {
    if (B == 4) return __byte_perm(w, 0u, 0x4440u | (uint32_t)t);
    return (w >> (4 * t)) & 0xFu;  // B == 2: a pair is one nibble
}

// Shared-memory layout of attn_chunk_mma_kernel (bytes).
template <int BITS, int NREP>
struct MmaSmem {
    static constexpr int kRow = kAD * BITS / 8;                       // packed token row
    static constexpr int kStage = kAttnChunk * kRow;                  // one chunk of one tensor
    static constexpr int bars = 0;                                    // [2 stages][K, V] mbarriers
    static constexpr int flags = 32;                                  // abort flags
    static constexpr int codes = 64;                                  // [2 stages][K, V][kStage]
    static constexpr int qs = codes + 4 * kStage;                     // [NREP][128] q'
    static constexpr int c32 = qs + NREP * kAD * 4;                   // [NREP][4]
    static constexpr int run = c32 + NREP * 4 * 4;                    // [NREP] max, sum, alpha; [NREP][4] W, Z
    static constexpr int scratch = run + NREP * (3 + 8) * 4;          // [4 warps][NREP * 4]
    static constexpr int outv = scratch + 4 * NREP * 4 * 4;           // [NREP * 4] reduction results
    static constexpr int sk = outv + NREP * 4 * 4;                    // [2][chunk][4] key scales
    static constexpr int sv = sk + 2 * kAttnChunk * 4 * 4;            // [2][chunk][4] value scales
    static constexpr int p = sv + 2 * kAttnChunk * 4 * 4;             // [chunk][NREP] scores / p; red
    static constexpr int pbytes = NREP * kAttnChunk * 4, rbytes = (kMThreads / 16) * NREP * kAD * 4;
    static constexpr int total = p + (pbytes > rbytes ? pbytes : rbytes);
};

// One CTA per (l, b, h) and part: the part's chunks in order, the next chunk's key and value
// codes arriving by bulk copy into the other stage (and its scales by loads held in registers)
// while this one is computed, and an online softmax over the chunks (running max; earlier sums
// rescaled by exp(old - new); each thread keeps its own sums until the end).
template <int BITS, int NREP>
__global__ void __launch_bounds__(kMThreads, 3) attn_chunk_mma_kernel(AttnArgs a) {
    static_assert(BITS == 2 || BITS == 4, "tensor-core attention serves 2- and 4-bit codes");
    using SL = MmaSmem<BITS, NREP>;
    constexpr int kWords = kAD * BITS / 32;  // code words per token row
    constexpr int kRow = SL::kRow;
    constexpr float kOff = (float)(1 << BITS);
    extern __shared__ __align__(16) unsigned char smem[];
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + SL::bars);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + SL::flags);  // [1] stays 0 (drains)
    float* qs = reinterpret_cast<float*>(smem + SL::qs);
    float* c32 = reinterpret_cast<float*>(smem + SL::c32);
    float* Mrun = reinterpret_cast<float*>(smem + SL::run);
    float* Lrun = Mrun + NREP;
    float* alpha = Lrun + NREP;
    float* Wr = alpha + NREP;   // [NREP][4]
    float* Zr = Wr + NREP * 4;  // [NREP][4]
    float* scratch = reinterpret_cast<float*>(smem + SL::scratch);
    uint32_t* SKb = reinterpret_cast<uint32_t*>(smem + SL::sk);
    uint32_t* SVb = reinterpret_cast<uint32_t*>(smem + SL::sv);
    float* P = reinterpret_cast<float*>(smem + SL::p);
    float* outv = reinterpret_cast<float*>(smem + SL::outv);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5, g = lane >> 2, t = lane & 3;
    const int unit = blockIdx.y;
    const int l = unit / (a.B * a.H), bh = unit - l * a.B * a.H, b = bh / a.H, h = bh - (bh / a.H) * a.H;
    const int blk = a.blk, nb = kAD / blk;
    const int ch_lo = blockIdx.x * a.chunks_per_part;
    const int ch_hi = ch_lo + a.chunks_per_part < a.n_chunks ? ch_lo + a.chunks_per_part : a.n_chunks;

    auto chunk_tokens = [&](int ci) -> int {
        const int64_t c0 = (int64_t)ci * kAttnChunk;
        return a.T - c0 < kAttnChunk ? (int)(a.T - c0) : kAttnChunk;
    };
    auto issue = [&](int ci, int st) {  // thread 0: key and value codes of chunk ci into stage st
        const uint32_t bytes = (uint32_t)chunk_tokens(ci) * kRow;
        const int64_t c0 = (int64_t)ci * kAttnChunk;
        mbar_arrive_expect_tx(&bars[2 * st], bytes);
        bulk_load(smem + SL::codes + (2 * st) * SL::kStage, a.codes + a.cmap.at(l, 0, b, h, c0), bytes, &bars[2 * st]);
        mbar_arrive_expect_tx(&bars[2 * st + 1], bytes);
        bulk_load(smem + SL::codes + (2 * st + 1) * SL::kStage, a.codes + a.cmap.at(l, 1, b, h, c0), bytes,
                  &bars[2 * st + 1]);
    };

    // the key and value scales of a chunk's tokens: tokens tid, tid + 128, ... of the chunk
    auto load_scales = [&](int ci, uint32_t (&ks)[kAttnChunk / kMThreads][4], uint32_t (&vs)[kAttnChunk / kMThreads][4]) {
        const int64_t c0 = (int64_t)ci * kAttnChunk;
        const int n = chunk_tokens(ci);
#pragma unroll
        for (int q = 0; q < kAttnChunk / kMThreads; q++) {
            const int tt = tid + q * kMThreads;
#pragma unroll
            for (int k = 0; k < 4; k++) ks[q][k] = vs[q][k] = 0u;
            if (tt < n) {
                const uint32_t* kp = a.scales + a.smap.at(l, 0, b, h, c0 + tt);
                const uint32_t* vp = a.scales + a.smap.at(l, 1, b, h, c0 + tt);
#pragma unroll
                for (int k = 0; k < 4; k++)
                    if (k < nb) {
                        ks[q][k] = __ldg(kp + k);
                        vs[q][k] = __ldg(vp + k);
                    }
            }
        }
    };
    auto store_scales = [&](int bufi, const uint32_t (&ks)[kAttnChunk / kMThreads][4],
                            const uint32_t (&vs)[kAttnChunk / kMThreads][4]) {
#pragma unroll
        for (int q = 0; q < kAttnChunk / kMThreads; q++) {
            const int tt = tid + q * kMThreads;
#pragma unroll
            for (int k = 0; k < 4; k++) {
                SKb[(bufi * kAttnChunk + tt) * 4 + k] = ks[q][k];
                SVb[(bufi * kAttnChunk + tt) * 4 + k] = vs[q][k];
            }
        }
    };
    uint32_t nks[kAttnChunk / kMThreads][4], nvs[kAttnChunk / kMThreads][4];

    if (tid == 0) {
        abort_flag[0] = 0;
        abort_flag[1] = 0;
        for (int k = 0; k < 4; k++) mbar_init(&bars[k], 1);
        fence_barrier_init();
    }
    if (ch_lo < ch_hi) {
        load_scales(ch_lo, nks, nvs);
        store_scales(0, nks, nvs);
    }
    for (int e = tid; e < NREP * kAD; e += kMThreads) qs[e] = a.qrot[(int64_t)unit * NREP * kAD + e];
    if (tid < NREP) Mrun[tid] = -INFINITY;
    __syncthreads();
    if (tid == 0 && ch_lo < ch_hi) issue(ch_lo, 0);
    if (tid < NREP * 4) {
        const float* src = qs + (tid >> 2) * kAD + (tid & 3) * 32;
        float s = 0.0f;
        for (int k = 0; k < 32; k++) s += src[k];
        c32[tid] = s;
    }
    // B fragments of q' (query n = g; rows = channels 16 ks + 2t + {0, 1} and + 8), hi and lo
    uint32_t qh[8][2], ql[8][2];
#pragma unroll
    for (int ks = 0; ks < 8; ks++)
#pragma unroll
        for (int hf = 0; hf < 2; hf++) {
            const int ch = 16 * ks + 8 * hf + 2 * t;
            const float v0 = g < NREP ? qs[g * kAD + ch] : 0.0f, v1 = g < NREP ? qs[g * kAD + ch + 1] : 0.0f;
            split2(v0, v1, qh[ks][hf], ql[ks][hf]);
        }
    __syncthreads();

    // value sums of this thread: channels 8 oct .. 8 oct + 7, tokens vsl, vsl + 8, ...
    const int oct = tid & 15, vsl = tid >> 4, vbk = (8 * oct) / blk;
    float acc[NREP][8];
#pragma unroll
    for (int r = 0; r < NREP; r++)
#pragma unroll
        for (int k = 0; k < 8; k++) acc[r][k] = 0.0f;
    // this thread's share of the softmax sums: sum p, sum p s_V and sum p m_V per block
    float lsum[NREP], wsum[NREP][4], zsum[NREP][4];
#pragma unroll
    for (int r = 0; r < NREP; r++) {
        lsum[r] = 0.0f;
#pragma unroll
        for (int k = 0; k < 4; k++) wsum[r][k] = zsum[r][k] = 0.0f;
    }

    for (int ci = ch_lo; ci < ch_hi; ci++) {
        const int it = ci - ch_lo, st = it & 1;
        const uint32_t par = (uint32_t)(it >> 1) & 1u;
        const uint32_t* SK = SKb + st * kAttnChunk * 4;
        const uint32_t* SV = SVb + st * kAttnChunk * 4;
        if (ci + 1 < ch_hi) load_scales(ci + 1, nks, nvs);  // stored after this chunk
        const unsigned char* Kc = smem + SL::codes + (2 * st) * SL::kStage;
        const unsigned char* Vc = Kc + SL::kStage;
        const int64_t c0 = (int64_t)ci * kAttnChunk;
        const int n_tok = chunk_tokens(ci);
        const int ngrp = (n_tok + 15) / 16;
        // the other stage was released by the barrier that ended the previous chunk
        if (tid == 0 && ci + 1 < ch_hi) issue(ci + 1, st ^ 1);
        if (!__syncthreads_and(mbar_wait(&bars[2 * st], par, abort_flag, a.wait_ns))) {
            if (tid == 0) raise_flag(a.status, CG_FLAG_PIPE_TIMEOUT);
            // let every copy issued so far land (normal limit): this chunk's stage, and the next
            // chunk's stage if it was issued
            for (int sk = 0; sk < 2; sk++) {
                const int itk = sk == st ? it : it + 1;
                if (ch_lo + itk >= ch_hi) continue;
                const uint32_t pk = (uint32_t)(itk >> 1) & 1u;
                mbar_wait(&bars[2 * sk], pk, abort_flag + 1, tc::kWaitLimitNs);
                mbar_wait(&bars[2 * sk + 1], pk, abort_flag + 1, tc::kWaitLimitNs);
            }
            return;
        }

        // scores: a warp takes 16 tokens; thread rows g and g + 8, columns (queries) 2t, 2t + 1
        for (int grp = warp; grp < ngrp; grp += kMThreads / 32) {
            const int r0 = grp * 16 + g, r1 = r0 + 8;
            uint32_t w0[kWords], w1[kWords];
#pragma unroll
            for (int k = 0; k < kWords; k++) w0[k] = w1[k] = 0u;
            if (r0 < n_tok) {
                const uint4* row = reinterpret_cast<const uint4*>(Kc + r0 * kRow);
#pragma unroll
                for (int k = 0; k < kWords / 4; k++) {
                    const uint4 v = row[k];
                    w0[4 * k] = v.x; w0[4 * k + 1] = v.y; w0[4 * k + 2] = v.z; w0[4 * k + 3] = v.w;
                }
            }
            if (r1 < n_tok) {
                const uint4* row = reinterpret_cast<const uint4*>(Kc + r1 * kRow);
#pragma unroll
                for (int k = 0; k < kWords / 4; k++) {
                    const uint4 v = row[k];
                    w1[4 * k] = v.x; w1[4 * k + 1] = v.y; w1[4 * k + 2] = v.z; w1[4 * k + 3] = v.w;
                }
            }
            float d[4][4];
#pragma unroll
            for (int k = 0; k < 4; k++) d[k][0] = d[k][1] = d[k][2] = d[k][3] = 0.0f;
#pragma unroll
            for (int ks = 0; ks < 8; ks++) {
                // pair j = 8 ks + t (channels 16 ks + 2t, + 1) and j + 4 (channels + 8)
                const int wa = BITS == 4 ? 2 * ks : ks, wb = BITS == 4 ? 2 * ks + 1 : ks;
                const int ta = t, tb = BITS == 4 ? t : t + 4;
                const uint32_t a0 = pair_bf16<BITS>(pair_field<BITS>(w0[wa], ta));
                const uint32_t a1 = pair_bf16<BITS>(pair_field<BITS>(w1[wa], ta));
                const uint32_t a2 = pair_bf16<BITS>(pair_field<BITS>(w0[wb], tb));
                const uint32_t a3 = pair_bf16<BITS>(pair_field<BITS>(w1[wb], tb));
                mma16816(d[ks >> 1], a0, a1, a2, a3, qh[ks][0], qh[ks][1]);
                mma16816(d[ks >> 1], a0, a1, a2, a3, ql[ks][0], ql[ks][1]);
            }
#pragma unroll
            for (int half = 0; half < 2; half++) {
                const int r = half ? r1 : r0;
                if (r >= n_tok) continue;
                uint32_t sz[4];
#pragma unroll
                for (int k = 0; k < 4; k++) sz[k] = SK[r * 4 + k];
#pragma unroll
                for (int cq = 0; cq < 2; cq++) {
                    const int q = 2 * t + cq;
                    if (q >= NREP) continue;
                    float s = 0.0f;
#pragma unroll
                    for (int k = 0; k < 4; k++) {
                        const uint32_t z = pick4(sz, (32 * k) / blk);
                        const float sc = half_lo(z), mz = half_hi(z);
                        s += sc * d[k][2 * half + cq] + (mz - kOff * sc) * c32[q * 4 + k];
                    }
                    P[r * NREP + q] = s;
                }
            }
        }
        __syncthreads();

        // online softmax: the chunk's max, the new running max and the rescale factor
        {
            float v[NREP];
#pragma unroll
            for (int r = 0; r < NREP; r++) {
                v[r] = -INFINITY;
                for (int tt = tid; tt < n_tok; tt += kMThreads) v[r] = fmaxf(v[r], P[tt * NREP + r]);
            }
            block_reduce_n<NREP, true, kMThreads>(v, scratch, outv);
            if (tid < NREP) {
                const float mn = fmaxf(Mrun[tid], outv[tid]);
                alpha[tid] = __expf(Mrun[tid] - mn);  // 0 on the first chunk (old max -inf)
                Mrun[tid] = mn;
            }
            __syncthreads();
#pragma unroll
            for (int r = 0; r < NREP; r++) {
                const float al = alpha[r];
                lsum[r] *= al;
#pragma unroll
                for (int k = 0; k < 4; k++) {
                    wsum[r][k] *= al;
                    zsum[r][k] *= al;
                }
#pragma unroll
                for (int k = 0; k < 8; k++) acc[r][k] *= al;
            }
            for (int tt = tid; tt < n_tok; tt += kMThreads) {
                uint32_t z[4];
#pragma unroll
                for (int k = 0; k < 4; k++) z[k] = SV[tt * 4 + k];
#pragma unroll
                for (int r = 0; r < NREP; r++) {
                    const float p = __expf(P[tt * NREP + r] - Mrun[r]);
                    P[tt * NREP + r] = p;
                    lsum[r] += p;
#pragma unroll
                    for (int k = 0; k < 4; k++) {
                        wsum[r][k] = fmaf(p, half_lo(z[k]), wsum[r][k]);
                        zsum[r][k] = fmaf(p, half_hi(z[k]), zsum[r][k]);
                    }
                }
            }
        }
        __syncthreads();

        // values on CUDA cores: thread = 8 channels (one 32-bit group of 4-bit codes, half of
        // one for 2-bit) x token slice; sum_t (p s_V) f per channel, f = 1 + q 2^-b
        if (!__syncthreads_and(mbar_wait(&bars[2 * st + 1], par, abort_flag, a.wait_ns))) {
            if (tid == 0) raise_flag(a.status, CG_FLAG_PIPE_TIMEOUT);
            if (ci + 1 < ch_hi) {
                mbar_wait(&bars[2 * (st ^ 1)], (uint32_t)((it + 1) >> 1) & 1u, abort_flag + 1, tc::kWaitLimitNs);
                mbar_wait(&bars[2 * (st ^ 1) + 1], (uint32_t)((it + 1) >> 1) & 1u, abort_flag + 1, tc::kWaitLimitNs);
            }
            mbar_wait(&bars[2 * st + 1], par, abort_flag + 1, tc::kWaitLimitNs);
            return;
        }
        {
            const uint32_t* vrow = reinterpret_cast<const uint32_t*>(Vc);
            for (int tt = vsl; tt < n_tok; tt += kMThreads / 16) {
                const uint32_t word = vrow[tt * (kRow / 4) + (BITS == 4 ? oct : (oct >> 1))];
                const uint32_t bits = BITS == 4 ? word : (word >> (16 * (oct & 1)));
                const float s_v = half_lo(SV[tt * 4 + vbk]);
                float wgt[NREP];
#pragma unroll
                for (int r = 0; r < NREP; r++) wgt[r] = P[tt * NREP + r] * s_v;
                float f[8];
#pragma unroll
                for (int k = 0; k < 8; k++)
                    f[k] = __uint_as_float(0x3F800000u | (((bits >> (k * BITS)) & ((1u << BITS) - 1u)) << (23 - BITS)));
#pragma unroll
                for (int r = 0; r < NREP; r++)
#pragma unroll
                    for (int k = 0; k < 8; k += 2) ffma2(acc[r][k], acc[r][k + 1], wgt[r], f[k], f[k + 1]);
            }
        }
        __syncthreads();  // P, the scales and this stage's codes are free for the next chunk
        if (ci + 1 < ch_hi) store_scales(st ^ 1, nks, nvs);
    }
    // the sums over threads (one reduction of each, after the last chunk)
    block_reduce_n<NREP, false, kMThreads>(lsum, scratch, outv);
    if (tid < NREP) Lrun[tid] = outv[tid];
    __syncthreads();
    {
        float wv[NREP * 4];
#pragma unroll
        for (int r = 0; r < NREP; r++)
#pragma unroll
            for (int k = 0; k < 4; k++) wv[r * 4 + k] = wsum[r][k];
        block_reduce_n<NREP * 4, false, kMThreads>(wv, scratch, outv);
        if (tid < NREP * 4) Wr[tid] = outv[tid];
        __syncthreads();
#pragma unroll
        for (int r = 0; r < NREP; r++)
#pragma unroll
            for (int k = 0; k < 4; k++) wv[r * 4 + k] = zsum[r][k];
        block_reduce_n<NREP * 4, false, kMThreads>(wv, scratch, outv);
        if (tid < NREP * 4) Zr[tid] = outv[tid];
        __syncthreads();
    }

    // the slices' sums, then the sum over slices (red reuses P's space)
    float* red = P;  // [8 slices][NREP][128]
#pragma unroll
    for (int r = 0; r < NREP; r++)
#pragma unroll
        for (int k = 0; k < 8; k++) red[(vsl * NREP + r) * kAD + 8 * oct + k] = acc[r][k];
    __syncthreads();
    float* part = a.part + ((int64_t)unit * a.n_parts + blockIdx.x) * NREP * (kAD + 2);
    for (int e = tid; e < NREP * kAD; e += kMThreads) {
        const int r = e / kAD, c = e - r * kAD, k = c / blk;
        float s = 0.0f;
        for (int q = 0; q < kMThreads / 16; q++) s += red[(q * NREP + r) * kAD + c];
        part[r * (kAD + 2) + 2 + c] = kOff * (s - Wr[r * 4 + k]) + Zr[r * 4 + k];
    }
    if (tid < NREP) {
        part[tid * (kAD + 2)] = Mrun[tid];
        part[tid * (kAD + 2) + 1] = Lrun[tid];
    }
}

template <int BITS, int NREP>
size_t mma_smem() {
    return (size_t)MmaSmem<BITS, NREP>::total;
}

template <int BITS, int NREP>
cudaError_t launch_mma_chunks(const AttnArgs& a, cudaStream_t st) {
    const size_t smem = mma_smem<BITS, NREP>();
    cudaError_t e = cudaFuncSetAttribute(attn_chunk_mma_kernel<BITS, NREP>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)a.n_parts, (unsigned)(a.L * a.B * a.H));
    attn_chunk_mma_kernel<BITS, NREP><<<grid, kMThreads, smem, st>>>(a);
    return cudaGetLastError();
}

template <int BITS>
cudaError_t launch_mma_bits(const AttnArgs& a, cudaStream_t st) {
    switch (a.n_rep) {
        case 1: return launch_mma_chunks<BITS, 1>(a, st);
        case 2: return launch_mma_chunks<BITS, 2>(a, st);
        case 4: return launch_mma_chunks<BITS, 4>(a, st);
        case 8: return launch_mma_chunks<BITS, 8>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

template <int BITS, int NREP>
size_t chunk_smem() {
    const size_t fixed = (size_t)(NREP * kAD + NREP * 4 + 2 * NREP + 2 * NREP * 4 + 8 * NREP * 4) * 4 +
                         (size_t)kAttnChunk * 4 * 4;
    const size_t pbytes = (size_t)NREP * kAttnChunk * 4, rbytes = (size_t)kASlices * NREP * kAD * 4;
    return fixed + (pbytes > rbytes ? pbytes : rbytes);
}

template <int BITS, int NREP>
cudaError_t launch_chunks(const AttnArgs& a, cudaStream_t st) {
    const size_t smem = chunk_smem<BITS, NREP>();
    cudaError_t e = cudaFuncSetAttribute(attn_chunk_kernel<BITS, NREP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)a.n_parts, (unsigned)(a.L * a.B * a.H));
    attn_chunk_kernel<BITS, NREP><<<grid, kAThreads, smem, st>>>(a);
    return cudaGetLastError();
}

template <int BITS>
cudaError_t launch_chunks_bits(const AttnArgs& a, cudaStream_t st) {
    switch (a.n_rep) {
        case 1: return launch_chunks<BITS, 1>(a, st);
        case 2: return launch_chunks<BITS, 2>(a, st);
        case 4: return launch_chunks<BITS, 4>(a, st);
        case 8: return launch_chunks<BITS, 8>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

size_t attn_workspace_bytes(int64_t units, int n_rep, int d, int64_t T) {
    const int64_t n_chunks = (T + kAttnChunk - 1) / kAttnChunk;
    const size_t q = (((size_t)units * n_rep * d * 4) + 255) / 256 * 256;
    return q + (size_t)units * n_chunks * n_rep * (d + 2) * 4;
}

cudaError_t launch_attention(const AttnArgs& args, cudaStream_t st) {
    AttnArgs a = args;
    const bool mma = a.bits == 2 || a.bits == 4;
    if (mma) {
        // parts of consecutive chunks per (l, b, h): enough CTAs to fill the SMs a few times over
        int dev = 0, sms = 152;
        if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        const int64_t units = (int64_t)a.L * a.B * a.H, target = (int64_t)sms * 12;
        int64_t splits = (target + units - 1) / units;
        if (splits > a.n_chunks) splits = a.n_chunks;
        if (splits < 1) splits = 1;
        a.chunks_per_part = (int)((a.n_chunks + splits - 1) / splits);
        a.n_parts = (a.n_chunks + a.chunks_per_part - 1) / a.chunks_per_part;
    } else {
        a.chunks_per_part = 1;
        a.n_parts = a.n_chunks;
    }
    const size_t gsmem = (size_t)kAD * a.g * 4 + kAD * 4;
    cudaError_t e = cudaFuncSetAttribute(attn_query_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gsmem);
    if (e != cudaSuccess) return e;
    attn_query_kernel<<<dim3((unsigned)(a.L * a.H), (unsigned)((a.B + kQuerySeqs - 1) / kQuerySeqs)), kAD, gsmem, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    switch (a.bits) {
        case 2: e = launch_mma_bits<2>(a, st); break;
        case 3: e = launch_chunks_bits<3>(a, st); break;
        case 4: e = launch_mma_bits<4>(a, st); break;
        case 6: e = launch_chunks_bits<6>(a, st); break;
        case 8: e = launch_chunks_bits<8>(a, st); break;
        default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    attn_combine_kernel<<<(unsigned)(a.L * a.B * a.H), kAD, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace cg
