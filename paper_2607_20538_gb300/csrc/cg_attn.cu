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
// Kernels: attn_query_kernel (q' = scale * G_K q), attn_chunk_kernel (one CTA per 512 tokens of
// a (l, b, h): scores, chunk softmax, gauge-space weighted sum, written as a partial with its max
// and sum), attn_combine_kernel (merges the chunks and applies G_V^T).
#include "cg_launch.h"

namespace cg {
namespace {

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

// q' = scale * G_K q for every (b, query head) of one (l, h); G_K transposed in shared memory.
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
    for (int b = 0; b < a.B; b++)
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

// Deterministic block reduction of NV values per thread (sum or max), result in out[NV].
template <int NV, bool MAX>
__device__ __forceinline__ void block_reduce(float (&v)[NV], float* scratch, float* out) {
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
        for (int w = 1; w < kAThreads / 32; w++) {
            const float o = scratch[w * NV + threadIdx.x];
            r = MAX ? fmaxf(r, o) : r + o;
        }
        out[threadIdx.x] = r;
    }
    __syncthreads();
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
    uint32_t* SV = reinterpret_cast<uint32_t*>(scratch + 8 * NREP * 4);  // [512][4] value scales
    float* P = reinterpret_cast<float*>(SV + kAttnChunk * 4);    // [NREP][512] scores, then p;
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
    float* part = a.part + ((int64_t)unit * a.n_chunks + blockIdx.x) * NREP * (kAD + 2);
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
        const float* part = a.part + ((int64_t)unit * a.n_chunks * a.n_rep + r) * (kAD + 2);
        const int64_t stride = (int64_t)a.n_rep * (kAD + 2);
        float M = -INFINITY;
        for (int j = 0; j < a.n_chunks; j++) M = fmaxf(M, part[j * stride]);
        float Ls = 0.0f, o = 0.0f;
        for (int j = 0; j < a.n_chunks; j++) {
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
    dim3 grid((unsigned)a.n_chunks, (unsigned)(a.L * a.B * a.H));
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

cudaError_t launch_attention(const AttnArgs& a, cudaStream_t st) {
    const size_t gsmem = (size_t)kAD * a.g * 4 + kAD * 4;
    cudaError_t e = cudaFuncSetAttribute(attn_query_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)gsmem);
    if (e != cudaSuccess) return e;
    attn_query_kernel<<<(unsigned)(a.L * a.H), kAD, gsmem, st>>>(a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    switch (a.bits) {
        case 2: e = launch_chunks_bits<2>(a, st); break;
        case 3: e = launch_chunks_bits<3>(a, st); break;
        case 4: e = launch_chunks_bits<4>(a, st); break;
        case 6: e = launch_chunks_bits<6>(a, st); break;
        case 8: e = launch_chunks_bits<8>(a, st); break;
        default: return cudaErrorInvalidValue;
    }
    if (e != cudaSuccess) return e;
    attn_combine_kernel<<<(unsigned)(a.L * a.B * a.H), kAD, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace cg
