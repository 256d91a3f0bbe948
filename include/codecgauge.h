/*
 * codecgauge.h -- C ABI of libcodecgauge, the GB300 (sm_103a) encode/decode path of
 * Codec-Gauge's inference-time cache-coordinate layer (arxiv 2607.20538).
 *
 * The method (Sec. 3, the encode/decode equations): for every layer l, cache type
 * s in {K, V}, head h and channel group r, a fixed orthogonal gauge G_{l,s,h,r}
 * (g x g) maps each g-channel slice of a cached key/value vector into codec-facing
 * coordinates, Z = G X; a fixed backend codes Z into a byte buffer B_c = C(Z); decode
 * recovers Zhat = D(B_c) and restores Xhat = G^{-1} Zhat = G^T Zhat (Sec. 4.1: the
 * gauge is exp(A - A^T), so its inverse is its transpose). The gauge mixes channels
 * only inside a group; it never mixes tokens, heads or layers (Sec. 1, Sec. 3).
 * Backends (Sec. 4.3): block-uniform asymmetric min/max quantization and KIVI-style
 * quantization (per-channel key ranges, per-token value ranges, full-precision
 * residual window), at 2, 3, 4, 6 or 8 bits.
 *
 * Conventions shared by every entry point
 *   - All data pointers are DEVICE pointers owned by the caller. The library never
 *     allocates, frees or retains them. Calls are asynchronous on `stream`
 *     (a cudaStream_t passed as void*; NULL = legacy default stream).
 *   - Every entry point returns an int status: CG_OK or a negative CG_E* code. On
 *     CG_EINVAL, CG_EUNSUPPORTED and CG_ERANGE nothing was launched. A KIVI call launches
 *     up to three kernels (keys, values, residual copy) in order, so a CG_ECUDA from it may
 *     follow launches that were already queued; the outputs are then invalid.
 *     cg_last_error() returns a message.
 *   - Numbers: bf16 = IEEE binary16-brain (8-bit significand), fp16 = IEEE binary16,
 *     fp32 = IEEE binary32, all little-endian.
 *
 * Tensor layouts (row-major, leftmost index slowest; layer-major so one layer's bytes
 * are contiguous and a per-layer call is made with L = 1 and pointers offset by the
 * L = 1 byte counts of cg_packed_bytes):
 *   KV input/output  X  : bf16 [L][2][B][H][T][d]      (s = 0 keys, s = 1 values; Sec. 3)
 *   gauges           G  : fp32 [L][2][H][d/g][g][g]    G[i][j] row-major, z_i = sum_j G[i][j] x_j
 *   block-uniform (CG_BLOCK_UNIFORM), history of T_cap tokens:
 *     codes  : u8    [L][2][B][H][T_cap][d/block][block*bits/8]
 *     scales : half2 [L][2][B][H][T_cap][d/block]      .x = scale s, .y = zero (block min m)
 *   block-uniform tiles (CG_BLOCK_TILE), T_b = CG_TILE_TOKENS, n_tiles = ceil(T_cap / T_b):
 *     codes  : u8    [L][2][B][H][T_cap][d/block][block*bits/8]   (as CG_BLOCK_UNIFORM)
 *     scales : half2 [L][2][B][H][n_tiles][d/block]  range of tokens [k T_b, (k+1) T_b) x block
 *     A tile's range covers the tokens of the call that wrote it: the last tile of a call
 *     may hold fewer than T_b tokens (its range covers those only), and a call starts at a
 *     tile boundary (t0 % T_b == 0), so appending to an open tile means re-encoding it
 *     from its first token.
 *   KIVI-style (CG_KIVI), n_q = max(0, floor((T - residual)/block)) * block quantized tokens:
 *     codes  per layer: keys  u8 [B][H][n_q/block][d][block*bits/8]   (per-channel token streams)
 *                       then values u8 [B][H][n_q][d/block][block*bits/8]
 *     scales per layer: keys  half2 [B][H][n_q/block][d], then values half2 [B][H][n_q][d/block]
 *     residual        : bf16 [L][2][B][H][T - n_q][d]   newest tokens, raw (un-gauged) X
 *   no-compression (CG_NONE, the sanity rows of Sec. 4.4):
 *     codes  : fp32 [L][2][B][H][T_cap][d]  the gauge-space tensor Z itself
 *
 * Bit packing: inside one block payload, code k occupies bits [k*bits, (k+1)*bits) of a
 * little-endian bit stream (bit 0 = LSB of byte 0). For KIVI keys a "block" is the
 * stream of `block` consecutive tokens of one channel.
 *
 * Quantization rule (Sec. 4.3 names an asymmetric min/max range per block; the
 * arithmetic below is this library's fixed reading of it):
 *   z      = fp32 gauge-space value z_i = sum_j G[i][j] x_j in a fixed order: pairwise
 *            summation of the fp32 products G[i][j] * x_j (S(a,b) = S(a,m) + S(m,b),
 *            m = (a+b)/2, S(j,j+1) = the product), every product and sum rounded to fp32.
 *   s32    = (max - min) / (2^bits - 1) over the block, or over the tile for
 *            CG_BLOCK_TILE (fp32 subtract, fp32 divide)
 *   s, m   = fp16 round-to-nearest-even of s32 and of min; stored as half2 {s, m}
 *   q      = clamp(rint((z - m) / s), 0, 2^bits - 1)  (fp32; q = 0 when s == 0)
 *   decode : zhat = q * s + m ; xhat_i = sum_j G[j][i] zhat_j ; bf16 round-to-nearest-even.
 */
#ifndef CODECGAUGE_H
#define CODECGAUGE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define CG_OK            0
#define CG_EINVAL       (-1)  /* a bad argument: shape, parameter, null or misaligned pointer  */
#define CG_EUNSUPPORTED (-2)  /* valid in the method but not provided (e.g. KIVI append)        */
#define CG_ECUDA        (-3)  /* a CUDA launch or runtime call failed; see cg_last_error()      */
#define CG_ERANGE       (-4)  /* a byte count or index does not fit the library's integer types */

/* Backends (Sec. 4.3 compression conditions; CG_NONE = the no-compression rows of Sec. 4.4).
 * CG_BLOCK_TILE is block-uniform with one range per T_b x block tile, the block shape that
 * Sec. 4.3 gives for block-uniform (T_b = 16 tokens, Sec. 4.2; block = d is its T_b x d_l
 * tile); CG_BLOCK_UNIFORM takes one range per block of one token. */
#define CG_BLOCK_UNIFORM 0
#define CG_KIVI          1
#define CG_NONE          2
#define CG_BLOCK_TILE    3

/* T_b: tokens per block-uniform tile (CG_BLOCK_TILE). */
#define CG_TILE_TOKENS   16

/* Device status bits, accumulated by kernels and read by cg_get_status(). */
#define CG_FLAG_NONFINITE_INPUT 0x1  /* a NaN/Inf bf16 input value was seen                 */
#define CG_FLAG_FP16_OVERFLOW   0x2  /* a block scale or zero did not fit in fp16 (became inf) */
#define CG_FLAG_PIPE_TIMEOUT    0x4  /* a bounded pipeline wait gave up; outputs are invalid  */

/* Cache shape (Sec. 3 notation: B batch, H KV heads, T tokens, d head dimension, L layers).
 * d in {32, 64, 128, 256}; L*2*H <= 65535 and L*B*H <= 65535.
 * t0, T_cap: block-uniform (both kinds) only. Encode writes tokens [t0, t0+T) of a history
 * that holds T_cap tokens per (l, s, b, h); decode reads tokens [t0, t0+T) of it and writes a
 * dense [L][2][B][H][T][d] output. T_cap = 0 means T_cap = t0 + T. CG_BLOCK_TILE requires
 * t0 % CG_TILE_TOKENS == 0 (CG_EUNSUPPORTED otherwise). KIVI requires t0 = 0 and
 * T_cap in {0, T}. */
typedef struct {
    int32_t L, B, H, T, d;
    int32_t t0, T_cap;
} cg_shape;

/* Codec parameters.
 *   backend  : CG_BLOCK_UNIFORM, CG_BLOCK_TILE, CG_KIVI or CG_NONE
 *   group    : gauge group g (Sec. 3, R = d/g groups per head); g in {8,16,32,64,128}, d % g == 0
 *   bits     : 2, 3, 4, 6 or 8 (Sec. 4.3 bit settings; ignored by CG_NONE)
 *   block    : a power of two >= 8 with d % block == 0 and block*bits % 8 == 0;
 *              block-uniform: channels per block (per tile for CG_BLOCK_TILE); KIVI: the
 *              key token-group length and the value channel-group length
 *   residual : KIVI full-precision window length R >= 0 (ignored otherwise)           */
typedef struct {
    int32_t backend;
    int32_t group, bits, block, residual;
} cg_params;

/* Byte counts of the three output buffers for (shape, params): codes, scales and the KIVI
 * residual (0 when the backend has none). Closed form of the layouts above (the measured
 * bytes behind the paper's actual bits/value, Appendix metric table). Host-only; launches
 * nothing. Returns CG_EINVAL on invalid arguments, CG_ERANGE on size_t overflow. */
int cg_packed_bytes(const cg_shape* shape, const cg_params* params,
                    size_t* codes_bytes, size_t* scales_bytes, size_t* residual_bytes);

/* Encode (Sec. 3: Z = G X, B_c = C(Z)). Reads kv_bf16 [L][2][B][H][T][d] and gauges,
 * writes the codes / scales / residual ranges that this shape covers (bytes outside them
 * are left untouched). out_residual may be NULL unless the backend is CG_KIVI with
 * T - n_q > 0; out_scales may be NULL for CG_NONE. All pointers must be 16-byte aligned.
 * Non-finite inputs and fp16 overflow set device status bits (cg_get_status). */
int cg_encode(const cg_shape* shape, const cg_params* params,
              const void* kv_bf16, const float* gauges,
              void* out_codes, void* out_scales, void* out_residual, void* stream);

/* Decode (Sec. 3: Zhat = D(B_c), Xhat = G^{-1} Zhat with G^{-1} = G^T, Sec. 4.1). Reads
 * the buffers written by cg_encode for the same params and writes out_kv_bf16
 * [L][2][B][H][T][d] (the recovered cache restored before attention, Fig. 1). KIVI's
 * residual tokens are copied back verbatim. Pointers 16-byte aligned. */
int cg_decode(const cg_shape* shape, const cg_params* params,
              const void* codes, const void* scales, const void* residual,
              const float* gauges, void* out_kv_bf16, void* stream);

/* ---- Hadamard gauge by fast Walsh-Hadamard transform (the structured Hadamard control of
 * Sec. 4.3) ----
 * Encode / decode with the gauge G_{l,s,h,r} = H_g / sqrt(g) for every (l, s, h, r), H_g the
 * Sylvester Hadamard matrix (H[i][j] = (-1)^popcount(i & j)), each entry stored as the fp32
 * value +-c, c = fp32(1 / sqrt(g)) (1 / sqrt(g) computed in double, then rounded to fp32).
 * No gauge tensor is read: the transform costs O(g log g) per group instead of g^2. The
 * results are those of cg_encode / cg_decode given that gauge tensor: every product of the
 * quantization rule is +-fl(c x_j), and its pairwise summation order over j is the butterfly
 * order of the transform, so codes, scales and zeros are bit for bit the same; decode runs
 * the transform in fp32. Block-uniform rows (CG_BLOCK_UNIFORM) only, any supported d, group,
 * bits and block, with t0 / T_cap as for cg_encode; CG_EUNSUPPORTED for other backends. */
int cg_encode_hadamard(const cg_shape* shape, const cg_params* params, const void* kv_bf16,
                       void* out_codes, void* out_scales, void* stream);
int cg_decode_hadamard(const cg_shape* shape, const cg_params* params, const void* codes,
                       const void* scales, void* out_kv_bf16, void* stream);

/* ---- KIVI streaming (Sec. 4.3 KIVI-style path; the growing cache of a decode loop) ----
 * A KIVI history of capacity T_cap tokens per (l, s, b, h) that grows by appends. Holding
 * T tokens, its first n_q(T) = max(0, floor((T - residual) / block)) * block tokens are
 * quantized and the newest T - n_q(T) stay raw (KIVI's full-precision window). Buffers:
 *   codes, scales : the CG_KIVI layouts above, sized for n_q(T_cap) quantized tokens
 *                   (a layer's keys for n_q(T_cap)/block groups, then its values); group k
 *                   and token t sit at the same place whatever T is
 *   ring          : bf16 [L][2][B][H][W][d], W = residual + block; raw token t lives in
 *                   slot t mod W (the window never holds more than W - 1 tokens)
 *   workspace     : device scratch of cg_kivi_stream_bytes' workspace size, owned by the
 *                   caller; an append that completes a key group stages the group's tokens
 *                   (ring and new input) there before quantizing them
 * The stream state after any sequence of appends equals the CG_KIVI encode of all tokens so
 * far (same codes and scales; the ring holds the raw window). */

/* Byte counts of the stream buffers for capacity shape->T_cap (shape->t0 and T must satisfy
 * t0 + T <= T_cap; they do not change the counts): codes, scales, ring, and the workspace an
 * append with t0 > 0 needs (L*2*B*H*block*d*2; 0 would do for appends that start at 0).
 * Host-only. CG_EINVAL on invalid arguments (backend must be CG_KIVI, T_cap >= 1). */
int cg_kivi_stream_bytes(const cg_shape* shape, const cg_params* params, size_t* codes_bytes,
                         size_t* scales_bytes, size_t* ring_bytes, size_t* workspace_bytes);

/* Append tokens [t0, t0 + T) to a stream that holds t0 tokens. kv_new: bf16 [L][2][B][H][T][d]
 * (the new tokens only). t0 = 0 starts the stream (a prefill of any length); after that an
 * append carries at most `block` tokens (CG_EUNSUPPORTED otherwise), so it completes at most
 * one key group. workspace may be NULL when t0 = 0; otherwise it must hold the workspace size
 * (CG_EINVAL if workspace_bytes is smaller). Launches up to four kernels in order on
 * `stream` (stage, keys, values, ring); a CG_ECUDA may follow queued launches, and the
 * stream state is then invalid. Pointers 16-byte aligned. */
int cg_kivi_append(const cg_shape* shape, const cg_params* params, const void* kv_new_bf16,
                   const float* gauges, void* codes, void* scales, void* ring, void* workspace,
                   size_t workspace_bytes, void* stream);

/* Bytes of the library's own workspace array used by cg_kivi_append_static. */
#define CG_KIVI_APPEND_STATIC_BYTES (32u * 1024u * 1024u)

/* cg_kivi_append without a caller-allocated workspace. The paper has no counterpart: this is
 * an interface for callers that cannot allocate device memory (a framework's memory pool with
 * no hook for extra buffers, memory reserved up front, a real-time loop where an allocation
 * could block or fail). The staging workspace is a fixed array of CG_KIVI_APPEND_STATIC_BYTES
 * in the library's device memory; the call allocates and frees nothing. Arguments and results
 * are those of cg_kivi_append. Shapes whose workspace size (cg_kivi_stream_bytes) exceeds the
 * array return CG_ERANGE whatever t0 is (call per layer instead). The first call on each
 * device looks up the array's address with that device current: make it before any stream
 * capture. All calls share the array, so calls whose kernels overlap on the GPU race on it.
 * Nothing in it needs to start at zero. */
int cg_kivi_append_static(const cg_shape* shape, const cg_params* params, const void* kv_new_bf16,
                          const float* gauges, void* codes, void* scales, void* ring, void* stream);

/* Decode the T tokens a stream holds (shape->t0 must be 0, T <= T_cap): quantized tokens as
 * cg_decode does, raw tokens copied from the ring, into out_kv_bf16 [L][2][B][H][T][d]. */
int cg_kivi_stream_decode(const cg_shape* shape, const cg_params* params, const void* codes,
                          const void* scales, const void* ring, const float* gauges,
                          void* out_kv_bf16, void* stream);

/* ---- Attention straight from a block-uniform cache (Fig. 1: the recovered cache is consumed
 * by softmax attention; Sec. 3: recovery can be folded into the surrounding computation) ----
 * One decoding query per sequence, n_rep query heads per KV head (grouped queries; 1 = MHA):
 *   s_t = scale * q . khat_t,  p = softmax_t(s),  o = sum_t p_t vhat_t
 * over tokens [t0, t0 + T) of the cache, where khat, vhat are what cg_decode would recover.
 * The inverse gauge is folded out of the token loop: q is rotated once into gauge space
 * (q . G^T zhat = (G q) . zhat) and the weighted sum of values stays in gauge space until one
 * G_V^T per query, so the kernels read only codes and scales. Arithmetic is fp32 (scores,
 * softmax, sums); the result is fp32, not bit-exact (see the tolerance in the tests).
 * Supported: CG_BLOCK_UNIFORM and CG_BLOCK_TILE caches with d = 128 and block in {32, 64, 128},
 * any group and bit width; n_rep in {1, 2, 4, 8}; T >= 1. q: bf16 [L][B][H][n_rep][d];
 * out: fp32 [L][B][H][n_rep][d]. workspace: caller-owned device scratch of
 * cg_attention_workspace_bytes (rotated queries and per-512-token partial results). */
int cg_attention_workspace_bytes(const cg_shape* shape, const cg_params* params, int n_rep,
                                 size_t* workspace_bytes);

/* Launches three kernels in order on `stream` (query rotation, per-chunk attention, merge);
 * a CG_ECUDA may follow queued launches, and `out` is then invalid. Pointers 16-byte aligned;
 * CG_EINVAL if workspace_bytes is below the required size or scale is not finite. */
int cg_attention(const cg_shape* shape, const cg_params* params, int n_rep, float scale,
                 const void* q_bf16, const void* codes, const void* scales, const float* gauges,
                 float* out, void* workspace, size_t workspace_bytes, void* stream);

/* Reads and clears (in one atomic step, ordered on `stream`) the accumulated CG_FLAG_* bits
 * of the current device, synchronizes `stream` and returns them in *device_flags. Returns
 * CG_ECUDA if a launch, copy or the synchronize fails. The limit of each bounded pipeline
 * wait in the tensor-core kernels is 4 s; the environment variable CODECGAUGE_PIPE_WAIT_NS
 * (read at every encode/decode call, nanoseconds, at most 4e9; other values are ignored)
 * lowers it. It is a diagnostic knob: below 1 ms the waits poll without suspending, so a
 * limit of a few hundred nanoseconds makes them give up and raise CG_FLAG_PIPE_TIMEOUT
 * without any fault (the outputs of that call are then invalid). The drains of copies
 * already in flight keep the 4 s limit. */
int cg_get_status(void* stream, int32_t* device_flags);

/* Message for the most recent failing call on this host thread ("" if none). The pointer
 * stays valid until the next library call on the same thread. */
const char* cg_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* CODECGAUGE_H */
