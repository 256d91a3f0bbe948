// cg_launch.h -- internal launcher interface between the C ABI (cg_api.cu) and the kernel
// translation units. Not installed; not part of the public ABI.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "cg_common.cuh"

namespace cg {

// One "row" = one token vector of one (l, s, b, h) unit. Row kernels process, for each
// (l, s, h) that shares a gauge, the rows (b, t) for b < B and t < t_count.
struct RowArgs {
    const uint16_t* x;      // encode: bf16 input [L][2][B][H][T_x][d]
    uint16_t* out;          // decode: bf16 output [L][2][B][H][T_x][d]
    const float* G;         // [L][2][H][d/g][g][g]
    uint8_t* codes;         // packed codes (or fp32 z for CG_NONE)
    uint32_t* scales;       // half2 {s, m} per block
    int32_t* status;
    int L, B, H, d, g, bits, blk;
    int s_lo, s_n;          // cache types handled: s in [s_lo, s_lo + s_n)
    int64_t T_x;            // tokens per unit in the dense x / out tensor
    int64_t t_count;        // tokens processed per unit
    int none_mode;          // 1 = CG_NONE (codes hold fp32 z rows)
    uint64_t wait_ns;       // limit of each bounded pipeline wait of the tensor-core kernels
    RowMap cmap;            // byte offset of a row's codes
    RowMap smap;            // u32 index of a row's first block scale
};

// KIVI keys: one CTA per (l, b, h, token group); per-channel ranges over Gt tokens.
struct KeyArgs {
    const uint16_t* x;      // encode input  [L][2][B][H][T][d] (keys are s = 0)
    uint16_t* out;          // decode output [L][2][B][H][T][d]
    const float* G;
    uint8_t* codes;         // whole codes buffer
    uint32_t* scales;       // whole scales buffer
    int32_t* status;
    int L, B, H, d, g, bits, Gt;
    int64_t T, nq;
    int64_t layer_codes, layer_scales;  // bytes / u32 per layer
    int64_t key_codes_per_bh, key_scales_per_bh;
};

struct ResidArgs {
    const uint16_t* src;
    uint16_t* dst;
    int64_t units;          // L*2*B*H
    int64_t T, nq, d;
    int to_residual;        // 1: x -> residual window, 0: residual window -> out
};

// Token-row moves of the KIVI stream: rows t in [t_lo, t_hi) of every (l, s, b, h) unit.
// Source row t: ring slot t mod W when t < src_split, else row t - x_t0 of the dense x
// ([units][T_x][d]). Destination: ring slot t mod W (dst_ring) or dense row t - dst_t0 of
// [units][dst_T][d].
struct MoveArgs {
    const uint16_t* ring_src;
    const uint16_t* x;
    uint16_t* dst;
    int64_t units, d, W;
    int64_t T_x, x_t0, src_split;
    int64_t t_lo, t_hi;
    int dst_ring;
    int64_t dst_T, dst_t0;
};

// Attention of one query per sequence over a block-uniform cache, from the packed codes.
struct AttnArgs {
    const uint16_t* q;      // bf16 [L][B][H][n_rep][d]
    const float* G;         // [L][2][H][d/g][g][g]
    const uint8_t* codes;   // block-uniform codes (rows layout)
    const uint32_t* scales; // half2 {s, m} per block (per token, or per 16-token tile)
    RowMap cmap, smap;      // row maps of tokens [t0, t0 + T)
    float* qrot;            // workspace: scale * G_K q, [L*B*H][n_rep][d]
    float* part;            // workspace: [L*B*H][n_chunks][n_rep][d + 2] (max, sum, o')
    float* out;             // fp32 [L][B][H][n_rep][d]
    int L, B, H, d, g, bits, blk, n_rep;
    int64_t T;              // tokens attended
    int n_chunks;           // 256-token chunks of [t0, t0 + T)
    int n_parts;            // partial results per (l, b, h), each over chunks_per_part chunks
    int chunks_per_part;
    float scale;
    int32_t* status;
    uint64_t wait_ns;       // limit of the bounded waits on the chunk copies
};

constexpr int kAttnChunk = 128;  // tokens per chunk of the chunk kernels
size_t attn_workspace_bytes(int64_t units, int n_rep, int d, int64_t T);
cudaError_t launch_attention(const AttnArgs& a, cudaStream_t st);

// Sets the message cg_last_error() returns on this host thread; returns code.
int set_error(int code, const char* fmt, ...) __attribute__((format(printf, 2, 3)));

cudaError_t launch_row_encode_simt(const RowArgs& a, cudaStream_t st);
cudaError_t launch_row_move(const MoveArgs& a, cudaStream_t st);
cudaError_t launch_row_decode_simt(const RowArgs& a, cudaStream_t st);
cudaError_t launch_tile_encode_simt(const RowArgs& a, cudaStream_t st);
// Hadamard gauge by fast Walsh-Hadamard transform (no gauge tensor): encode or decode.
cudaError_t launch_hadamard(const RowArgs& a, bool encode, cudaStream_t st);
cudaError_t launch_key_encode_simt(const KeyArgs& a, cudaStream_t st);
cudaError_t launch_key_decode_simt(const KeyArgs& a, cudaStream_t st);
cudaError_t launch_residual_copy(const ResidArgs& a, cudaStream_t st);

// Shared-memory bytes the SIMT kernels need (0 = shape not supported by them).
size_t row_simt_smem(int d, int g);
size_t tile_simt_smem(int d, int g);
size_t key_simt_smem(int d, int g, int Gt, int bits);

}  // namespace cg
