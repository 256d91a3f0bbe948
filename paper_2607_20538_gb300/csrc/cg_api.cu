// cg_api.cu -- the extern "C" boundary of libcodecgauge: argument validation, the
// closed-form byte counts, kernel selection, the device status word and error strings.
// Declarations and the full contract: include/codecgauge.h.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>

#include <cstdlib>

#include "cg_launch.h"
#include "cg_tc.h"
#include "cg_tc_common.cuh"

// The library is built with hidden symbol visibility; only the C ABI is exported.
#define CG_EXPORT __attribute__((visibility("default")))

namespace cg {

__device__ int32_t g_status_word = 0;
__device__ int32_t g_status_taken = 0;

// Reads and clears the status word in one atomic step, on the caller's stream, so a flag
// raised by a kernel on another stream between a read and a clear cannot be lost.
__global__ void status_take_kernel(int32_t* status, int32_t* taken) { *taken = atomicExch(status, 0); }

namespace {

thread_local std::string t_err;

int fail(int code, const char* fmt, ...) __attribute__((format(printf, 2, 3)));
int fail(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_err = buf;
    return code;
}

int cuda_fail(cudaError_t e, const char* what) {
    return fail(CG_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

bool pow2(int v) { return v > 0 && (v & (v - 1)) == 0; }
bool valid_bits(int b) { return b == 2 || b == 3 || b == 4 || b == 6 || b == 8; }
bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Address of this device's status word (looked up once per device).
int status_ptr(int32_t** out) {
    static std::mutex mu;
    static int32_t* ptrs[64] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 64) return fail(CG_EUNSUPPORTED, "device ordinal %d out of range", dev);
    std::lock_guard<std::mutex> lk(mu);
    if (!ptrs[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_status_word);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(status)");
        ptrs[dev] = static_cast<int32_t*>(p);
    }
    *out = ptrs[dev];
    return CG_OK;
}

struct Sizes {
    int64_t tcap, ntiles, nq, nb, pay;
    size_t codes, scales, resid;
    int64_t layer_codes, layer_scales, key_codes_per_bh, key_scales_per_bh, val_codes_per_bh, val_scales_per_bh;
};

bool mul_ok(size_t a, size_t b, size_t* out) {
    if (a && b > SIZE_MAX / a) return false;
    *out = a * b;
    return true;
}

int validate(const cg_shape* sh, const cg_params* p, Sizes* z) {
    if (!sh || !p) return fail(CG_EINVAL, "null shape or params");
    if (sh->L < 1 || sh->B < 1 || sh->H < 1 || sh->T < 0 || sh->d < 1)
        return fail(CG_EINVAL, "shape needs L,B,H,d >= 1 and T >= 0 (got L=%d B=%d H=%d T=%d d=%d)", sh->L, sh->B,
                    sh->H, sh->T, sh->d);
    if (!(sh->d == 32 || sh->d == 64 || sh->d == 128 || sh->d == 256))
        return fail(CG_EUNSUPPORTED, "head dim d=%d: supported d is 32, 64, 128 or 256", sh->d);
    const int g = p->group;
    if (!(g == 8 || g == 16 || g == 32 || g == 64 || g == 128) || sh->d % g)
        return fail(CG_EINVAL, "group=%d: must be one of 8,16,32,64,128 and divide d=%d", g, sh->d);
    if (sh->t0 < 0 || sh->T_cap < 0) return fail(CG_EINVAL, "t0 and T_cap must be >= 0");
    if (p->backend == CG_BLOCK_UNIFORM || p->backend == CG_KIVI || p->backend == CG_BLOCK_TILE) {
        if (!valid_bits(p->bits)) return fail(CG_EINVAL, "bits=%d: must be 2, 3, 4, 6 or 8", p->bits);
        if (!pow2(p->block) || p->block < 8 || sh->d % p->block)
            return fail(CG_EINVAL, "block=%d: must be a power of two >= 8 that divides d=%d", p->block, sh->d);
        if ((p->block * p->bits) % 8) return fail(CG_EINVAL, "block*bits must be a whole number of bytes");
    } else if (p->backend != CG_NONE) {
        return fail(CG_EINVAL, "unknown backend %d", p->backend);
    }
    if (p->backend == CG_BLOCK_TILE) {
        if (sh->t0 % CG_TILE_TOKENS)
            return fail(CG_EUNSUPPORTED, "block-uniform tiles: t0=%d must be a multiple of %d (a call re-encodes "
                        "whole tiles)", sh->t0, CG_TILE_TOKENS);
        if (tile_simt_smem(sh->d, g) == 0)
            return fail(CG_EUNSUPPORTED, "block-uniform tiles: the gauge set of d=%d, group=%d does not fit one CTA",
                        sh->d, g);
    }
    if (p->backend == CG_KIVI) {
        if (p->residual < 0) return fail(CG_EINVAL, "residual must be >= 0");
        if (sh->t0 != 0 || (sh->T_cap != 0 && sh->T_cap != sh->T))
            return fail(CG_EUNSUPPORTED, "KIVI append into a history (t0 > 0 or T_cap != T) is not provided");
        if (key_simt_smem(sh->d, g, p->block, p->bits) > 200 * 1024)
            return fail(CG_EUNSUPPORTED, "KIVI key group of %d tokens x d=%d does not fit one CTA", p->block, sh->d);
    }
    const int64_t tcap = sh->T_cap ? sh->T_cap : (int64_t)sh->t0 + sh->T;
    if ((int64_t)sh->t0 + sh->T > tcap) return fail(CG_EINVAL, "t0 + T = %lld exceeds T_cap = %lld",
                                                     (long long)sh->t0 + sh->T, (long long)tcap);
    if ((int64_t)sh->L * 2 * sh->H > 65535 || (int64_t)sh->L * sh->B * sh->H > 65535)
        return fail(CG_ERANGE, "L*2*H and L*B*H must be <= 65535");
    const int64_t units = (int64_t)sh->L * 2 * sh->B * sh->H;
    z->tcap = tcap;
    z->ntiles = (tcap + CG_TILE_TOKENS - 1) / CG_TILE_TOKENS;
    z->nq = 0;
    z->resid = 0;
    z->layer_codes = z->layer_scales = z->key_codes_per_bh = z->key_scales_per_bh = 0;
    z->val_codes_per_bh = z->val_scales_per_bh = 0;
    size_t rows, tmp;
    if (!mul_ok((size_t)units, (size_t)tcap, &rows)) return fail(CG_ERANGE, "size overflow");
    if (p->backend == CG_NONE) {
        z->nb = 0;
        z->pay = 0;
        if (!mul_ok(rows, (size_t)sh->d * 4, &z->codes)) return fail(CG_ERANGE, "size overflow");
        z->scales = 0;
    } else if (p->backend == CG_BLOCK_UNIFORM || p->backend == CG_BLOCK_TILE) {
        z->nb = sh->d / p->block;
        z->pay = (int64_t)p->block * p->bits / 8;
        if (!mul_ok(rows, (size_t)(z->nb * z->pay), &z->codes)) return fail(CG_ERANGE, "size overflow");
        const size_t nranges = p->backend == CG_BLOCK_UNIFORM ? rows : (size_t)units * (size_t)z->ntiles;
        if (!mul_ok(nranges, (size_t)z->nb * 4, &z->scales)) return fail(CG_ERANGE, "size overflow");
    } else {
        const int64_t Gt = p->block, d = sh->d;
        z->nq = kivi_nq(sh->T, p->residual, Gt);
        z->nb = d / Gt;
        z->pay = Gt * p->bits / 8;
        z->key_codes_per_bh = (z->nq / Gt) * d * z->pay;
        z->val_codes_per_bh = z->nq * z->nb * z->pay;
        z->key_scales_per_bh = (z->nq / Gt) * d;
        z->val_scales_per_bh = z->nq * z->nb;
        const int64_t BH = (int64_t)sh->B * sh->H;
        z->layer_codes = BH * (z->key_codes_per_bh + z->val_codes_per_bh);
        z->layer_scales = BH * (z->key_scales_per_bh + z->val_scales_per_bh);
        if (!mul_ok((size_t)sh->L, (size_t)z->layer_codes, &z->codes)) return fail(CG_ERANGE, "size overflow");
        if (!mul_ok((size_t)sh->L, (size_t)z->layer_scales * 4, &z->scales)) return fail(CG_ERANGE, "size overflow");
        if (!mul_ok((size_t)units, (size_t)(sh->T - z->nq) * d * 2, &z->resid)) return fail(CG_ERANGE, "size overflow");
    }
    if (!mul_ok(rows, (size_t)sh->d * 2, &tmp)) return fail(CG_ERANGE, "size overflow");
    return CG_OK;
}

// Row map for the block-uniform / none history layout [L][2][B][H][T_cap][...]. With
// tile = true the scales are per 16-token tile, [L][2][B][H][ceil(T_cap/16)][d/block]
// (t0 is then a multiple of 16).
void bu_maps(const cg_shape* sh, const Sizes& z, int64_t rowbytes, int64_t rowscales, RowMap* cm, RowMap* sm,
             bool tile = false) {
    const int64_t tc = z.tcap;
    cm->sT = rowbytes;
    cm->sH = tc * rowbytes;
    cm->sB = (int64_t)sh->H * cm->sH;
    cm->sS = (int64_t)sh->B * cm->sB;
    cm->sL = 2 * cm->sS;
    cm->base = (int64_t)sh->t0 * rowbytes;
    cm->tshift = 0;
    const int64_t nranges = tile ? z.ntiles : tc;
    sm->sT = rowscales;
    sm->sH = nranges * rowscales;
    sm->sB = (int64_t)sh->H * sm->sH;
    sm->sS = (int64_t)sh->B * sm->sB;
    sm->sL = 2 * sm->sS;
    sm->tshift = tile ? 4 : 0;
    sm->base = (int64_t)(sh->t0 >> sm->tshift) * rowscales;
}

// Row map for KIVI keys seen as rows of the key tensor: codes [B][H][n_q/Gt][d][pay] at the
// start of each layer, addressed per token so that a key group's first token t0 (a multiple
// of Gt) lands on the group's first channel stream; scales [B][H][n_q/Gt][d] likewise.
void kivi_key_maps(const cg_shape* sh, const cg_params* p, const Sizes& z, RowMap* cm, RowMap* sm) {
    const int64_t Gt = p->block;
    cm->base = 0;
    cm->sL = z.layer_codes;
    cm->sS = 0;
    cm->sH = z.key_codes_per_bh;
    cm->sB = (int64_t)sh->H * cm->sH;
    cm->sT = (int64_t)sh->d * z.pay / Gt;
    cm->tshift = 0;
    sm->base = 0;
    sm->tshift = 0;
    sm->sL = z.layer_scales;
    sm->sS = 0;
    sm->sH = z.key_scales_per_bh;
    sm->sB = (int64_t)sh->H * sm->sH;
    sm->sT = (int64_t)sh->d / Gt;
}

// Row map for KIVI values: codes [B][H][n_q][d/blk][pay] after the layer's key part.
void kivi_value_maps(const cg_shape* sh, const Sizes& z, RowMap* cm, RowMap* sm) {
    const int64_t BH = (int64_t)sh->B * sh->H;
    cm->sT = z.nb * z.pay;
    cm->sH = z.val_codes_per_bh;
    cm->sB = (int64_t)sh->H * cm->sH;
    cm->sS = 0;
    cm->sL = z.layer_codes;
    cm->base = BH * z.key_codes_per_bh;
    cm->tshift = 0;
    sm->sT = z.nb;
    sm->tshift = 0;
    sm->sH = z.val_scales_per_bh;
    sm->sB = (int64_t)sh->H * sm->sH;
    sm->sS = 0;
    sm->sL = z.layer_scales;
    sm->base = BH * z.key_scales_per_bh;
}

// Limit of each bounded pipeline wait in the tensor-core kernels: 4 s, or the value of the
// environment variable CODECGAUGE_PIPE_WAIT_NS (a diagnostic knob: a tiny limit makes the
// waits give up, which exercises the CG_FLAG_PIPE_TIMEOUT path without any fault). The
// drains of copies already issued always keep the 4 s limit.
uint64_t pipe_wait_ns() {
    const char* v = getenv("CODECGAUGE_PIPE_WAIT_NS");
    if (!v || !*v) return tc::kWaitLimitNs;
    char* end = nullptr;
    const unsigned long long n = strtoull(v, &end, 10);
    return (end && *end == 0 && n <= tc::kWaitLimitNs) ? (uint64_t)n : tc::kWaitLimitNs;
}

RowArgs row_args(const cg_shape* sh, const cg_params* p, int32_t* status) {
    RowArgs a{};
    a.wait_ns = pipe_wait_ns();
    a.status = status;
    a.L = sh->L;
    a.B = sh->B;
    a.H = sh->H;
    a.d = sh->d;
    a.g = p->group;
    a.bits = p->bits;
    a.blk = p->block;
    a.s_lo = 0;
    a.s_n = 2;
    a.T_x = sh->T;
    a.t_count = sh->T;
    a.none_mode = p->backend == CG_NONE;
    return a;
}

KeyArgs key_args(const cg_shape* sh, const cg_params* p, const Sizes& z, int32_t* status) {
    KeyArgs k{};
    k.status = status;
    k.L = sh->L;
    k.B = sh->B;
    k.H = sh->H;
    k.d = sh->d;
    k.g = p->group;
    k.bits = p->bits;
    k.Gt = p->block;
    k.T = sh->T;
    k.nq = z.nq;
    k.layer_codes = z.layer_codes;
    k.layer_scales = z.layer_scales;
    k.key_codes_per_bh = z.key_codes_per_bh;
    k.key_scales_per_bh = z.key_scales_per_bh;
    return k;
}

// KIVI quantized part, encode: the t_count tokens (whole key groups) in rows [0, t_count) of
// x [L][2][B][H][T_x][d] become quantized tokens [tok0, tok0 + t_count) of the layout z (tok0 a
// multiple of the group length). Keys on tensor cores where eligible, else on CUDA cores;
// values through the row kernels. Sets *what to the failing launch.
cudaError_t kivi_encode_groups(const cg_shape* sh, const cg_params* p, const Sizes& z, const uint16_t* x,
                               int64_t T_x, int64_t t_count, int64_t tok0, const float* G, uint8_t* codes,
                               uint32_t* scales, int32_t* status, cudaStream_t st, const char** what) {
    const int64_t Gt = p->block, gi = tok0 / Gt;
    RowArgs a = row_args(sh, p, status);
    a.x = x;
    a.G = G;
    a.codes = codes;
    a.scales = scales;
    a.T_x = T_x;
    a.t_count = t_count;
    RowArgs ka = a;  // keys: s = 0, one block per channel and key group
    ka.s_lo = 0;
    ka.s_n = 1;
    kivi_key_maps(sh, p, z, &ka.cmap, &ka.smap);
    ka.cmap.base += gi * sh->d * z.pay;
    ka.smap.base += gi * sh->d;
    cudaError_t e;
    if (tc_key_encode_eligible(ka)) {
        e = tc_launch_key_encode(ka, st);
    } else {
        KeyArgs k = key_args(sh, p, z, status);
        k.x = x;
        k.T = T_x;
        k.nq = t_count;
        k.G = G;
        k.codes = codes + gi * sh->d * z.pay;
        k.scales = scales + gi * sh->d;
        e = launch_key_encode_simt(k, st);
    }
    if (e != cudaSuccess) {
        *what = "KIVI key encode launch";
        return e;
    }
    a.s_lo = 1;
    a.s_n = 1;
    kivi_value_maps(sh, z, &a.cmap, &a.smap);
    a.cmap.base += tok0 * z.nb * z.pay;
    a.smap.base += tok0 * z.nb;
    e = tc_row_encode_eligible(a) ? tc_launch_row_encode(a, st) : launch_row_encode_simt(a, st);
    if (e != cudaSuccess) *what = "KIVI value encode launch";
    return e;
}

// KIVI quantized part, decode: quantized tokens [0, t_count) of the layout z into rows
// [0, t_count) of out [L][2][B][H][T_x][d].
cudaError_t kivi_decode_groups(const cg_shape* sh, const cg_params* p, const Sizes& z, const uint8_t* codes,
                               const uint32_t* scales, const float* G, uint16_t* out, int64_t T_x, int64_t t_count,
                               int32_t* status, cudaStream_t st, const char** what) {
    RowArgs a = row_args(sh, p, status);
    a.out = out;
    a.G = G;
    a.codes = const_cast<uint8_t*>(codes);
    a.scales = const_cast<uint32_t*>(scales);
    a.T_x = T_x;
    a.t_count = t_count;
    RowArgs ka = a;  // keys: s = 0, one 128-token group per tile
    ka.s_lo = 0;
    ka.s_n = 1;
    kivi_key_maps(sh, p, z, &ka.cmap, &ka.smap);
    cudaError_t e;
    if (tc_key_decode_eligible(ka)) {
        e = tc_launch_key_decode(ka, st);
    } else {
        KeyArgs k = key_args(sh, p, z, status);
        k.out = out;
        k.T = T_x;
        k.nq = t_count;
        k.G = G;
        k.codes = a.codes;
        k.scales = a.scales;
        e = launch_key_decode_simt(k, st);
    }
    if (e != cudaSuccess) {
        *what = "KIVI key decode launch";
        return e;
    }
    a.s_lo = 1;
    a.s_n = 1;
    kivi_value_maps(sh, z, &a.cmap, &a.smap);
    e = tc_row_decode_eligible(a) ? tc_launch_row_decode(a, st) : launch_row_decode_simt(a, st);
    if (e != cudaSuccess) *what = "KIVI value decode launch";
    return e;
}

// Sizes of a KIVI stream of capacity sh->T_cap: the CG_KIVI layout at T_cap tokens, the ring
// of W = residual + block slots and the staging workspace of one key group per unit.
struct StreamSizes {
    Sizes z;
    int64_t W;
    size_t ring, workspace;
};

int validate_stream(const cg_shape* sh, const cg_params* p, StreamSizes* ss) {
    if (!sh || !p) return fail(CG_EINVAL, "null shape or params");
    if (p->backend != CG_KIVI) return fail(CG_EINVAL, "KIVI streaming needs backend CG_KIVI");
    if (sh->T_cap < 1 || sh->t0 < 0 || sh->T < 0 || (int64_t)sh->t0 + sh->T > sh->T_cap)
        return fail(CG_EINVAL, "KIVI stream: needs T_cap >= 1 and 0 <= t0, t0 + T <= T_cap (t0=%d T=%d T_cap=%d)",
                    sh->t0, sh->T, sh->T_cap);
    cg_shape cap = *sh;
    cap.t0 = 0;
    cap.T = sh->T_cap;
    cap.T_cap = 0;
    int rc = validate(&cap, p, &ss->z);
    if (rc) return rc;
    ss->W = (int64_t)p->residual + p->block;
    const size_t units = (size_t)sh->L * 2 * sh->B * sh->H;
    size_t row = (size_t)sh->d * 2;
    if (!mul_ok(units * row, (size_t)ss->W, &ss->ring)) return fail(CG_ERANGE, "size overflow");
    if (!mul_ok(units * row, (size_t)p->block, &ss->workspace)) return fail(CG_ERANGE, "size overflow");
    return CG_OK;
}

MoveArgs move_args(const cg_shape* sh, int64_t W) {
    MoveArgs m{};
    m.units = (int64_t)sh->L * 2 * sh->B * sh->H;
    m.d = sh->d;
    m.W = W;
    return m;
}

}  // namespace

int set_error(int code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    t_err = buf;
    return code;
}

}  // namespace cg

using namespace cg;

extern "C" {

CG_EXPORT const char* cg_last_error(void) { return t_err.c_str(); }

CG_EXPORT int cg_packed_bytes(const cg_shape* shape, const cg_params* params, size_t* codes_bytes, size_t* scales_bytes,
                    size_t* residual_bytes) {
    t_err.clear();
    Sizes z;
    int rc = validate(shape, params, &z);
    if (rc) return rc;
    if (codes_bytes) *codes_bytes = z.codes;
    if (scales_bytes) *scales_bytes = z.scales;
    if (residual_bytes) *residual_bytes = z.resid;
    return CG_OK;
}

CG_EXPORT int cg_encode(const cg_shape* shape, const cg_params* params, const void* kv_bf16, const float* gauges,
              void* out_codes, void* out_scales, void* out_residual, void* stream) {
    t_err.clear();
    Sizes z;
    int rc = validate(shape, params, &z);
    if (rc) return rc;
    const bool kivi = params->backend == CG_KIVI, none = params->backend == CG_NONE;
    const bool tile = params->backend == CG_BLOCK_TILE;
    if (shape->T == 0) return CG_OK;
    if (!kv_bf16 || !gauges) return fail(CG_EINVAL, "null kv or gauges pointer");
    if (z.codes && !out_codes) return fail(CG_EINVAL, "null out_codes");
    if (!none && z.scales && !out_scales) return fail(CG_EINVAL, "null out_scales");
    if (kivi && z.resid && !out_residual) return fail(CG_EINVAL, "null out_residual");
    if (!aligned16(kv_bf16) || !aligned16(gauges) || !aligned16(out_codes) || !aligned16(out_scales) ||
        !aligned16(out_residual))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    RowArgs a = row_args(shape, params, status);
    a.x = static_cast<const uint16_t*>(kv_bf16);
    a.G = gauges;
    a.codes = static_cast<uint8_t*>(out_codes);
    a.scales = static_cast<uint32_t*>(out_scales);
    if (tile) {
        bu_maps(shape, z, z.nb * z.pay, z.nb, &a.cmap, &a.smap, true);
        e = launch_tile_encode_simt(a, st);
        if (e != cudaSuccess) return cuda_fail(e, "tile encode launch");
        return CG_OK;
    }
    if (!kivi) {
        bu_maps(shape, z, none ? (int64_t)shape->d * 4 : z.nb * z.pay, z.nb, &a.cmap, &a.smap);
        if (!none && tc_row_encode_eligible(a)) {
            e = tc_launch_row_encode(a, st);
        } else {
            e = launch_row_encode_simt(a, st);
        }
        if (e != cudaSuccess) return cuda_fail(e, "row encode launch");
        return CG_OK;
    }
    if (z.nq > 0) {
        const char* what = "";
        e = kivi_encode_groups(shape, params, z, a.x, shape->T, z.nq, 0, gauges, a.codes, a.scales, status, st, &what);
        if (e != cudaSuccess) return cuda_fail(e, what);
    }
    if (shape->T - z.nq > 0) {
        ResidArgs r{};
        r.src = a.x;
        r.dst = static_cast<uint16_t*>(out_residual);
        r.units = (int64_t)shape->L * 2 * shape->B * shape->H;
        r.T = shape->T;
        r.nq = z.nq;
        r.d = shape->d;
        r.to_residual = 1;
        e = launch_residual_copy(r, st);
        if (e != cudaSuccess) return cuda_fail(e, "KIVI residual copy launch");
    }
    return CG_OK;
}

CG_EXPORT int cg_decode(const cg_shape* shape, const cg_params* params, const void* codes, const void* scales,
              const void* residual, const float* gauges, void* out_kv_bf16, void* stream) {
    t_err.clear();
    Sizes z;
    int rc = validate(shape, params, &z);
    if (rc) return rc;
    const bool kivi = params->backend == CG_KIVI, none = params->backend == CG_NONE;
    const bool tile = params->backend == CG_BLOCK_TILE;
    if (shape->T == 0) return CG_OK;
    if (!out_kv_bf16 || !gauges) return fail(CG_EINVAL, "null output or gauges pointer");
    if (z.codes && !codes) return fail(CG_EINVAL, "null codes");
    if (!none && z.scales && !scales) return fail(CG_EINVAL, "null scales");
    if (kivi && z.resid && !residual) return fail(CG_EINVAL, "null residual");
    if (!aligned16(codes) || !aligned16(scales) || !aligned16(residual) || !aligned16(gauges) ||
        !aligned16(out_kv_bf16))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaSuccess;
    RowArgs a = row_args(shape, params, status);
    a.out = static_cast<uint16_t*>(out_kv_bf16);
    a.G = gauges;
    a.codes = const_cast<uint8_t*>(static_cast<const uint8_t*>(codes));
    a.scales = const_cast<uint32_t*>(static_cast<const uint32_t*>(scales));
    if (!kivi) {
        bu_maps(shape, z, none ? (int64_t)shape->d * 4 : z.nb * z.pay, z.nb, &a.cmap, &a.smap, tile);
        if (!none && tc_row_decode_eligible(a)) {
            e = tc_launch_row_decode(a, st);
        } else {
            e = launch_row_decode_simt(a, st);
        }
        if (e != cudaSuccess) return cuda_fail(e, "row decode launch");
        return CG_OK;
    }
    if (z.nq > 0) {
        const char* what = "";
        e = kivi_decode_groups(shape, params, z, a.codes, a.scales, gauges, a.out, shape->T, z.nq, status, st, &what);
        if (e != cudaSuccess) return cuda_fail(e, what);
    }
    if (shape->T - z.nq > 0) {
        ResidArgs r{};
        r.src = static_cast<const uint16_t*>(residual);
        r.dst = a.out;
        r.units = (int64_t)shape->L * 2 * shape->B * shape->H;
        r.T = shape->T;
        r.nq = z.nq;
        r.d = shape->d;
        r.to_residual = 0;
        e = launch_residual_copy(r, st);
        if (e != cudaSuccess) return cuda_fail(e, "KIVI residual copy launch");
    }
    return CG_OK;
}

CG_EXPORT int cg_encode_hadamard(const cg_shape* shape, const cg_params* params, const void* kv_bf16,
                                 void* out_codes, void* out_scales, void* stream) {
    t_err.clear();
    Sizes z;
    int rc = validate(shape, params, &z);
    if (rc) return rc;
    if (params->backend != CG_BLOCK_UNIFORM)
        return fail(CG_EUNSUPPORTED, "the Hadamard transform path encodes block-uniform rows");
    if (shape->T == 0) return CG_OK;
    if (!kv_bf16 || !out_codes || !out_scales) return fail(CG_EINVAL, "null kv, codes or scales pointer");
    if (!aligned16(kv_bf16) || !aligned16(out_codes) || !aligned16(out_scales))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    RowArgs a = row_args(shape, params, status);
    a.x = static_cast<const uint16_t*>(kv_bf16);
    a.codes = static_cast<uint8_t*>(out_codes);
    a.scales = static_cast<uint32_t*>(out_scales);
    bu_maps(shape, z, z.nb * z.pay, z.nb, &a.cmap, &a.smap);
    cudaError_t e = launch_hadamard(a, true, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "Hadamard encode launch");
    return CG_OK;
}

CG_EXPORT int cg_decode_hadamard(const cg_shape* shape, const cg_params* params, const void* codes,
                                 const void* scales, void* out_kv_bf16, void* stream) {
    t_err.clear();
    Sizes z;
    int rc = validate(shape, params, &z);
    if (rc) return rc;
    if (params->backend != CG_BLOCK_UNIFORM)
        return fail(CG_EUNSUPPORTED, "the Hadamard transform path decodes block-uniform rows");
    if (shape->T == 0) return CG_OK;
    if (!codes || !scales || !out_kv_bf16) return fail(CG_EINVAL, "null codes, scales or output pointer");
    if (!aligned16(codes) || !aligned16(scales) || !aligned16(out_kv_bf16))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    RowArgs a = row_args(shape, params, status);
    a.out = static_cast<uint16_t*>(out_kv_bf16);
    a.codes = const_cast<uint8_t*>(static_cast<const uint8_t*>(codes));
    a.scales = const_cast<uint32_t*>(static_cast<const uint32_t*>(scales));
    bu_maps(shape, z, z.nb * z.pay, z.nb, &a.cmap, &a.smap);
    cudaError_t e = launch_hadamard(a, false, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "Hadamard decode launch");
    return CG_OK;
}

CG_EXPORT int cg_kivi_stream_bytes(const cg_shape* shape, const cg_params* params, size_t* codes_bytes,
                                   size_t* scales_bytes, size_t* ring_bytes, size_t* workspace_bytes) {
    t_err.clear();
    StreamSizes ss;
    int rc = validate_stream(shape, params, &ss);
    if (rc) return rc;
    if (codes_bytes) *codes_bytes = ss.z.codes;
    if (scales_bytes) *scales_bytes = ss.z.scales;
    if (ring_bytes) *ring_bytes = ss.ring;
    if (workspace_bytes) *workspace_bytes = ss.workspace;
    return CG_OK;
}

CG_EXPORT int cg_kivi_append(const cg_shape* shape, const cg_params* params, const void* kv_new_bf16,
                             const float* gauges, void* codes, void* scales, void* ring, void* workspace,
                             size_t workspace_bytes, void* stream) {
    t_err.clear();
    StreamSizes ss;
    int rc = validate_stream(shape, params, &ss);
    if (rc) return rc;
    const int64_t t0 = shape->t0, T = shape->T, Gt = params->block, R = params->residual;
    if (t0 > 0 && T > Gt)
        return fail(CG_EUNSUPPORTED, "KIVI stream: an append after the first call carries at most block=%d tokens "
                    "(got T=%d)", params->block, shape->T);
    if (T == 0) return CG_OK;
    const int64_t nq_old = kivi_nq(t0, R, Gt), nq_new = kivi_nq(t0 + T, R, Gt);
    const bool stage = t0 > 0 && nq_new > nq_old;
    if (!kv_new_bf16 || !gauges || !ring) return fail(CG_EINVAL, "null kv, gauges or ring pointer");
    if (nq_new > nq_old && (!codes || !scales)) return fail(CG_EINVAL, "null codes or scales");
    if (stage && (!workspace || workspace_bytes < ss.workspace))
        return fail(CG_EINVAL, "this append completes a key group: workspace needs %zu bytes (got %zu)", ss.workspace,
                    workspace ? workspace_bytes : (size_t)0);
    if (!aligned16(kv_new_bf16) || !aligned16(gauges) || !aligned16(codes) || !aligned16(scales) ||
        !aligned16(ring) || !aligned16(workspace))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const uint16_t* x = static_cast<const uint16_t*>(kv_new_bf16);
    uint16_t* rg = static_cast<uint16_t*>(ring);
    cudaError_t e = cudaSuccess;
    const char* what = "";
    if (nq_new > nq_old) {
        if (stage) {
            // the completed group's tokens, from the ring (t < t0) and the new input, staged
            // as a dense [L][2][B][H][block][d] input
            MoveArgs m = move_args(shape, ss.W);
            m.ring_src = rg;
            m.x = x;
            m.T_x = T;
            m.x_t0 = t0;
            m.src_split = t0;
            m.t_lo = nq_old;
            m.t_hi = nq_new;
            m.dst = static_cast<uint16_t*>(workspace);
            m.dst_T = Gt;
            m.dst_t0 = nq_old;
            if ((e = launch_row_move(m, st)) != cudaSuccess) return cuda_fail(e, "KIVI stream staging launch");
            e = kivi_encode_groups(shape, params, ss.z, static_cast<const uint16_t*>(workspace), Gt, Gt, nq_old,
                                   gauges, static_cast<uint8_t*>(codes), static_cast<uint32_t*>(scales), status, st,
                                   &what);
        } else {
            e = kivi_encode_groups(shape, params, ss.z, x, T, nq_new, 0, gauges, static_cast<uint8_t*>(codes),
                                   static_cast<uint32_t*>(scales), status, st, &what);
        }
        if (e != cudaSuccess) return cuda_fail(e, what);
    }
    // new tokens that stay raw go to their ring slots (after the staging read above)
    MoveArgs m = move_args(shape, ss.W);
    m.x = x;
    m.T_x = T;
    m.x_t0 = t0;
    m.src_split = 0;
    m.t_lo = nq_new > t0 ? nq_new : t0;
    m.t_hi = t0 + T;
    m.dst = rg;
    m.dst_ring = 1;
    if ((e = launch_row_move(m, st)) != cudaSuccess) return cuda_fail(e, "KIVI stream ring launch");
    return CG_OK;
}

CG_EXPORT int cg_kivi_stream_decode(const cg_shape* shape, const cg_params* params, const void* codes,
                                    const void* scales, const void* ring, const float* gauges, void* out_kv_bf16,
                                    void* stream) {
    t_err.clear();
    StreamSizes ss;
    int rc = validate_stream(shape, params, &ss);
    if (rc) return rc;
    if (shape->t0 != 0) return fail(CG_EUNSUPPORTED, "KIVI stream decode reads the whole history: t0 must be 0");
    const int64_t T = shape->T, nq = kivi_nq(T, params->residual, params->block);
    if (T == 0) return CG_OK;
    if (!out_kv_bf16 || !gauges || !ring) return fail(CG_EINVAL, "null output, gauges or ring pointer");
    if (nq > 0 && (!codes || !scales)) return fail(CG_EINVAL, "null codes or scales");
    if (!aligned16(codes) || !aligned16(scales) || !aligned16(ring) || !aligned16(gauges) || !aligned16(out_kv_bf16))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    uint16_t* out = static_cast<uint16_t*>(out_kv_bf16);
    cudaError_t e = cudaSuccess;
    if (nq > 0) {
        const char* what = "";
        e = kivi_decode_groups(shape, params, ss.z, static_cast<const uint8_t*>(codes),
                               static_cast<const uint32_t*>(scales), gauges, out, T, nq, status, st, &what);
        if (e != cudaSuccess) return cuda_fail(e, what);
    }
    MoveArgs m = move_args(shape, ss.W);
    m.ring_src = static_cast<const uint16_t*>(ring);
    m.src_split = T;  // every raw token comes from the ring
    m.t_lo = nq;
    m.t_hi = T;
    m.dst = out;
    m.dst_T = T;
    m.dst_t0 = 0;
    if ((e = launch_row_move(m, st)) != cudaSuccess) return cuda_fail(e, "KIVI stream window launch");
    return CG_OK;
}

namespace {

// Attention arguments common to the size query and the call.
int validate_attention(const cg_shape* sh, const cg_params* p, int n_rep, Sizes* z) {
    int rc = validate(sh, p, z);
    if (rc) return rc;
    if (p->backend != CG_BLOCK_UNIFORM && p->backend != CG_BLOCK_TILE)
        return fail(CG_EUNSUPPORTED, "attention reads block-uniform caches (rows or tiles)");
    if (sh->d != 128) return fail(CG_EUNSUPPORTED, "attention: head dim d=%d (d = 128 is provided)", sh->d);
    if (!(p->block == 32 || p->block == 64 || p->block == 128))
        return fail(CG_EUNSUPPORTED, "attention: block=%d (32, 64 or 128 are provided)", p->block);
    if (!(n_rep == 1 || n_rep == 2 || n_rep == 4 || n_rep == 8))
        return fail(CG_EINVAL, "n_rep=%d: query heads per KV head must be 1, 2, 4 or 8", n_rep);
    if (sh->T < 1) return fail(CG_EINVAL, "attention needs T >= 1 tokens");
    return CG_OK;
}

}  // namespace

CG_EXPORT int cg_attention_workspace_bytes(const cg_shape* shape, const cg_params* params, int n_rep,
                                           size_t* workspace_bytes) {
    t_err.clear();
    Sizes z;
    int rc = validate_attention(shape, params, n_rep, &z);
    if (rc) return rc;
    if (workspace_bytes)
        *workspace_bytes = attn_workspace_bytes((int64_t)shape->L * shape->B * shape->H, n_rep, shape->d, shape->T);
    return CG_OK;
}

CG_EXPORT int cg_attention(const cg_shape* shape, const cg_params* params, int n_rep, float scale, const void* q_bf16,
                           const void* codes, const void* scales, const float* gauges, float* out,
                           void* workspace, size_t workspace_bytes, void* stream) {
    t_err.clear();
    Sizes z;
    int rc = validate_attention(shape, params, n_rep, &z);
    if (rc) return rc;
    if (!(scale == scale) || scale == INFINITY || scale == -INFINITY)
        return fail(CG_EINVAL, "softmax scale must be finite");
    if (!q_bf16 || !codes || !scales || !gauges || !out || !workspace)
        return fail(CG_EINVAL, "null q, codes, scales, gauges, out or workspace pointer");
    const size_t need = attn_workspace_bytes((int64_t)shape->L * shape->B * shape->H, n_rep, shape->d, shape->T);
    if (workspace_bytes < need) return fail(CG_EINVAL, "workspace needs %zu bytes (got %zu)", need, workspace_bytes);
    if (!aligned16(q_bf16) || !aligned16(codes) || !aligned16(scales) || !aligned16(gauges) || !aligned16(out) ||
        !aligned16(workspace))
        return fail(CG_EINVAL, "pointers must be 16-byte aligned");
    int32_t* status = nullptr;
    if ((rc = status_ptr(&status))) return rc;
    AttnArgs a{};
    a.q = static_cast<const uint16_t*>(q_bf16);
    a.G = gauges;
    a.codes = static_cast<const uint8_t*>(codes);
    a.scales = static_cast<const uint32_t*>(scales);
    bu_maps(shape, z, z.nb * z.pay, z.nb, &a.cmap, &a.smap, params->backend == CG_BLOCK_TILE);
    const int64_t units = (int64_t)shape->L * shape->B * shape->H;
    a.qrot = static_cast<float*>(workspace);
    a.part = reinterpret_cast<float*>(static_cast<unsigned char*>(workspace) +
                                      ((size_t)units * n_rep * shape->d * 4 + 255) / 256 * 256);
    a.out = out;
    a.L = shape->L;
    a.B = shape->B;
    a.H = shape->H;
    a.d = shape->d;
    a.g = params->group;
    a.bits = params->bits;
    a.blk = params->block;
    a.n_rep = n_rep;
    a.T = shape->T;
    a.n_chunks = (int)((shape->T + kAttnChunk - 1) / kAttnChunk);
    a.scale = scale;
    a.status = status;
    a.wait_ns = pipe_wait_ns();
    cudaError_t e = launch_attention(a, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "attention launch");
    return CG_OK;
}

CG_EXPORT int cg_get_status(void* stream, int32_t* device_flags) {
    t_err.clear();
    if (!device_flags) return fail(CG_EINVAL, "null device_flags");
    int32_t* status = nullptr;
    int rc = status_ptr(&status);
    if (rc) return rc;
    int32_t* taken = nullptr;
    cudaError_t e = cudaGetSymbolAddress(reinterpret_cast<void**>(&taken), g_status_taken);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(status slot)");
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    status_take_kernel<<<1, 1, 0, st>>>(status, taken);
    e = cudaGetLastError();
    if (e != cudaSuccess) return cuda_fail(e, "status read launch");
    int32_t v = 0;
    e = cudaMemcpyAsync(&v, taken, sizeof v, cudaMemcpyDeviceToHost, st);
    if (e != cudaSuccess) return cuda_fail(e, "read status");
    e = cudaStreamSynchronize(st);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    *device_flags = v;
    return CG_OK;
}

}  // extern "C"
