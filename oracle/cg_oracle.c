/*
 * cg_oracle.c -- CPU oracle for the Codec-Gauge encode/decode path (arxiv 2607.20538).
 *
 * TEST INFRASTRUCTURE ONLY. Only the tests, the smoke check and the benchmark's CPU
 * baseline leg load this library. The product path (libcodecgauge) never calls it, and
 * the two share no source, header, table or helper.
 *
 * Plain, slow and direct: every function writes out the definition it cites, with no
 * blocking, fusion or reordering. Arithmetic precision:
 *   - gauge-space values z are fp32 (Sec. 4.3: the paper hands the backend FP32
 *     transformed tensors); each z_i = sum_j G[i][j] x_j (Sec. 3, Z = G X) is summed in a
 *     fixed order so that fp32 ranges are reproducible: pairwise summation of the fp32
 *     products p_j = G[i][j] * x_j, S(a, b) = S(a, m) + S(m, b) with m = (a + b) / 2 and
 *     S(j, j + 1) = p_j, each product and each sum rounded to fp32;
 *   - the quantizer (Sec. 4.3 "asymmetric min/max") works in fp32 with fp16 scale/zero;
 *   - decode (Sec. 3: Zhat = D(B_c), Xhat = G^{-1} Zhat, and G^{-1} = G^T by Sec. 4.1)
 *     is evaluated in fp64 and returned as fp64.
 * Compiled without fast-math and with -ffp-contract=off, so every operation below is
 * the single IEEE operation it reads as.
 *
 * Status of the pins (tests/test_oracle_pins.py, tests/test_oracle_tile_pins.py,
 * tests/test_oracle_stream_pins.py, tests/test_oracle_attention_pins.py): every
 * exported function is pinned against closed forms, brute force, worked examples or
 * library routines; none is "parity unpinned".
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ---- interface structs (same field layout as the library's; restated here) ---- */
typedef struct { int32_t L, B, H, T, d, t0, T_cap; } cgo_shape;
typedef struct { int32_t backend, group, bits, block, residual; } cgo_params;

enum { CGO_BU = 0, CGO_KIVI = 1, CGO_NONE = 2, CGO_BU_TILE = 3 };
/* Block-uniform tile height: the paper partitions the token axis into blocks of T_b = 16
 * tokens (Sec. 4.2, the value used for every checkpoint) and gives block-uniform one range
 * per T_b x d_l block (Sec. 4.3). */
enum { CGO_TILE_TOKENS = 16 };
enum { CGO_OK = 0, CGO_EINVAL = -1, CGO_EUNSUP = -2, CGO_ERANGE = -4 };
enum { CGO_FLAG_NONFINITE = 1, CGO_FLAG_FP16_OVERFLOW = 2 };

/* ------------------------------------------------------------------------------ */
/* IEEE conversions, written from the format definitions                          */
/* ------------------------------------------------------------------------------ */

/* binary32 -> binary16, round to nearest, ties to even (IEEE 754 default rounding). */
uint16_t cgo_f32_to_f16(float f)
{
    uint32_t x;
    memcpy(&x, &f, 4);
    uint32_t sign = (x >> 16) & 0x8000u;
    uint32_t e32 = (x >> 23) & 0xffu;
    uint32_t man = x & 0x7fffffu;
    if (e32 == 0xffu) return (uint16_t)(sign | 0x7c00u | (man ? 0x200u : 0u));
    if (e32 == 0u) return (uint16_t)sign; /* fp32 subnormals are far below half's range */
    uint32_t sig = man | 0x800000u;       /* 24-bit significand, value = sig * 2^(e32-150) */
    int32_t e16 = (int32_t)e32 - 127 + 15;
    if (e16 >= 1) {
        /* normal half: keep 11 significant bits, drop 13 */
        uint32_t q = sig >> 13, rem = sig & 0x1fffu;
        if (rem > 0x1000u || (rem == 0x1000u && (q & 1u))) q++;
        if (q == 0x800u) { q = 0x400u; e16++; }
        if (e16 >= 31) return (uint16_t)(sign | 0x7c00u);
        return (uint16_t)(sign | ((uint32_t)e16 << 10) | (q & 0x3ffu));
    }
    /* subnormal half: unit 2^-24, q = sig * 2^(e32-150+24) = sig >> (126 - e32) */
    uint32_t shift = 126u - e32; /* >= 14 here */
    if (shift > 25u) return (uint16_t)sign;
    uint32_t q = sig >> shift, rem = sig & ((1u << shift) - 1u), half = 1u << (shift - 1u);
    if (rem > half || (rem == half && (q & 1u))) q++;
    return (uint16_t)(sign | q); /* q == 0x400 lands on the smallest normal exactly */
}

float cgo_f16_to_f32(uint16_t h)
{
    uint32_t sign = (uint32_t)(h & 0x8000u) << 16;
    uint32_t e = (h >> 10) & 0x1fu, m = h & 0x3ffu;
    float v;
    if (e == 0u) {
        v = ldexpf((float)m, -24);
    } else if (e == 31u) {
        v = m ? NAN : INFINITY;
    } else {
        v = ldexpf((float)(m | 0x400u), (int)e - 25);
    }
    uint32_t bits;
    memcpy(&bits, &v, 4);
    bits |= sign;
    memcpy(&v, &bits, 4);
    return v;
}

float cgo_bf16_to_f32(uint16_t b)
{
    uint32_t bits = (uint32_t)b << 16;
    float v;
    memcpy(&v, &bits, 4);
    return v;
}

/* ------------------------------------------------------------------------------ */
/* Sizes and the KIVI split                                                        */
/* ------------------------------------------------------------------------------ */

static int valid_bits(int b) { return b == 2 || b == 3 || b == 4 || b == 6 || b == 8; }

/* KIVI split (Sec. 4.3 KIVI-style path with a full-precision window): quantized tokens
 * form whole token groups of length `block`; the newest T - n_q >= residual tokens stay
 * raw. */
int64_t cgo_kivi_nq(int64_t T, int64_t R, int64_t Gt)
{
    if (T <= R) return 0;
    return ((T - R) / Gt) * Gt;
}

static int check_args(const cgo_shape* s, const cgo_params* p)
{
    if (!s || !p) return CGO_EINVAL;
    if (s->L < 1 || s->B < 1 || s->H < 1 || s->T < 0 || s->d < 1) return CGO_EINVAL;
    int g = p->group;
    if (!(g == 8 || g == 16 || g == 32 || g == 64 || g == 128)) return CGO_EINVAL;
    if (s->d % g) return CGO_EINVAL;
    if (p->backend == CGO_BU) {
        if (!valid_bits(p->bits) || p->block < 1 || s->d % p->block || (p->block * p->bits) % 8)
            return CGO_EINVAL;
    } else if (p->backend == CGO_BU_TILE) {
        if (!valid_bits(p->bits) || p->block < 1 || s->d % p->block || (p->block * p->bits) % 8)
            return CGO_EINVAL;
        /* a call starts at a tile boundary: a tile's range covers the tokens of one call */
        if (s->t0 > 0 && s->t0 % CGO_TILE_TOKENS) return CGO_EUNSUP;
    } else if (p->backend == CGO_KIVI) {
        if (!valid_bits(p->bits) || p->block < 1 || s->d % p->block || (p->block * p->bits) % 8 ||
            p->residual < 0)
            return CGO_EINVAL;
        if (s->t0 != 0 || (s->T_cap != 0 && s->T_cap != s->T)) return CGO_EUNSUP;
    } else if (p->backend != CGO_NONE) {
        return CGO_EINVAL;
    }
    if (s->t0 < 0 || s->T_cap < 0) return CGO_EINVAL;
    if (s->T_cap != 0 && s->t0 + s->T > s->T_cap) return CGO_EINVAL;
    return CGO_OK;
}

static int64_t tcap_of(const cgo_shape* s) { return s->T_cap ? s->T_cap : (int64_t)s->t0 + s->T; }
static int64_t ntiles_of(const cgo_shape* s) { return (tcap_of(s) + CGO_TILE_TOKENS - 1) / CGO_TILE_TOKENS; }

/* Measured bytes of each buffer (Appendix metric table: actual bits/value = measured
 * bytes / represented values), one count per stored item of the layouts. */
int cgo_packed_bytes(const cgo_shape* s, const cgo_params* p, int64_t* codes, int64_t* scales,
                     int64_t* resid)
{
    int rc = check_args(s, p);
    if (rc) return rc;
    int64_t units = (int64_t)s->L * 2 * s->B * s->H;
    int64_t d = s->d;
    if (p->backend == CGO_BU || p->backend == CGO_BU_TILE) {
        int64_t tc = tcap_of(s), nb = d / p->block, pay = (int64_t)p->block * p->bits / 8;
        /* one {scale, zero} pair per block of one token, or per block of one tile */
        int64_t nranges = p->backend == CGO_BU ? tc : ntiles_of(s);
        *codes = units * tc * nb * pay;
        *scales = units * nranges * nb * 4;
        *resid = 0;
    } else if (p->backend == CGO_KIVI) {
        int64_t nq = cgo_kivi_nq(s->T, p->residual, p->block);
        int64_t per_lbh_key = (nq / p->block) * d * ((int64_t)p->block * p->bits / 8);
        int64_t per_lbh_val = nq * (d / p->block) * ((int64_t)p->block * p->bits / 8);
        int64_t lbh = (int64_t)s->L * s->B * s->H;
        *codes = lbh * (per_lbh_key + per_lbh_val);
        *scales = lbh * ((nq / p->block) * d + nq * (d / p->block)) * 4;
        *resid = units * ((int64_t)s->T - nq) * d * 2;
    } else {
        *codes = units * tcap_of(s) * d * 4;
        *scales = 0;
        *resid = 0;
    }
    return CGO_OK;
}

/* ------------------------------------------------------------------------------ */
/* Gauge application, quantizer, packing                                           */
/* ------------------------------------------------------------------------------ */

/* Pairwise sum of the fp32 products Grow[j] * x[j] for j in [a, b) (b - a a power of two),
 * the fixed fp32 order of the file header. */
static float pairwise_dot(const float* Grow, const float* x, int a, int b)
{
    if (b - a == 1) return Grow[a] * x[a];
    int m = (a + b) / 2;
    return pairwise_dot(Grow, x, a, m) + pairwise_dot(Grow, x, m, b);
}

/* One gauge-space coordinate sum_j Grow[j] x[j] (g a power of two). */
static float gauge_dot(const float* Grow, const float* x, int g) { return pairwise_dot(Grow, x, 0, g); }

/* Z = G X for one token (Sec. 3): z[r*g + i] = sum_j G_r[i][j] x[r*g + j].
 * Gh points at this (l, s, h)'s R gauges. */
static void gauge_apply_f32(const float* Gh, const float* x, float* z, int d, int g)
{
    for (int r = 0; r < d / g; r++) {
        const float* Gr = Gh + (size_t)r * g * g;
        for (int i = 0; i < g; i++) z[r * g + i] = gauge_dot(Gr + (size_t)i * g, x + r * g, g);
    }
}

/* Xhat = G^T Zhat for one token (Sec. 3 decode equation with G^{-1} = G^T, Sec. 4.1),
 * in fp64: xh[r*g + i] = sum_j G_r[j][i] zh[r*g + j]. */
static void gauge_inverse_f64(const float* Gh, const double* zh, double* xh, int d, int g)
{
    for (int r = 0; r < d / g; r++) {
        const float* Gr = Gh + (size_t)r * g * g;
        for (int i = 0; i < g; i++) {
            double acc = 0.0;
            for (int j = 0; j < g; j++) acc += (double)Gr[(size_t)j * g + i] * zh[r * g + j];
            xh[r * g + i] = acc;
        }
    }
}

/* Asymmetric min/max quantizer over one block of n fp32 values (Sec. 4.3). Writes the
 * fp16 scale and zero, the codes, and optionally the near-boundary flag of each value
 * (pre-rounding value within 1e-4 steps of a half-integer). Returns status bits. */
static int quantize_block(const float* v, int n, int stride, int bits, uint16_t* s16_out,
                          uint16_t* m16_out, uint8_t* q_out, uint8_t* flag_out, int flag_stride)
{
    float mn = v[0], mx = v[0];
    for (int k = 1; k < n; k++) {
        float a = v[(size_t)k * stride];
        if (a < mn) mn = a;
        if (a > mx) mx = a;
    }
    const float qmax = (float)((1 << bits) - 1);
    float s32 = (mx - mn) / qmax;
    uint16_t s16 = cgo_f32_to_f16(s32), m16 = cgo_f32_to_f16(mn);
    int st = 0;
    if ((s16 & 0x7fffu) == 0x7c00u || (m16 & 0x7fffu) == 0x7c00u) st |= CGO_FLAG_FP16_OVERFLOW;
    float s = cgo_f16_to_f32(s16), m = cgo_f16_to_f32(m16);
    for (int k = 0; k < n; k++) {
        uint8_t q = 0, fl = 0;
        if (s != 0.0f) {
            float t = (v[(size_t)k * stride] - m) / s;
            float r = rintf(t); /* round half to even under the default rounding mode */
            if (r < 0.0f) r = 0.0f;
            if (r > qmax) r = qmax;
            if (!(r == r)) r = 0.0f; /* inf scale: t is NaN or 0 */
            q = (uint8_t)r;
            float frac = t - floorf(t);
            if (fabsf(frac - 0.5f) < 1e-4f) fl = 1;
        }
        q_out[k] = q;
        if (flag_out) flag_out[(size_t)k * flag_stride] = fl;
    }
    *s16_out = s16;
    *m16_out = m16;
    return st;
}

/* Little-endian bit stream: code k occupies bits [k*bits, (k+1)*bits). */
static void pack_codes(const uint8_t* q, int n, int bits, uint8_t* out)
{
    memset(out, 0, (size_t)n * bits / 8);
    for (int k = 0; k < n; k++)
        for (int b = 0; b < bits; b++)
            if ((q[k] >> b) & 1) {
                int pos = k * bits + b;
                out[pos >> 3] |= (uint8_t)(1u << (pos & 7));
            }
}

static void unpack_codes(const uint8_t* in, int n, int bits, uint8_t* q)
{
    for (int k = 0; k < n; k++) {
        unsigned v = 0;
        for (int b = 0; b < bits; b++) {
            int pos = k * bits + b;
            v |= (unsigned)((in[pos >> 3] >> (pos & 7)) & 1u) << b;
        }
        q[k] = (uint8_t)v;
    }
}

void cgo_pack(const uint8_t* q, int n, int bits, uint8_t* out) { pack_codes(q, n, bits, out); }
void cgo_unpack(const uint8_t* in, int n, int bits, uint8_t* q) { unpack_codes(in, n, bits, q); }

static int has_nonfinite(const uint16_t* x, int64_t n)
{
    for (int64_t k = 0; k < n; k++)
        if (((x[k] >> 7) & 0xffu) == 0xffu) return 1;
    return 0;
}

/* ------------------------------------------------------------------------------ */
/* Work split over independent units (the gauge never mixes l, s, b, h: Sec. 3)     */
/* ------------------------------------------------------------------------------ */

typedef struct {
    const cgo_shape* s;
    const cgo_params* p;
    const uint16_t* x;
    const float* G;
    uint8_t* codes;
    uint16_t* scales;
    uint16_t* resid;
    float* z_out;
    uint8_t* flag_out;
    const uint8_t* in_codes;
    const uint16_t* in_scales;
    const uint16_t* in_resid;
    double* xhat;
    int64_t n_units;
    int64_t next;
    int status;
    pthread_mutex_t mu;
    void (*fn)(void* ctx, int64_t unit);
} pool_t;

static void* pool_worker(void* arg)
{
    pool_t* P = (pool_t*)arg;
    for (;;) {
        pthread_mutex_lock(&P->mu);
        int64_t u = P->next++;
        pthread_mutex_unlock(&P->mu);
        if (u >= P->n_units) break;
        P->fn(P, u);
    }
    return NULL;
}

static void run_pool(pool_t* P, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_mutex_init(&P->mu, NULL);
    P->next = 0;
    if (nthreads == 1) {
        pool_worker(P);
    } else {
        pthread_t th[256];
        for (int i = 0; i < nthreads; i++) pthread_create(&th[i], NULL, pool_worker, P);
        for (int i = 0; i < nthreads; i++) pthread_join(th[i], NULL);
    }
    pthread_mutex_destroy(&P->mu);
}

static void add_status(pool_t* P, int st)
{
    if (!st) return;
    pthread_mutex_lock(&P->mu);
    P->status |= st;
    pthread_mutex_unlock(&P->mu);
}

/* ---- block-uniform / none: one unit = (l, s, b, h) ---- */

static void bu_encode_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group;
    int64_t h = u % s->H, sidx = (u / ((int64_t)s->H * s->B)) % 2, l = u / ((int64_t)s->H * s->B * 2);
    const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
    int64_t tc = tcap_of(s);
    float* x = (float*)malloc(sizeof(float) * d);
    float* z = (float*)malloc(sizeof(float) * d);
    uint8_t* q = (uint8_t*)malloc(d > 0 ? (size_t)d : 1);
    int st = 0;
    for (int64_t t = 0; t < s->T; t++) {
        const uint16_t* xr = P->x + ((size_t)u * s->T + t) * d;
        if (has_nonfinite(xr, d)) st |= CGO_FLAG_NONFINITE;
        for (int c = 0; c < d; c++) x[c] = cgo_bf16_to_f32(xr[c]);
        gauge_apply_f32(Gh, x, z, d, g);
        int64_t th = s->t0 + t;
        if (P->z_out) memcpy(P->z_out + ((size_t)u * s->T + t) * d, z, sizeof(float) * d);
        if (p->backend == CGO_NONE) {
            memcpy((float*)P->codes + ((size_t)u * tc + th) * d, z, sizeof(float) * d);
            continue;
        }
        int nb = d / p->block, pay = p->block * p->bits / 8;
        for (int b = 0; b < nb; b++) {
            uint16_t s16, m16;
            uint8_t* fl = P->flag_out ? P->flag_out + ((size_t)u * s->T + t) * d + (size_t)b * p->block : NULL;
            st |= quantize_block(z + b * p->block, p->block, 1, p->bits, &s16, &m16, q, fl, 1);
            size_t blk_index = ((size_t)u * tc + th) * nb + b;
            pack_codes(q, p->block, p->bits, P->codes + blk_index * pay);
            P->scales[blk_index * 2 + 0] = s16;
            P->scales[blk_index * 2 + 1] = m16;
        }
    }
    add_status(P, st);
    free(x);
    free(z);
    free(q);
}

/* ---- block-uniform tiles: one range per T_b x block tile (Sec. 4.3, T_b = 16 by Sec. 4.2) ----
 * The tile's tokens are consecutive tokens of one (l, s, b, h); its range is the min/max of
 * Z over all of them and the block's channels. Codes keep the per-token layout of the
 * block-uniform rows; only the {scale, zero} pairs are per tile. The last tile of a call may
 * hold fewer than T_b tokens; its range covers the tokens it holds. */
static void tile_encode_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group, blk = p->block, nb = d / blk, pay = blk * p->bits / 8;
    int64_t h = u % s->H, sidx = (u / ((int64_t)s->H * s->B)) % 2, l = u / ((int64_t)s->H * s->B * 2);
    const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
    int64_t tc = tcap_of(s), ntc = ntiles_of(s);
    const int TB = CGO_TILE_TOKENS;
    float* x = (float*)malloc(sizeof(float) * d);
    float* zt = (float*)malloc(sizeof(float) * TB * d);   /* Z of the tile's tokens, [tt][c] */
    float* v = (float*)malloc(sizeof(float) * TB * blk);  /* one tile block, [tt][c] */
    uint8_t* q = (uint8_t*)malloc((size_t)TB * blk);
    uint8_t* fl = (uint8_t*)malloc((size_t)TB * blk);
    int st = 0;
    for (int64_t ta = 0; ta < s->T; ta += TB) {
        int nt = s->T - ta < TB ? (int)(s->T - ta) : TB;
        for (int tt = 0; tt < nt; tt++) {
            const uint16_t* xr = P->x + ((size_t)u * s->T + ta + tt) * d;
            if (has_nonfinite(xr, d)) st |= CGO_FLAG_NONFINITE;
            for (int c = 0; c < d; c++) x[c] = cgo_bf16_to_f32(xr[c]);
            gauge_apply_f32(Gh, x, zt + (size_t)tt * d, d, g);
            if (P->z_out) memcpy(P->z_out + ((size_t)u * s->T + ta + tt) * d, zt + (size_t)tt * d, sizeof(float) * d);
        }
        int64_t tile = (s->t0 + ta) / TB;
        for (int b = 0; b < nb; b++) {
            for (int tt = 0; tt < nt; tt++)
                for (int c = 0; c < blk; c++) v[tt * blk + c] = zt[(size_t)tt * d + b * blk + c];
            uint16_t s16, m16;
            st |= quantize_block(v, nt * blk, 1, p->bits, &s16, &m16, q, P->flag_out ? fl : NULL, 1);
            for (int tt = 0; tt < nt; tt++) {
                int64_t th = s->t0 + ta + tt;
                pack_codes(q + tt * blk, blk, p->bits, P->codes + (((size_t)u * tc + th) * nb + b) * pay);
                if (P->flag_out)
                    memcpy(P->flag_out + ((size_t)u * s->T + ta + tt) * d + (size_t)b * blk, fl + tt * blk, blk);
            }
            size_t rng_index = ((size_t)u * ntc + tile) * nb + b;
            P->scales[rng_index * 2 + 0] = s16;
            P->scales[rng_index * 2 + 1] = m16;
        }
    }
    add_status(P, st);
    free(x);
    free(zt);
    free(v);
    free(q);
    free(fl);
}

static void bu_decode_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group;
    int64_t h = u % s->H, sidx = (u / ((int64_t)s->H * s->B)) % 2, l = u / ((int64_t)s->H * s->B * 2);
    const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
    int64_t tc = tcap_of(s);
    double* zh = (double*)malloc(sizeof(double) * d);
    uint8_t* q = (uint8_t*)malloc((size_t)d);
    for (int64_t t = 0; t < s->T; t++) {
        int64_t th = s->t0 + t;
        if (p->backend == CGO_NONE) {
            const float* zr = (const float*)P->in_codes + ((size_t)u * tc + th) * d;
            for (int c = 0; c < d; c++) zh[c] = (double)zr[c];
        } else {
            int nb = d / p->block, pay = p->block * p->bits / 8;
            for (int b = 0; b < nb; b++) {
                size_t blk_index = ((size_t)u * tc + th) * nb + b;
                /* the block's range: this token's own, or that of the tile holding it */
                size_t rng_index = p->backend == CGO_BU_TILE
                                       ? ((size_t)u * ntiles_of(s) + (size_t)(th / CGO_TILE_TOKENS)) * nb + b
                                       : blk_index;
                unpack_codes(P->in_codes + blk_index * pay, p->block, p->bits, q);
                double sc = (double)cgo_f16_to_f32(P->in_scales[rng_index * 2 + 0]);
                double mz = (double)cgo_f16_to_f32(P->in_scales[rng_index * 2 + 1]);
                for (int k = 0; k < p->block; k++) zh[b * p->block + k] = (double)q[k] * sc + mz;
            }
        }
        gauge_inverse_f64(Gh, zh, P->xhat + ((size_t)u * s->T + t) * d, d, g);
    }
    free(zh);
    free(q);
}

/* ---- KIVI: one unit = (l, b, h); keys and values handled together ---- */

static void kivi_offsets(const cgo_shape* s, const cgo_params* p, int64_t l, int64_t bh, int64_t* key_codes,
                         int64_t* val_codes, int64_t* key_scales, int64_t* val_scales)
{
    int64_t d = s->d, Gt = p->block, nq = cgo_kivi_nq(s->T, p->residual, Gt);
    int64_t pay = Gt * p->bits / 8;
    int64_t key_per = (nq / Gt) * d * pay, val_per = nq * (d / Gt) * pay;
    int64_t BH = (int64_t)s->B * s->H;
    int64_t layer_codes = BH * (key_per + val_per);
    *key_codes = l * layer_codes + bh * key_per;
    *val_codes = l * layer_codes + BH * key_per + bh * val_per;
    int64_t ks_per = (nq / Gt) * d, vs_per = nq * (d / Gt);
    int64_t layer_scales = BH * (ks_per + vs_per);
    *key_scales = l * layer_scales + bh * ks_per;
    *val_scales = l * layer_scales + BH * ks_per + bh * vs_per;
}

static void kivi_encode_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group, Gt = p->block, bits = p->bits, pay = Gt * bits / 8;
    int64_t T = s->T, nq = cgo_kivi_nq(T, p->residual, Gt);
    int64_t bh = u % ((int64_t)s->B * s->H), l = u / ((int64_t)s->B * s->H), h = bh % s->H, b = bh / s->H;
    int64_t kc, vc, ks, vs;
    kivi_offsets(s, p, l, bh, &kc, &vc, &ks, &vs);
    float* x = (float*)malloc(sizeof(float) * d);
    float* Z = (float*)malloc(sizeof(float) * (size_t)(nq > 0 ? nq : 1) * d);
    uint8_t* q = (uint8_t*)malloc((size_t)(Gt > d ? Gt : d));
    int st = 0;
    for (int sidx = 0; sidx < 2; sidx++) {
        int64_t unit5 = ((l * 2 + sidx) * s->B + b) * s->H + h; /* index of (l,s,b,h) */
        const uint16_t* X = P->x + (size_t)unit5 * T * d;
        const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
        if (has_nonfinite(X, T * d)) st |= CGO_FLAG_NONFINITE;
        /* gauge-space tensor of the quantized tokens */
        for (int64_t t = 0; t < nq; t++) {
            for (int c = 0; c < d; c++) x[c] = cgo_bf16_to_f32(X[t * d + c]);
            gauge_apply_f32(Gh, x, Z + (size_t)t * d, d, g);
        }
        if (P->z_out) memcpy(P->z_out + (size_t)unit5 * T * d, Z, sizeof(float) * (size_t)nq * d);
        if (sidx == 0) {
            /* keys: one range per channel over each group of Gt tokens (KIVI per-channel keys) */
            for (int64_t tg = 0; tg < nq / Gt; tg++)
                for (int c = 0; c < d; c++) {
                    uint16_t s16, m16;
                    uint8_t* fl = P->flag_out ? P->flag_out + ((size_t)unit5 * T + tg * Gt) * d + c : NULL;
                    st |= quantize_block(Z + (size_t)tg * Gt * d + c, Gt, d, bits, &s16, &m16, q, fl, d);
                    int64_t idx = tg * d + c;
                    pack_codes(q, Gt, bits, P->codes + kc + idx * pay);
                    P->scales[(ks + idx) * 2 + 0] = s16;
                    P->scales[(ks + idx) * 2 + 1] = m16;
                }
        } else {
            /* values: one range per token over each group of Gt channels (KIVI per-token values) */
            int nb = d / Gt;
            for (int64_t t = 0; t < nq; t++)
                for (int blk = 0; blk < nb; blk++) {
                    uint16_t s16, m16;
                    uint8_t* fl = P->flag_out ? P->flag_out + ((size_t)unit5 * T + t) * d + (size_t)blk * Gt : NULL;
                    st |= quantize_block(Z + (size_t)t * d + (size_t)blk * Gt, Gt, 1, bits, &s16, &m16, q, fl, 1);
                    int64_t idx = t * nb + blk;
                    pack_codes(q, Gt, bits, P->codes + vc + idx * pay);
                    P->scales[(vs + idx) * 2 + 0] = s16;
                    P->scales[(vs + idx) * 2 + 1] = m16;
                }
        }
        /* residual window: the newest T - nq tokens, raw bf16 */
        if (T - nq > 0)
            memcpy(P->resid + (size_t)unit5 * (T - nq) * d, X + (size_t)nq * d, sizeof(uint16_t) * (size_t)(T - nq) * d);
    }
    add_status(P, st);
    free(x);
    free(Z);
    free(q);
}

static void kivi_decode_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group, Gt = p->block, bits = p->bits, pay = Gt * bits / 8;
    int64_t T = s->T, nq = cgo_kivi_nq(T, p->residual, Gt);
    int64_t bh = u % ((int64_t)s->B * s->H), l = u / ((int64_t)s->B * s->H), h = bh % s->H, b = bh / s->H;
    int64_t kc, vc, ks, vs;
    kivi_offsets(s, p, l, bh, &kc, &vc, &ks, &vs);
    double* Zh = (double*)malloc(sizeof(double) * (size_t)(nq > 0 ? nq : 1) * d);
    uint8_t* q = (uint8_t*)malloc((size_t)(Gt > d ? Gt : d));
    for (int sidx = 0; sidx < 2; sidx++) {
        int64_t unit5 = ((l * 2 + sidx) * s->B + b) * s->H + h;
        const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
        if (sidx == 0) {
            for (int64_t tg = 0; tg < nq / Gt; tg++)
                for (int c = 0; c < d; c++) {
                    int64_t idx = tg * d + c;
                    unpack_codes(P->in_codes + kc + idx * pay, Gt, bits, q);
                    double sc = (double)cgo_f16_to_f32(P->in_scales[(ks + idx) * 2 + 0]);
                    double mz = (double)cgo_f16_to_f32(P->in_scales[(ks + idx) * 2 + 1]);
                    for (int k = 0; k < Gt; k++) Zh[(size_t)(tg * Gt + k) * d + c] = (double)q[k] * sc + mz;
                }
        } else {
            int nb = d / Gt;
            for (int64_t t = 0; t < nq; t++)
                for (int blk = 0; blk < nb; blk++) {
                    int64_t idx = t * nb + blk;
                    unpack_codes(P->in_codes + vc + idx * pay, Gt, bits, q);
                    double sc = (double)cgo_f16_to_f32(P->in_scales[(vs + idx) * 2 + 0]);
                    double mz = (double)cgo_f16_to_f32(P->in_scales[(vs + idx) * 2 + 1]);
                    for (int k = 0; k < Gt; k++) Zh[(size_t)t * d + (size_t)blk * Gt + k] = (double)q[k] * sc + mz;
                }
        }
        double* out = P->xhat + (size_t)unit5 * T * d;
        for (int64_t t = 0; t < nq; t++) gauge_inverse_f64(Gh, Zh + (size_t)t * d, out + (size_t)t * d, d, g);
        for (int64_t t = nq; t < T; t++)
            for (int c = 0; c < d; c++)
                out[(size_t)t * d + c] = (double)cgo_bf16_to_f32(P->in_resid[((size_t)unit5 * (T - nq) + (t - nq)) * d + c]);
    }
    free(Zh);
    free(q);
}

/* ------------------------------------------------------------------------------ */
/* Exported entry points                                                           */
/* ------------------------------------------------------------------------------ */

/* Encode (Sec. 3: Z = G X, B_c = C(Z)). z_out (fp32 [L][2][B][H][T][d]) and flag_out (u8,
 * same layout: 1 = pre-rounding value within 1e-4 steps of a rounding boundary) are
 * optional. Returns a CGO_* code; *status_out receives the CGO_FLAG_* bits. */
int cgo_encode(const cgo_shape* s, const cgo_params* p, const uint16_t* x, const float* G, uint8_t* codes,
               uint16_t* scales, uint16_t* resid, float* z_out, uint8_t* flag_out, int nthreads,
               int32_t* status_out)
{
    int rc = check_args(s, p);
    if (rc) return rc;
    pool_t P;
    memset(&P, 0, sizeof P);
    P.s = s; P.p = p; P.x = x; P.G = G; P.codes = codes; P.scales = scales; P.resid = resid;
    P.z_out = z_out; P.flag_out = flag_out;
    if (p->backend == CGO_KIVI) {
        P.n_units = (int64_t)s->L * s->B * s->H;
        P.fn = kivi_encode_unit;
    } else {
        P.n_units = (int64_t)s->L * 2 * s->B * s->H;
        P.fn = p->backend == CGO_BU_TILE ? tile_encode_unit : bu_encode_unit;
    }
    run_pool(&P, nthreads);
    if (status_out) *status_out = P.status;
    return CGO_OK;
}

/* Decode (Sec. 3: Zhat = D(B_c), Xhat = G^T Zhat). xhat: fp64 [L][2][B][H][T][d]. */
int cgo_decode(const cgo_shape* s, const cgo_params* p, const uint8_t* codes, const uint16_t* scales,
               const uint16_t* resid, const float* G, double* xhat, int nthreads)
{
    int rc = check_args(s, p);
    if (rc) return rc;
    pool_t P;
    memset(&P, 0, sizeof P);
    P.s = s; P.p = p; P.G = G; P.in_codes = codes; P.in_scales = scales; P.in_resid = resid; P.xhat = xhat;
    if (p->backend == CGO_KIVI) {
        P.n_units = (int64_t)s->L * s->B * s->H;
        P.fn = kivi_decode_unit;
    } else {
        P.n_units = (int64_t)s->L * 2 * s->B * s->H;
        P.fn = bu_decode_unit;
    }
    run_pool(&P, nthreads);
    return CGO_OK;
}

/* The gauge-space value of one coordinate, exposed so that tests can pin the chain. */
float cgo_gauge_coord(const float* Grow, const float* x, int g) { return gauge_dot(Grow, x, g); }

/* ------------------------------------------------------------------------------ */
/* KIVI streaming (Sec. 4.3 KIVI-style path; a rolling cache of Sec. 4.4)          */
/* ------------------------------------------------------------------------------ */
/* A KIVI history of capacity T_cap tokens per (l, s, b, h) grows by appends. After T tokens
 * the quantized part holds the first n_q(T) = cgo_kivi_nq(T, R, Gt) tokens, in the batch
 * layout sized for n_q(T_cap) tokens (quantized groups at fixed places), and the newest
 * T - n_q(T) tokens stay raw in a ring of W = R + Gt token slots: token t lives in slot
 * t mod W. The window never holds more than R + Gt - 1 tokens, so no two of its tokens
 * share a slot. An append of tokens [t0, t0 + T) quantizes every key group that completes,
 * [n_q(t0), n_q(t0 + T)), reading tokens below t0 from the ring and the others from the new
 * input, and then stores the new tokens that stay raw. The result equals the batch encode
 * of all t0 + T tokens (keys and values in the same places, the ring holding the window). */

static int64_t ring_slots(const cgo_params* p) { return (int64_t)p->residual + p->block; }

static int check_stream(const cgo_shape* s, const cgo_params* p)
{
    if (!s || !p || p->backend != CGO_KIVI) return CGO_EINVAL;
    cgo_shape whole = *s;
    whole.t0 = 0;
    whole.T = s->T_cap;
    whole.T_cap = 0;
    int rc = check_args(&whole, p);
    if (rc) return rc;
    if (s->T_cap < 1 || s->t0 < 0 || s->T < 0 || (int64_t)s->t0 + s->T > s->T_cap) return CGO_EINVAL;
    return CGO_OK;
}

/* Byte counts of the stream buffers: codes and scales for n_q(T_cap) quantized tokens
 * (the batch layout at that length), and the ring [L][2][B][H][W][d] of bf16. */
int cgo_kivi_stream_bytes(const cgo_shape* s, const cgo_params* p, int64_t* codes, int64_t* scales,
                          int64_t* ring)
{
    int rc = check_stream(s, p);
    if (rc) return rc;
    cgo_shape cap = *s;
    cap.t0 = 0;
    cap.T = s->T_cap;
    cap.T_cap = 0;
    int64_t r;
    cgo_packed_bytes(&cap, p, codes, scales, &r);
    *ring = (int64_t)s->L * 2 * s->B * s->H * ring_slots(p) * s->d * 2;
    return CGO_OK;
}

static const uint16_t* stream_token(const pool_t* P, int64_t unit5, int64_t t)
{
    const cgo_shape* s = P->s;
    int64_t W = ring_slots(P->p);
    if (t < s->t0) return P->resid + ((size_t)unit5 * W + (size_t)(t % W)) * s->d;
    return P->x + ((size_t)unit5 * s->T + (size_t)(t - s->t0)) * s->d;
}

static void kivi_append_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group, Gt = p->block, bits = p->bits, pay = Gt * bits / 8, nb = d / Gt;
    int64_t R = p->residual, W = ring_slots(p);
    int64_t nq_old = cgo_kivi_nq(s->t0, R, Gt), nq_new = cgo_kivi_nq((int64_t)s->t0 + s->T, R, Gt);
    int64_t bh = u % ((int64_t)s->B * s->H), l = u / ((int64_t)s->B * s->H), h = bh % s->H, b = bh / s->H;
    cgo_shape cap = *s;   /* offsets of the layout sized for the capacity */
    cap.t0 = 0;
    cap.T = s->T_cap;
    cap.T_cap = 0;
    int64_t kc, vc, ks, vs;
    kivi_offsets(&cap, p, l, bh, &kc, &vc, &ks, &vs);
    float* x = (float*)malloc(sizeof(float) * d);
    float* Z = (float*)malloc(sizeof(float) * (size_t)Gt * d);
    uint8_t* q = (uint8_t*)malloc((size_t)(Gt > d ? Gt : d));
    int st = 0;
    for (int sidx = 0; sidx < 2; sidx++) {
        int64_t unit5 = ((l * 2 + sidx) * s->B + b) * s->H + h;
        const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
        if (has_nonfinite(P->x + (size_t)unit5 * s->T * d, (int64_t)s->T * d)) st |= CGO_FLAG_NONFINITE;
        for (int64_t tg = nq_old / Gt; tg < nq_new / Gt; tg++) {
            for (int k = 0; k < Gt; k++) {   /* Z of the group's tokens */
                const uint16_t* xr = stream_token(P, unit5, tg * Gt + k);
                for (int c = 0; c < d; c++) x[c] = cgo_bf16_to_f32(xr[c]);
                gauge_apply_f32(Gh, x, Z + (size_t)k * d, d, g);
            }
            if (sidx == 0) {   /* keys: per channel over the group */
                for (int c = 0; c < d; c++) {
                    uint16_t s16, m16;
                    st |= quantize_block(Z + c, Gt, d, bits, &s16, &m16, q, NULL, 0);
                    int64_t idx = tg * d + c;
                    pack_codes(q, Gt, bits, P->codes + kc + idx * pay);
                    P->scales[(ks + idx) * 2 + 0] = s16;
                    P->scales[(ks + idx) * 2 + 1] = m16;
                }
            } else {           /* values: per token over blocks of Gt channels */
                for (int k = 0; k < Gt; k++)
                    for (int blk = 0; blk < nb; blk++) {
                        uint16_t s16, m16;
                        st |= quantize_block(Z + (size_t)k * d + (size_t)blk * Gt, Gt, 1, bits, &s16, &m16, q, NULL, 0);
                        int64_t idx = (tg * Gt + k) * nb + blk;
                        pack_codes(q, Gt, bits, P->codes + vc + idx * pay);
                        P->scales[(vs + idx) * 2 + 0] = s16;
                        P->scales[(vs + idx) * 2 + 1] = m16;
                    }
            }
        }
        /* the new tokens that stay raw go to their ring slots (after the reads above) */
        for (int64_t t = (nq_new > s->t0 ? nq_new : s->t0); t < (int64_t)s->t0 + s->T; t++)
            memcpy(P->resid + ((size_t)unit5 * W + (size_t)(t % W)) * d,
                   P->x + ((size_t)unit5 * s->T + (size_t)(t - s->t0)) * d, sizeof(uint16_t) * d);
    }
    add_status(P, st);
    free(x);
    free(Z);
    free(q);
}

/* Append tokens [t0, t0 + T) (x_new: bf16 [L][2][B][H][T][d]) to a KIVI stream of capacity
 * T_cap that holds t0 tokens: codes, scales and ring as laid out above. */
int cgo_kivi_append(const cgo_shape* s, const cgo_params* p, const uint16_t* x_new, const float* G, uint8_t* codes,
                    uint16_t* scales, uint16_t* ring, int nthreads, int32_t* status_out)
{
    int rc = check_stream(s, p);
    if (rc) return rc;
    pool_t P;
    memset(&P, 0, sizeof P);
    P.s = s; P.p = p; P.x = x_new; P.G = G; P.codes = codes; P.scales = scales; P.resid = ring;
    P.n_units = (int64_t)s->L * s->B * s->H;
    P.fn = kivi_append_unit;
    run_pool(&P, nthreads);
    if (status_out) *status_out = P.status;
    return CGO_OK;
}

static void kivi_stream_decode_unit(void* ctx, int64_t u)
{
    pool_t* P = (pool_t*)ctx;
    const cgo_shape* s = P->s;
    const cgo_params* p = P->p;
    int d = s->d, g = p->group, Gt = p->block, bits = p->bits, pay = Gt * bits / 8, nb = d / Gt;
    int64_t W = ring_slots(p), T = s->T, nq = cgo_kivi_nq(T, p->residual, Gt);
    int64_t bh = u % ((int64_t)s->B * s->H), l = u / ((int64_t)s->B * s->H), h = bh % s->H, b = bh / s->H;
    cgo_shape cap = *s;
    cap.t0 = 0;
    cap.T = s->T_cap;
    cap.T_cap = 0;
    int64_t kc, vc, ks, vs;
    kivi_offsets(&cap, p, l, bh, &kc, &vc, &ks, &vs);
    double* zh = (double*)malloc(sizeof(double) * d);
    uint8_t* q = (uint8_t*)malloc((size_t)(Gt > d ? Gt : d));
    for (int sidx = 0; sidx < 2; sidx++) {
        int64_t unit5 = ((l * 2 + sidx) * s->B + b) * s->H + h;
        const float* Gh = P->G + ((size_t)(l * 2 + sidx) * s->H + h) * (size_t)d * g;
        double* out = P->xhat + (size_t)unit5 * T * d;
        for (int64_t t = 0; t < nq; t++) {
            for (int c = 0; c < d; c++) {   /* zhat of token t */
                int64_t idx, k;
                uint16_t sc16, mz16;
                if (sidx == 0) {
                    idx = (t / Gt) * d + c;
                    k = t % Gt;
                    unpack_codes(P->in_codes + kc + idx * pay, Gt, bits, q);
                    sc16 = P->in_scales[(ks + idx) * 2 + 0];
                    mz16 = P->in_scales[(ks + idx) * 2 + 1];
                } else {
                    idx = t * nb + c / Gt;
                    k = c % Gt;
                    unpack_codes(P->in_codes + vc + idx * pay, Gt, bits, q);
                    sc16 = P->in_scales[(vs + idx) * 2 + 0];
                    mz16 = P->in_scales[(vs + idx) * 2 + 1];
                }
                zh[c] = (double)q[k] * (double)cgo_f16_to_f32(sc16) + (double)cgo_f16_to_f32(mz16);
            }
            gauge_inverse_f64(Gh, zh, out + (size_t)t * d, d, g);
        }
        for (int64_t t = nq; t < T; t++)
            for (int c = 0; c < d; c++)
                out[(size_t)t * d + c] = (double)cgo_bf16_to_f32(P->in_resid[((size_t)unit5 * W + (size_t)(t % W)) * d + c]);
    }
    free(zh);
    free(q);
}

/* Decode the first T tokens of a KIVI stream (t0 must be 0): xhat fp64 [L][2][B][H][T][d]. */
int cgo_kivi_stream_decode(const cgo_shape* s, const cgo_params* p, const uint8_t* codes, const uint16_t* scales,
                           const uint16_t* ring, const float* G, double* xhat, int nthreads)
{
    int rc = check_stream(s, p);
    if (rc) return rc;
    if (s->t0 != 0) return CGO_EUNSUP;
    pool_t P;
    memset(&P, 0, sizeof P);
    P.s = s; P.p = p; P.G = G; P.in_codes = codes; P.in_scales = scales; P.in_resid = ring; P.xhat = xhat;
    P.n_units = (int64_t)s->L * s->B * s->H;
    P.fn = kivi_stream_decode_unit;
    run_pool(&P, nthreads);
    return CGO_OK;
}

/* ------------------------------------------------------------------------------ */
/* Attention over the recovered cache (Fig. 1: the inverse gauge restores the cache  */
/* before attention; standard softmax attention, grouped queries, Sec. 3)          */
/* ------------------------------------------------------------------------------ */
/* One decoding query per sequence: n_rep query heads share each KV head (grouped-query
 * attention; n_rep = 1 is multi-head attention). For query head r of KV head h:
 *   s_t = scale * sum_c q[c] Khat[t][c],  p_t = exp(s_t - max_t s_t) / sum_t exp(...),
 *   o[c] = sum_t p_t Vhat[t][c],
 * all in fp64, with Khat, Vhat the decoded cache xhat [L][2][B][H][T][d] (s = 0 keys, 1 values)
 * and q bf16 [L][B][H][n_rep][d]. out: fp64 [L][B][H][n_rep][d]. */
int cgo_attention(int L, int B, int H, int T, int d, int n_rep, const uint16_t* q, const double* xhat,
                  double scale, double* out)
{
    if (L < 1 || B < 1 || H < 1 || T < 1 || d < 1 || n_rep < 1) return CGO_EINVAL;
    double* s = (double*)malloc(sizeof(double) * (size_t)T);
    for (int l = 0; l < L; l++)
        for (int b = 0; b < B; b++)
            for (int h = 0; h < H; h++) {
                const double* K = xhat + ((((size_t)l * 2 + 0) * B + b) * H + h) * (size_t)T * d;
                const double* V = xhat + ((((size_t)l * 2 + 1) * B + b) * H + h) * (size_t)T * d;
                for (int r = 0; r < n_rep; r++) {
                    size_t qi = ((((size_t)l * B + b) * H + h) * n_rep + r) * (size_t)d;
                    double mx = -INFINITY;
                    for (int t = 0; t < T; t++) {
                        double acc = 0.0;
                        for (int c = 0; c < d; c++) acc += (double)cgo_bf16_to_f32(q[qi + c]) * K[(size_t)t * d + c];
                        s[t] = scale * acc;
                        if (s[t] > mx) mx = s[t];
                    }
                    double z = 0.0;
                    for (int t = 0; t < T; t++) {
                        s[t] = exp(s[t] - mx);
                        z += s[t];
                    }
                    for (int c = 0; c < d; c++) {
                        double acc = 0.0;
                        for (int t = 0; t < T; t++) acc += s[t] * V[(size_t)t * d + c];
                        out[qi + c] = acc / z;
                    }
                }
            }
    free(s);
    return CGO_OK;
}
