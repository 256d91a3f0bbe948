// cg_tc_common.cuh -- tile scheduling shared by the tensor-core row kernels (d = 128).
//
// A "unit" is one (l, s, b, h) token sequence; units are ordered with b fastest, then h,
// s and l, so consecutive units share the gauge set of (l, s, h) for B units in a row (a
// "segment"). A unit is cut into 128-token tiles; each persistent CTA takes a contiguous
// range of the tile list, which keeps the gauge in shared memory across tiles.
#pragma once

#include <cuda_runtime.h>

#include "cg_launch.h"

namespace cg {
namespace tc {

constexpr int kD = 128;
constexpr uint64_t kWaitLimitNs = 4000000000ull;  // bounded pipeline waits (4 s)

struct Sched {
    int64_t n_units, tiles_per_unit, n_tiles;
};

__host__ __device__ __forceinline__ Sched make_sched(const RowArgs& a) {
    Sched s;
    s.n_units = (int64_t)a.L * a.s_n * a.B * a.H;
    s.tiles_per_unit = (a.t_count + 127) / 128;
    s.n_tiles = s.n_units * s.tiles_per_unit;
    return s;
}

struct TileInfo {
    int l, s, b, h;
    int64_t t0;       // first token of the tile inside the unit
    int64_t seg;      // global segment (gauge set) index
    int rows_valid;   // tokens of the tile that exist (<= 128)
};

__device__ __forceinline__ TileInfo tile_info(const RowArgs& a, const Sched& S, int64_t tile) {
    TileInfo ti;
    const int64_t u = tile / S.tiles_per_unit;
    ti.t0 = (tile - u * S.tiles_per_unit) * 128;
    ti.b = (int)(u % a.B);
    ti.seg = u / a.B;
    int64_t r = ti.seg;
    ti.h = (int)(r % a.H);
    r /= a.H;
    ti.s = a.s_lo + (int)(r % a.s_n);
    ti.l = (int)(r / a.s_n);
    const int64_t left = a.t_count - ti.t0;
    ti.rows_valid = (int)(left < 128 ? left : 128);
    return ti;
}

// Walks a CTA's tile range in steps of 1 or 2 tiles without integer division (the full
// decomposition is done once, at init).
struct TileIter {
    int tt;        // tile within the unit
    int tpu;       // tiles per unit
    int l, s, b, h;
    int64_t seg;

    __device__ __forceinline__ void init(const RowArgs& a, const Sched& S, int64_t tile) {
        const TileInfo ti = tile_info(a, S, tile);
        tpu = (int)S.tiles_per_unit;
        tt = (int)(ti.t0 >> 7);
        l = ti.l;
        s = ti.s;
        b = ti.b;
        h = ti.h;
        seg = ti.seg;
    }
    __device__ __forceinline__ void next_unit(const RowArgs& a) {
        if (++b == a.B) {
            b = 0;
            seg++;
            if (++h == a.H) {
                h = 0;
                if (++s == a.s_lo + a.s_n) {
                    s = a.s_lo;
                    l++;
                }
            }
        }
    }
    __device__ __forceinline__ void step(const RowArgs& a, int k) {
        tt += k;
        while (tt >= tpu) {
            tt -= tpu;
            next_unit(a);
        }
    }
    // last tile of its gauge segment (the segment's units are B consecutive units)
    __device__ __forceinline__ bool seg_last(const RowArgs& a) const { return tt == tpu - 1 && b == a.B - 1; }
    __device__ __forceinline__ TileInfo info(const RowArgs& a) const {
        TileInfo ti;
        ti.l = l;
        ti.s = s;
        ti.b = b;
        ti.h = h;
        ti.seg = seg;
        ti.t0 = (int64_t)tt * 128;
        const int64_t left = a.t_count - ti.t0;
        ti.rows_valid = (int)(left < 128 ? left : 128);
        return ti;
    }
};

// Row of unit (l, s, b, h) in the dense [L][2][B][H][T_x][d] tensor.
__device__ __forceinline__ int64_t dense_row(const RowArgs& a, const TileInfo& ti) {
    return (((int64_t)(ti.l * 2 + ti.s) * a.B + ti.b) * a.H + ti.h) * a.T_x + ti.t0;
}

__device__ __forceinline__ int64_t gauge_set(const RowArgs& a, const TileInfo& ti) {
    return (int64_t)(ti.l * 2 + ti.s) * a.H + ti.h;
}

inline int num_sms() {
    static int n[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (!n[dev]) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        n[dev] = v > 0 ? v : 148;
    }
    return n[dev];
}

}  // namespace tc
}  // namespace cg
