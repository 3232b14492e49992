// sfc_curve.cuh -- generalized Hilbert curve position -> output tile.
//
// The SFC GEMM orders the Mt x Nt output-tile grid along a generalized
// Hilbert curve (Sec. II-B, Fig. 2) and maps each curve position to a tile
// (map_sfc_index in Listing 1).  Instead of storing the map, the kernel decodes
// a position directly: the curve is defined by recursive cuts of a rectangle
// (origin, major axis vector a, minor axis vector b) into two pieces (a region
// much longer than wide, 2|a| > 3|b|, cut across a) or three pieces (a corner
// block of the first half of a by the first, even-rounded part of b, walked
// with a and b exchanged; the strip across all of a over the rest of b; the
// other corner block walked back with exchanged, negated axes).  Every piece
// has a known cell count, so a position is located by descending into the
// piece that contains it, O(log max(Mt, Nt)) steps, no memory.
//
// Conventions: x runs along tn (columns of C tiles), y along tm (rows); the
// curve starts at tile (0,0).  The major axis is the longer side of the grid,
// except that an odd longer side with an even shorter side makes the even
// side the major axis (that is the orientation for which every consecutive
// pair of tiles can share an edge).
#pragma once

#include <cstdint>

namespace sfc {

struct TileCoord {
    int tm;
    int tn;
};

__host__ __device__ __forceinline__ int sgn_i(int v) { return (v > 0) - (v < 0); }
__host__ __device__ __forceinline__ int abs_i(int v) { return v < 0 ? -v : v; }

// s in [0, Mt*Nt), Mt*Nt < 2^31: every count below fits in 32 bits, which
// keeps this single-thread dependent chain short on the GPU.
__host__ __device__ inline TileCoord curve_decode(int s, int Mt, int Nt) {
    // current region: origin (x, y), major vector (ax, ay), minor vector (bx, by)
    int x = 0, y = 0, ax, ay, bx, by;
    bool major_is_x = Nt >= Mt;
    const int longer = major_is_x ? Nt : Mt;
    const int shorter = major_is_x ? Mt : Nt;
    if ((longer & 1) && !(shorter & 1)) major_is_x = !major_is_x;
    if (major_is_x) { ax = Nt; ay = 0; bx = 0; by = Mt; }
    else            { ax = 0;  ay = Mt; bx = Nt; by = 0; }

    int r = s;  // rank of the wanted cell inside the current region
    for (;;) {
        const int w = abs_i(ax + ay), h = abs_i(bx + by);
        const int ux = sgn_i(ax), uy = sgn_i(ay);  // unit step along the major axis
        const int vx = sgn_i(bx), vy = sgn_i(by);  // unit step along the minor axis
        if (h == 1) { x += r * ux; y += r * uy; break; }
        if (w == 1) { x += r * vx; y += r * vy; break; }

        int hax = ax / 2, hay = ay / 2;  // first part of the major axis
        int hbx = bx / 2, hby = by / 2;  // first part of the minor axis
        int hw = abs_i(hax + hay), hh = abs_i(hbx + hby);

        if (2 * w > 3 * h) {
            // two pieces along the major axis, first one even when possible
            if ((hw & 1) && w > 2) { hax += ux; hay += uy; ++hw; }
            const int first = hw * h;
            if (r < first) { ax = hax; ay = hay; }
            else { r -= first; x += hax; y += hay; ax -= hax; ay -= hay; }
            continue;
        }

        if ((hh & 1) && h > 2) { hbx += vx; hby += vy; ++hh; }
        const int corner = hh * hw;       // first corner block
        const int strip = w * (h - hh);   // strip across
        if (r < corner) {
            // axes exchanged: major = first part of b, minor = first half of a
            const int nax = hbx, nay = hby;
            bx = hax; by = hay; ax = nax; ay = nay;
        } else if (r < corner + strip) {
            r -= corner;
            x += hbx; y += hby; bx -= hbx; by -= hby;
        } else {
            r -= corner + strip;
            // far corner: one step short of the end of a, top of the first part of b
            const int nx = x + (ax - ux) + (hbx - vx);
            const int ny = y + (ay - uy) + (hby - vy);
            const int nax = -hbx, nay = -hby;
            const int nbx = -(ax - hax), nby = -(ay - hay);
            x = nx; y = ny; ax = nax; ay = nay; bx = nbx; by = nby;
        }
    }
    return TileCoord{y, x};
}

__host__ __device__ __forceinline__ TileCoord raster_decode(int s, int Nt) {
    const int tm = s / Nt;
    return TileCoord{tm, s - tm * Nt};
}

}  // namespace sfc
