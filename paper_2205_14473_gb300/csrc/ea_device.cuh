// ea_device.cuh -- device building blocks of the round kernels: Philox4x32-10, the compensated
// l1 reduction, the quantizers of Definition 1 / Examples 1-2 / Definition 3, code packing.
//
// Every per-coordinate expression uses the explicit round-to-nearest intrinsics (__fadd_rn,
// __fmul_rn, __fdiv_rn, __fsqrt_rn), so nothing is contracted into an FMA and the order of
// Algorithms 1-2 is kept: the result is the binary32 evaluation of the paper's expressions.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "ea_internal.h"

namespace ea {

// ------------------------------------------------------------------------------ Philox4x32-10
// The counter-based generator of Salmon, Moraes, Dror and Shaw (SC'11): ten rounds of two 32x32
// multiplies of the even words, the odd words and the key xored into the high halves, the key
// advanced by the Weyl constants between rounds.  Coordinate j draws word j mod 4 of the counter
// (j/4 low, j/4 high, id, round) under the key (seed low, seed high).
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint2 k)
{
#pragma unroll
    for (int r = 0; r < 10; ++r) {
        const uint32_t hi0 = __umulhi(0xD2511F53u, c.x), lo0 = 0xD2511F53u * c.x;
        const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z), lo1 = 0xCD9E8D57u * c.z;
        c = make_uint4(hi1 ^ c.y ^ k.x, lo1, hi0 ^ c.w ^ k.y, lo0);
        k.x += 0x9E3779B9u;
        k.y += 0xBB67AE85u;
    }
    return c;
}

// The four uniform variates U in [0, 1) (24 bits) of coordinates j0 .. j0+3 (j0 % 4 == 0).
__device__ __forceinline__ void uniforms4(uint64_t seed, uint32_t id, uint32_t t, int64_t j0, float U[4])
{
    const uint64_t blk = static_cast<uint64_t>(j0) >> 2;
    const uint4 w = philox4x32_10(make_uint4(static_cast<uint32_t>(blk), static_cast<uint32_t>(blk >> 32), id, t),
                                  make_uint2(static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32)));
    U[0] = __fmul_rn(__uint2float_rn(w.x >> 8), 0x1p-24f);
    U[1] = __fmul_rn(__uint2float_rn(w.y >> 8), 0x1p-24f);
    U[2] = __fmul_rn(__uint2float_rn(w.z >> 8), 0x1p-24f);
    U[3] = __fmul_rn(__uint2float_rn(w.w >> 8), 0x1p-24f);
}

// -------------------------------------------------------------------- compensated summation
// Sums of |u| are carried as an unevaluated pair hi + lo of binary32 numbers: TwoSum keeps the
// rounding error of every addition, so a 4096-term sum is accurate to ~2^-44 relative without the
// (on this part, scarce) binary64 pipeline.  Only the CTA total is converted to binary64.
struct DF {
    float hi, lo;
};

__device__ __forceinline__ void two_sum(float a, float b, float &s, float &err)
{
    s = __fadd_rn(a, b);
    const float bb = __fsub_rn(s, a);
    err = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

__device__ __forceinline__ DF df_add(DF a, DF b)
{
    float s, e;
    two_sum(a.hi, b.hi, s, e);
    float lo = __fadd_rn(__fadd_rn(a.lo, b.lo), e);
    const float hi = __fadd_rn(s, lo);
    lo = __fsub_rn(lo, __fsub_rn(hi, s));
    return {hi, lo};
}

// Add x >= 0 to an accumulator of non-negative terms, its error terms collected in acc.lo.  With
// a = max(acc.hi, x) >= b = min(acc.hi, x) >= 0, Dekker's Fast2Sum gives s + e = a + b exactly.
__device__ __forceinline__ void df_accumulate(DF &acc, float x)
{
    const float a = fmaxf(acc.hi, x), b = fminf(acc.hi, x);
    const float s = __fadd_rn(a, b);
    const float e = __fsub_rn(b, __fsub_rn(s, a));
    acc.hi = s;
    acc.lo = __fadd_rn(acc.lo, e);
}

// Barrier over the 256 compute threads (named barrier 1), so that a CTA may also hold a producer
// warp that does not take part in the reductions.
__device__ __forceinline__ void compute_sync() { asm volatile("bar.sync 1, %0;" ::"n"(kThreads) : "memory"); }

// CTA-wide sum; every thread receives the same binary64 value (fixed combination order).
__device__ __forceinline__ double block_sum(DF v, DF *red, double *bcast)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        DF w{__shfl_down_sync(0xffffffffu, v.hi, o), __shfl_down_sync(0xffffffffu, v.lo, o)};
        v = df_add(v, w);
    }
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) red[warp] = v;
    compute_sync();
    if (threadIdx.x == 0) {
        DF t = red[0];
#pragma unroll
        for (int w = 1; w < kWarps; ++w) t = df_add(t, red[w]);
        *bcast = static_cast<double>(t.hi) + static_cast<double>(t.lo);
    }
    compute_sync();
    const double r = *bcast;
    return r;
}

// Group scale of the scaled sign, ||u||_1 / G, for a group that is exactly this CTA's tile.
// Every thread leaves its partial pair in red256; warp 0 combines the 256 pairs (8 per lane in a
// tree, then a 5-level shuffle tree) and broadcasts the scale through *bcastf.  For G a
// power of two, RN32((hi + lo) / G) = RN32(hi + lo) * 2^-k is one binary32 addition and an exact
// scaling; other lengths (a ragged last tile) divide in binary64.  Two barriers; red256 and bcastf
// may be reused after the function returns.
__device__ __forceinline__ float block_sign_scale(DF v, int64_t len, DF *red256, float *bcastf)
{
    red256[threadIdx.x] = v;
    compute_sync();
    if (threadIdx.x < 32) {
        static_assert(kThreads == 256, "eight partials per lane");
        DF p[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) p[j] = red256[threadIdx.x + 32 * j];
        // a tree of depth 3 over the lane's eight partials, then five shuffle levels: eight
        // dependent additions in all
        DF t = df_add(df_add(df_add(p[0], p[1]), df_add(p[2], p[3])), df_add(df_add(p[4], p[5]), df_add(p[6], p[7])));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            DF w{__shfl_down_sync(0xffffffffu, t.hi, o), __shfl_down_sync(0xffffffffu, t.lo, o)};
            t = df_add(t, w);
        }
        if (threadIdx.x == 0) {
            float s = 0.0f;
            if (len > 0 && (len & (len - 1)) == 0) {  // len <= 4096 here: 2^-k is a normal binary32
                const int k = __ffsll(static_cast<long long>(len)) - 1;
                s = __fmul_rn(__fadd_rn(t.hi, t.lo), __uint_as_float(static_cast<uint32_t>(127 - k) << 23));
            } else if (len > 0) {
                const double l1 = static_cast<double>(t.hi) + static_cast<double>(t.lo);
                s = __double2float_rn(__ddiv_rn(l1, static_cast<double>(len)));
            }
            *bcastf = s;
        }
    }
    compute_sync();
    return *bcastf;
}

// CTA-wide compensated sum of the 256 threads' pairs, combined by warp 0 as in block_sign_scale
// (eight pairs per lane in a tree, then five shuffle levels); the result is valid in thread 0
// only.  One barrier; red256 may be reused after the next barrier.
__device__ __forceinline__ DF block_sum_lane0(DF v, DF *red256)
{
    red256[threadIdx.x] = v;
    compute_sync();
    DF t{0.0f, 0.0f};
    if (threadIdx.x < 32) {
        DF p[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) p[j] = red256[threadIdx.x + 32 * j];
        t = df_add(df_add(df_add(p[0], p[1]), df_add(p[2], p[3])), df_add(df_add(p[4], p[5]), df_add(p[6], p[7])));
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            DF w{__shfl_down_sync(0xffffffffu, t.hi, o), __shfl_down_sync(0xffffffffu, t.lo, o)};
            t = df_add(t, w);
        }
    }
    return t;
}

// CTA-wide maximum for a group that is exactly this CTA's tile: one barrier, every thread combines
// the warp maxima itself.  The caller must barrier before `red` is reused.
__device__ __forceinline__ float block_max_all(float a, uint32_t *red)
{
    const uint32_t b = __reduce_max_sync(0xffffffffu, __float_as_uint(a));
    const int lane = threadIdx.x & 31;
    if (lane == 0) red[threadIdx.x >> 5] = b;
    compute_sync();
    return __uint_as_float(__reduce_max_sync(0xffffffffu, lane < kWarps ? red[lane] : 0u));
}

// CTA-wide maximum of non-negative values (exact: compares bit patterns).
__device__ __forceinline__ float block_max(float a, uint32_t *red, float *bcast)
{
    const uint32_t b = __reduce_max_sync(0xffffffffu, __float_as_uint(a));
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) red[warp] = b;
    compute_sync();
    if (threadIdx.x == 0) {
        uint32_t m = red[0];
#pragma unroll
        for (int w = 1; w < kWarps; ++w) m = max(m, red[w]);
        *bcast = __uint_as_float(m);
    }
    compute_sync();
    const float r = *bcast;
    return r;
}

// Group scale of the scaled sign: ||u||_1 / G, the division in binary64, one rounding to binary32.
__device__ __forceinline__ float sign_scale(double l1, int64_t len)
{
    return len > 0 ? __double2float_rn(__ddiv_rn(l1, static_cast<double>(len))) : 0.0f;
}

// ------------------------------------------------------------------------------- quantizers
// Codes: sign 1 = (u >= 0); uniform q + L with L = 2^(b-1) - 1; pow2 sign bit b-1 and exponent
// index below it, all-ones index = 0; identity = the binary32 pattern.

__device__ __forceinline__ int unif_L(int bits) { return (1 << (bits - 1)) - 1; }

// Example 1: z = u / s, y = z L, nearest grid index (ties to even) or stochastic rounding.
__device__ __forceinline__ int unif_index(float u, float s, float Lf, bool stochastic, float U)
{
    if (!(s > 0.0f)) return 0;
    const float z = __fdiv_rn(u, s);
    const float y = __fmul_rn(z, Lf);
    if (stochastic) {
        const float f = floorf(y);
        const float frac = __fsub_rn(y, f);
        return static_cast<int>(f) + (U < frac ? 1 : 0);
    }
    return __float2int_rn(y);
}

// Example 2: the nearest of {2^k, ..., 2^K} to |u| (ties up), read off the binary32 exponent.
__device__ __forceinline__ uint32_t pow2_code(float u, int k, int K, int bits)
{
    const uint32_t zero_idx = (1u << (bits - 1)) - 1u;
    if (u == 0.0f) return zero_idx;
    const uint32_t ub = __float_as_uint(u);
    const uint32_t sign = (ub >> 31) << (bits - 1);
    const uint32_t ab = ub & 0x7fffffffu;
    const uint32_t lo_b = static_cast<uint32_t>(k + 127) << 23, hi_b = static_cast<uint32_t>(K + 127) << 23;
    int j;
    if (ab <= lo_b) j = k;
    else if (ab >= hi_b) j = K;
    else j = static_cast<int>(ab >> 23) - 127 + ((ab & 0x400000u) ? 1 : 0);  // mantissa >= 1.5 goes up
    return sign | static_cast<uint32_t>(j - k);
}

__device__ __forceinline__ float pow2_value(uint32_t code, int k, int bits)
{
    const uint32_t zero_idx = (1u << (bits - 1)) - 1u;
    const uint32_t idx = code & zero_idx;
    if (idx == zero_idx) return 0.0f;
    const float mag = __uint_as_float(static_cast<uint32_t>(k + static_cast<int>(idx) + 127) << 23);
    return (code >> (bits - 1)) ? -mag : mag;
}

// Encode one coordinate, returning the code and the decoded value Q(u).
// qtab (may be null): fl(i / L) for i = -L .. L at qtab[i + L], the same values the division gives.
template <int QK>
__device__ __forceinline__ uint32_t encode1(float u, float s, const QParams &q, float Lf, int L, float U, float &dec,
                                            const float *qtab = nullptr)
{
    if constexpr (QK == QK_SIGN) {
        const bool pos = u >= 0.0f;
        dec = pos ? s : -s;
        return pos ? 1u : 0u;
    } else if constexpr (QK == QK_UNIF) {
        const int qi = unif_index(u, s, Lf, q.stochastic != 0, U);
        dec = __fmul_rn(s, qtab ? qtab[qi + L] : __fdiv_rn(static_cast<float>(qi), Lf));
        return static_cast<uint32_t>(qi + L);
    } else if constexpr (QK == QK_POW2) {
        const uint32_t c = pow2_code(u, q.pow2_k, q.pow2_K, q.bits);
        dec = pow2_value(c, q.pow2_k, q.bits);
        return c;
    } else {
        dec = u;
        return __float_as_uint(u);
    }
}

// Decode one coordinate of a received message.  utab (may be null) holds fl(i / L), i = -L..L.
template <int QK>
__device__ __forceinline__ float decode1(uint32_t code, float s, const QParams &q, float Lf, int L, const float *utab)
{
    if constexpr (QK == QK_SIGN) {
        return code ? s : -s;
    } else if constexpr (QK == QK_UNIF) {
        const float r = utab ? utab[code] : __fdiv_rn(static_cast<float>(static_cast<int>(code) - L), Lf);
        return __fmul_rn(s, r);
    } else if constexpr (QK == QK_POW2) {
        return pow2_value(code, q.pow2_k, q.bits);
    } else {
        return __uint_as_float(code);
    }
}

template <int QK>
__device__ __forceinline__ constexpr bool has_scale()
{
    return QK == QK_SIGN || QK == QK_UNIF;
}

// The uniform grid's fl(i / L), i = -L .. L, into tab[0 .. 2L] (no barrier; the caller orders it).
// Returns tab, or null when the grid has more than 8 bits (then the division is used directly).
template <int QK>
__device__ __forceinline__ const float *build_qtab(const QParams &q, float *tab)
{
    if (QK != QK_UNIF || q.bits > 8) return nullptr;
    const int L = (1 << (q.bits - 1)) - 1;
    for (int i = threadIdx.x; i <= 2 * L; i += blockDim.x)
        tab[i] = __fdiv_rn(static_cast<float>(i - L), static_cast<float>(L));
    return tab;
}

// Code width: fixed by the kind for the sign (1) and identity (32) mappings, else configured.
template <int QK>
__device__ __forceinline__ int code_bits(const QParams &q)
{
    return QK == QK_SIGN ? 1 : (QK == QK_IDENT ? 32 : q.bits);
}

// ----------------------------------------------------------------------------- scale groups
// (The lookups below read the segment offsets from global memory one by one; per-coordinate
// lookups on tiles that hold several segments go through TileGroups instead.)

__device__ __forceinline__ int64_t group_begin(const Grouping &g, int64_t gi, int64_t d)
{
    if (g.gkind == GK_WHOLE) return 0;
    if (g.gkind == GK_BLOCK) return gi * g.G;
    return g.offsets[gi];
}

__device__ __forceinline__ int64_t group_end(const Grouping &g, int64_t gi, int64_t d)
{
    if (g.gkind == GK_WHOLE) return d;
    if (g.gkind == GK_BLOCK) return min((gi + 1) * g.G, d);
    return g.offsets[gi + 1];
}

// Group of coordinate j; `hint` must be a group index <= the answer (used for segments).
__device__ __forceinline__ int64_t group_of(const Grouping &g, int64_t j, int64_t hint)
{
    if (g.gkind == GK_WHOLE) return 0;
    if (g.gkind == GK_BLOCK) return g.log2G >= 0 ? (j >> g.log2G) : j / g.G;
    int64_t gi = hint;
    while (g.offsets[gi + 1] <= j) ++gi;
    return gi;
}

__device__ __forceinline__ int64_t first_group_of_tile(const Grouping &g, int64_t tile)
{
    if (g.gkind == GK_WHOLE) return 0;
    if (g.gkind == GK_BLOCK) return g.log2G >= 0 ? (tile * kTile) >> g.log2G : (tile * kTile) / g.G;
    return g.tile_group[tile];
}

// The group that holds every coordinate of tile `tile` (of [0, d)), or -1 when the tile spans a
// group boundary.  Uniform over the CTA.
__device__ __forceinline__ int64_t tile_single_group(const Grouping &g, int64_t tile, int64_t d)
{
    if (g.gkind == GK_WHOLE) return 0;
    const int64_t last = min(tile * kTile + static_cast<int64_t>(kTile), d) - 1;
    if (g.gkind == GK_BLOCK) {
        if (g.log2G >= 12) return (tile * kTile) >> g.log2G;  // power-of-two blocks of >= 4096 hold whole tiles
        const int64_t g0 = first_group_of_tile(g, tile);
        return group_of(g, last, g0) == g0 ? g0 : -1;
    }
    const int64_t g0 = g.tile_group[tile];
    return g.offsets[g0 + 1] > last ? g0 : -1;
}

// The segments (GK_SEG) of one tile, for per-coordinate lookups from shared memory: the tile's
// first group and the offsets, from the tile's start, of the groups that start inside it.
constexpr int kTileBounds = 64;
struct TileGroups {
    int64_t g0;
    int nb;                          // groups starting inside the tile; > kTileBounds: not cached
    uint16_t b[kTileBounds];
};

// Fill tg for tile `tile` (all threads; the caller puts a barrier between this and the lookups).
__device__ __forceinline__ void cache_tile_groups(const Grouping &g, int64_t tile, int64_t d, TileGroups &tg)
{
    const int64_t tl = tile * kTile;
    const int64_t n_tiles = (d + kTile - 1) / kTile;
    const int64_t g0 = g.tile_group[tile];
    int64_t last;  // the group holding the tile's last coordinate
    if (tile + 1 < n_tiles) {
        const int64_t gn = g.tile_group[tile + 1];
        last = g.offsets[gn] == tl + kTile ? gn - 1 : gn;
    } else {
        last = g.n_groups - 1;
    }
    const int nb = static_cast<int>(last - g0);
    if (threadIdx.x == 0) {
        tg.g0 = g0;
        tg.nb = nb;
    }
    if (nb <= kTileBounds)
        for (int i = threadIdx.x; i < nb; i += blockDim.x)
            tg.b[i] = static_cast<uint16_t>(g.offsets[g0 + 1 + i] - tl);
}

// Group of coordinate j of the cached tile (falls back to the global scan past kTileBounds groups).
__device__ __forceinline__ int64_t tile_group_of(const Grouping &g, const TileGroups &tg, int64_t tile, int64_t j)
{
    if (tg.nb > kTileBounds) return group_of(g, j, tg.g0);
    const uint32_t x = static_cast<uint32_t>(j - tile * kTile);
    int c = 0;
    for (int i = 0; i < tg.nb; ++i) c += tg.b[i] <= x ? 1 : 0;
    return tg.g0 + c;
}

// --------------------------------------------------------------------------------- packing
// Coordinate j's b-bit code sits at bit j*b of the little-endian word stream.  A float4 slot q
// (coordinates 4q .. 4q+3) spans 4b bits, so for b <= 8 it lies inside word (q*b)/8.

// Load the four codes of slot q.
__device__ __forceinline__ void load_codes4(const uint32_t *__restrict__ words, int64_t q, int bits, uint32_t c[4])
{
    if (bits <= 8) {
        const uint32_t w = __ldg(words + ((q * bits) >> 3));
        const int sh = static_cast<int>((q * bits) & 7) * 4;
        const uint32_t mask = (1u << bits) - 1u;
#pragma unroll
        for (int i = 0; i < 4; ++i) c[i] = (w >> (sh + i * bits)) & mask;
    } else if (bits == 16) {
        const uint2 w = __ldg(reinterpret_cast<const uint2 *>(words) + q);
        c[0] = w.x & 0xffffu;
        c[1] = w.x >> 16;
        c[2] = w.y & 0xffffu;
        c[3] = w.y >> 16;
    } else {
        const uint4 w = __ldg(reinterpret_cast<const uint4 *>(words) + q);
        c[0] = w.x;
        c[1] = w.y;
        c[2] = w.z;
        c[3] = w.w;
    }
}

// Spread the 8 bits of x to bit positions 0, 4, 8, ..., 28.
__device__ __forceinline__ uint32_t spread8_by4(uint32_t x)
{
    x &= 0xffu;
    x = (x | (x << 12)) & 0x000f000fu;
    x = (x | (x << 6)) & 0x03030303u;
    x = (x | (x << 3)) & 0x11111111u;
    return x;
}

// Store the four codes of slot q (the same slot index on every lane is q_lane0 + lane).  Must be
// called by all 32 lanes of the warp.  Only words whose first coordinate lies in [lo, hi) are
// written (lo starts a word; codes of coordinates >= hi are 0, the caller's job), so that two
// ranges that meet at a word boundary never write the same word.
// b = 1: one ballot per component; lanes 8g .. 8g+7 fill word (q_lane0 / 8) + g, whose bit
// 4l + c is component c of lane 8g + l.
// b in {2, 4, 8}: the slot's 4b bits, shifted to its place in the word and OR-ed across the 8/b
// lanes that share the word (compile-time width).
template <int B, bool FULL>
__device__ __forceinline__ void store_codes4_narrow(uint32_t *__restrict__ words, int64_t q, const uint32_t c[4],
                                                    int64_t lo, int64_t hi)
{
    constexpr int per_word = 8 / B;  // slots per word: 4 (b=2), 2 (b=4), 1 (b=8)
    uint32_t v = c[0] | (c[1] << B) | (c[2] << (2 * B)) | (c[3] << (3 * B));
    const int pos = static_cast<int>(q & (per_word - 1));
    v <<= pos * 4 * B;
    if (per_word >= 2) v |= __shfl_xor_sync(0xffffffffu, v, 1);
    if (per_word >= 4) v |= __shfl_xor_sync(0xffffffffu, v, 2);
    const int64_t wi = (q * B) >> 3;
    const int64_t first = 4 * q;  // pos == 0: the word's first coordinate
    if (pos == 0 && (FULL || (first >= lo && first < hi))) words[wi] = v;
}

template <bool FULL = false, bool BALLOT = true>
__device__ __forceinline__ void store_codes4(uint32_t *__restrict__ words, int64_t q, int bits, const uint32_t c[4],
                                             int64_t lo, int64_t hi)
{
    const int lane = threadIdx.x & 31;
    if (bits == 1 && !BALLOT) {
        // b = 1 with three shuffles: lane l's nibble goes to bits 4(l mod 8) of its 8-lane word
        uint32_t v = (c[0] | (c[1] << 1) | (c[2] << 2) | (c[3] << 3)) << (4 * (lane & 7));
        v |= __shfl_xor_sync(0xffffffffu, v, 1);
        v |= __shfl_xor_sync(0xffffffffu, v, 2);
        v |= __shfl_xor_sync(0xffffffffu, v, 4);
        const int64_t wi = q >> 3;
        if ((lane & 7) == 0 && (FULL || (32 * wi >= lo && 32 * wi < hi))) words[wi] = v;
    } else if (bits == 1) {
        const uint32_t b0 = __ballot_sync(0xffffffffu, c[0] != 0);
        const uint32_t b1 = __ballot_sync(0xffffffffu, c[1] != 0);
        const uint32_t b2 = __ballot_sync(0xffffffffu, c[2] != 0);
        const uint32_t b3 = __ballot_sync(0xffffffffu, c[3] != 0);
        if (lane < 4) {
            const int sh = 8 * lane;
            const uint32_t w = spread8_by4(b0 >> sh) | (spread8_by4(b1 >> sh) << 1) | (spread8_by4(b2 >> sh) << 2) |
                               (spread8_by4(b3 >> sh) << 3);
            const int64_t wi = ((q - lane) >> 3) + lane;  // q - lane is lane 0's slot
            if (FULL || (32 * wi >= lo && 32 * wi < hi)) words[wi] = w;
        }
    } else if (bits == 2) {
        store_codes4_narrow<2, FULL>(words, q, c, lo, hi);
    } else if (bits == 4) {
        store_codes4_narrow<4, FULL>(words, q, c, lo, hi);
    } else if (bits == 8) {
        store_codes4_narrow<8, FULL>(words, q, c, lo, hi);
    } else if (bits == 16) {
        if (FULL || (4 * q >= lo && 4 * q < hi))
            reinterpret_cast<uint2 *>(words)[q] = make_uint2(c[0] | (c[1] << 16), c[2] | (c[3] << 16));
    } else {
        if (FULL || (4 * q >= lo && 4 * q < hi))
            reinterpret_cast<uint4 *>(words)[q] = make_uint4(c[0], c[1], c[2], c[3]);
    }
}

// The Adam moment update and step.  Form 0, the paper's (Algorithm 2): no bias correction, eps
// only as v_0, step alpha m / sqrt(v).  Form 1, the textbook one: v_0 = 0 and step
// alpha (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps).
__device__ __forceinline__ float adam_step(float g, float &m, float &v, const Hyper &h)
{
    v = __fadd_rn(__fmul_rn(h.beta2, v), __fmul_rn(h.c2, __fmul_rn(g, g)));
    m = __fadd_rn(__fmul_rn(h.beta1, m), __fmul_rn(h.c1, g));
    if (h.form == 0) return __fdiv_rn(__fmul_rn(h.alpha, m), __fsqrt_rn(v));
    const float mh = __fdiv_rn(m, h.bc1), vh = __fdiv_rn(v, h.bc2);
    return __fdiv_rn(__fmul_rn(h.alpha, mh), __fadd_rn(__fsqrt_rn(vh), h.eps));
}

// ------------------------------------------------------------------------ vector helpers

__device__ __forceinline__ void to_arr(const float4 &v, float a[4])
{
    a[0] = v.x;
    a[1] = v.y;
    a[2] = v.z;
    a[3] = v.w;
}

__device__ __forceinline__ float4 to_f4(const float a[4]) { return make_float4(a[0], a[1], a[2], a[3]); }

// Load slot q of p (4 coordinates from 4q) into a; coordinates >= d read as 0.  FULL: the caller
// knows the slot lies inside [0, d).
template <bool FULL = false>
__device__ __forceinline__ void load4(const float *__restrict__ p, int64_t q, int64_t d, float a[4])
{
    const int64_t j0 = 4 * q;
    if (FULL || j0 + 4 <= d) {
        to_arr(__ldcs(reinterpret_cast<const float4 *>(p) + q), a);
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) a[i] = (j0 + i < d) ? p[j0 + i] : 0.0f;
    }
}

template <bool FULL = false>
__device__ __forceinline__ void store4(float *__restrict__ p, int64_t q, int64_t d, const float a[4])
{
    const int64_t j0 = 4 * q;
    if (FULL || j0 + 4 <= d) {
        __stcs(reinterpret_cast<float4 *>(p) + q, to_f4(a));
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (j0 + i < d) p[j0 + i] = a[i];
    }
}

}  // namespace ea
