// ea_tile.cuh -- the common end of a worker or server tile: given the residual-corrected input u
// of the tile's 4096 coordinates (16 per thread, in registers or parked in shared memory), form
// the group scale, encode and pack the message, and keep the residual e = u - Q(u) (Algorithm 1 /
// Algorithm 2).
#pragma once

#include "ea_device.cuh"

namespace ea {

struct TileSmem {
    DF red256[kThreads];  // per-thread partial pairs of the l1 scale
    DF red[kWarps];
    uint32_t redm[kWarps];
    double bcast;
    float bcastf;
    float qtab[256];  // the uniform grid's fl(i / L) of the tile's own quantizer (build_qtab)
};

// Slot k of this thread in tile `tile`: coordinates 4q .. 4q+3.  Consecutive threads own
// consecutive float4 slots, so every warp access is one contiguous 512-byte segment.
__device__ __forceinline__ int64_t slot_of(int64_t tile, int k)
{
    return tile * (kTile / 4) + k * kThreads + threadIdx.x;
}

// Where a tile's u comes from: this thread's registers (16 values), or shared memory, one float4 per
// slot at ls = k * kThreads + threadIdx.x.
struct URegs {
    float (*u)[4];
    __device__ __forceinline__ void get(int k, float (&o)[4]) const
    {
#pragma unroll
        for (int i = 0; i < 4; ++i) o[i] = u[k][i];
    }
};
struct USmem {
    const float4 *p;
    __device__ __forceinline__ void get(int k, float (&o)[4]) const
    {
        const float4 v = p[k * kThreads + threadIdx.x];
        o[0] = v.x, o[1] = v.y, o[2] = v.z, o[3] = v.w;
    }
};

// Example 1's grid index of u (|u| <= s, s > 0) without a division.  z = RN(u / s) and y = RN(z L)
// are stood in for by z' = RN(u r), y' = RN(z' L) with r = RN(1 / s), which the caller computes
// once per tile.  For s in [2^-125, 2^125] the relative errors of r, z', z and the two products
// (each at most 2^-24, |z| <= 1) give |y' - y| <= 5.01 * 2^-24 * L, below the margin m = L * 2^-20.
// The index changes only where y crosses a half-integer (round to nearest even) or, for the
// stochastic rule, an integer or the draw U; when y' is farther than m from every such point, y
// lies on the same side of each and gets the same index (so does u = 0, where y' = y = 0).
// Returns false otherwise, and for r = NaN, which the caller passes for scales outside the range:
// the caller then takes the index from unif_index, whose division gives z itself.
template <bool STO>
__device__ __forceinline__ bool unif_index_fast(float u, float r, float Lf, float m, float U, int &qi)
{
    const float y = __fmul_rn(__fmul_rn(u, r), Lf);
    if constexpr (STO) {
        const float f = floorf(y);
        const float fr = __fsub_rn(y, f);  // exact: |y| <= L + 1 < 2^23
        qi = static_cast<int>(f) + (U < fr ? 1 : 0);
        // u = 0 gives y' = y = 0 and index 0 exactly
        return (fr > m && fr < __fsub_rn(1.0f, m) && fabsf(__fsub_rn(U, fr)) > m) || u == 0.0f;
    } else {
        const float rn = rintf(y);
        qi = static_cast<int>(rn);
        return fabsf(__fsub_rn(y, rn)) < __fsub_rn(0.5f, m);
    }
}

// Encode u (valid coordinates only) with scale s, store codes (all lanes) and the residual.
// FULL: the whole tile lies inside [0, d), so no coordinate needs a bounds check.
// Variants of the per-coordinate encode, chosen once per tile: the uniform grid's zero scale
// (every q = 0), deterministic or stochastic rounding, decode from the fl(i/L) table or by division.
enum EncVar : int { ENC_PLAIN = 0, ENC_UZERO, ENC_UDET_TAB, ENC_UDET_DIV, ENC_USTO_TAB, ENC_USTO_DIV };

// BITS: the code width as a compile-time constant (0: code_bits of the kind, or q.bits).
// Only the coordinates of [lo, d) are encoded and stored (lo: 0, or the start of a word and a slot).
template <int QK, bool FULL, bool BALLOT, int VAR, int BITS, class USrc>
__device__ __forceinline__ void encode_store_v(const USrc &src, float s, int64_t tile, int64_t d,
                                               const QParams &q, uint32_t *words, float *resid, int ef,
                                               uint64_t seed, uint32_t id, uint32_t t, const float *qtab,
                                               int64_t lo = 0)
{
    constexpr bool STO = VAR == ENC_USTO_TAB || VAR == ENC_USTO_DIV;
    constexpr bool TAB = VAR == ENC_UDET_TAB || VAR == ENC_USTO_TAB;
    constexpr bool GRID = VAR != ENC_PLAIN && VAR != ENC_UZERO;
    const int bits = BITS ? BITS : code_bits<QK>(q);
    const int L = (QK == QK_UNIF) ? unif_L(bits) : 0;
    const float Lf = static_cast<float>(L);
    float r = 0.0f, m = 0.0f;
    if (GRID) {
        r = (s >= 0x1p-125f && s <= 0x1p125f) ? __frcp_rn(s) : __int_as_float(0x7fc00000);
        m = __fmul_rn(Lf, 0x1p-20f);
    }
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t qs = slot_of(tile, k);
        const int64_t j0 = 4 * qs;
        float U[4] = {0.f, 0.f, 0.f, 0.f};
        if (STO && (FULL || j0 < d)) uniforms4(seed, id, t, j0, U);
        float uk[4];
        src.get(k, uk);
        uint32_t c[4];
        float e[4];
        int qi[4] = {0, 0, 0, 0};
        if (GRID) {
            // Example 1 with s > 0: the index of y = RN(RN(u / s) L) (see unif_index_fast)
            bool ok[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) ok[i] = unif_index_fast<STO>(uk[i], r, Lf, m, U[i], qi[i]);
            if (!(ok[0] && ok[1] && ok[2] && ok[3])) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (!ok[i]) qi[i] = unif_index(uk[i], s, Lf, STO, U[i]);
            }
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float dec = 0.0f;
            uint32_t code = 0u;
            if (VAR == ENC_PLAIN) {
                code = encode1<QK>(uk[i], s, q, Lf, L, U[i], dec, qtab);
            } else if (VAR == ENC_UZERO) {
                code = static_cast<uint32_t>(L);  // Example 1: Q = 0 when the scale is 0
            } else {
                dec = __fmul_rn(s, TAB ? qtab[qi[i] + L] : __fdiv_rn(static_cast<float>(qi[i]), Lf));
                code = static_cast<uint32_t>(qi[i] + L);
            }
            c[i] = (FULL || j0 + i < d) ? code : 0u;
            e[i] = ef ? __fsub_rn(uk[i], dec) : 0.0f;
        }
        store_codes4<FULL, BALLOT>(words, qs, bits, c, lo, d);
        if (ef && (FULL || (j0 >= lo && j0 < d))) store4<FULL>(resid, qs, d, e);
    }
}

// Encode u (valid coordinates only) with scale s, store codes (all lanes) and the residual.
// FULL: the whole tile lies inside [0, d), so no coordinate needs a bounds check.
// Example 1 with a compile-time width: for b <= 8 the caller passes qtab (fl(i/L) of the tile's
// quantizer) and the decode is a table read; 16-bit grids divide.
template <int QK, bool FULL, bool BALLOT, int BITS, class USrc>
__device__ __forceinline__ void encode_store_unif(const USrc &u, float s, int64_t tile, int64_t d,
                                                  const QParams &q, uint32_t *words, float *resid, int ef,
                                                  uint64_t seed, uint32_t id, uint32_t t, const float *qtab,
                                                  int64_t lo = 0)
{
    constexpr bool tab = BITS <= 8;
    if (!(s > 0.0f))
        encode_store_v<QK, FULL, BALLOT, ENC_UZERO, BITS>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo);
    else if (q.stochastic)
        encode_store_v<QK, FULL, BALLOT, tab ? ENC_USTO_TAB : ENC_USTO_DIV, BITS>(u, s, tile, d, q, words, resid, ef,
                                                                               seed, id, t, qtab, lo);
    else
        encode_store_v<QK, FULL, BALLOT, tab ? ENC_UDET_TAB : ENC_UDET_DIV, BITS>(u, s, tile, d, q, words, resid, ef,
                                                                               seed, id, t, qtab, lo);
}

// Encode and store a tile; the variant (and a configured code width) is chosen once per tile.
template <int QK, bool FULL, bool BALLOT, class USrc>
__device__ __forceinline__ void encode_store(const USrc &u, float s, int64_t tile, int64_t d,
                                             const QParams &q, uint32_t *words, float *resid, int ef,
                                             uint64_t seed, uint32_t id, uint32_t t, const float *qtab,
                                             int64_t lo = 0)
{
    if constexpr (QK == QK_UNIF) {
        switch (q.bits) {  // the widths ea_init accepts
        case 2: encode_store_unif<QK, FULL, BALLOT, 2>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo); break;
        case 4: encode_store_unif<QK, FULL, BALLOT, 4>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo); break;
        case 8: encode_store_unif<QK, FULL, BALLOT, 8>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo); break;
        default: encode_store_unif<QK, FULL, BALLOT, 16>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo); break;
        }
    } else if constexpr (QK == QK_POW2) {
        if (q.bits == 4)
            encode_store_v<QK, FULL, BALLOT, ENC_PLAIN, 4>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo);
        else
            encode_store_v<QK, FULL, BALLOT, ENC_PLAIN, 8>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo);
    } else {
        encode_store_v<QK, FULL, BALLOT, ENC_PLAIN, 0>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab, lo);
    }
}

// The tile's end when the tile is one scale group (or Q has no scale) and u sits in shared memory
// (USmem layout); l1 / mx are this thread's partial sum / maximum of |u| over its valid coordinates.
template <int QK, bool FULL, bool BALLOT>
__device__ __forceinline__ void finish_tile_smem(const float4 *ubuf, DF l1, float mx, int64_t tile, int64_t d,
                                                 const QParams &q, uint32_t *words, float *scales, float *resid,
                                                 int ef, uint64_t seed, uint32_t id, uint32_t t, TileSmem &sm)
{
    float s = 0.0f;
    if constexpr (has_scale<QK>()) {
        const int64_t tile_lo = tile * kTile;
        const int64_t tile_hi = min(tile_lo + static_cast<int64_t>(kTile), d);
        if constexpr (QK == QK_SIGN)
            s = block_sign_scale(l1, tile_hi - tile_lo, sm.red256, &sm.bcastf);
        else
            s = block_max_all(mx, sm.redm);
        if (threadIdx.x == 0) scales[tile] = s;
    }
    encode_store<QK, FULL, BALLOT>(USmem{ubuf}, s, tile, d, q, words, resid, ef, seed, id, t,
                                   (QK == QK_UNIF && q.bits <= 8) ? sm.qtab : nullptr);
}

// PASS_LAZY on a tile that lies inside one scale group: a compile-time refinement of the pass
// (one partial norm, no per-coordinate group bounds), chosen per tile by the lazy kernels.
constexpr int PASS_LAZY_ONE = 16;

// The tile's end for a quantizer with scale groups, u read through `src` (URegs or USmem).
//   PASS_FUSED: the tile is exactly one scale group (blocks of 4096): reduce, encode, store.
//   PASS_STASH: store u in resid and one partial norm per (tile, group) for finalize/encode.
// BALLOT: pack 1-bit codes with __ballot_sync (worker kernels) or with shuffles (the server, whose
// tile loop is instruction-bound).
// PASS: PASS_FUSED or PASS_STASH as a compile-time constant (the other path is then not compiled
// in), or -1 to follow `pass`.
// part_idx (PASS_LAZY_ONE): where the tile's partial norm goes, looked up early by the caller.
template <int QK, bool FULL = false, bool BALLOT = true, int PASS = -1, class USrc>
__device__ __forceinline__ void finish_tile(const USrc &src, int64_t tile, int64_t d, const QParams &q,
                                            uint32_t *words, float *scales, float *resid, int ef, int pass,
                                            uint64_t seed, uint32_t id, uint32_t t, double *partials,
                                            TileSmem &sm, int64_t part_idx = 0)
{
    if constexpr (PASS >= 0) pass = PASS;
    if constexpr (!has_scale<QK>()) {
        encode_store<QK, FULL, BALLOT>(src, 0.0f, tile, d, q, words, resid, ef, seed, id, t, nullptr);
        return;
    } else {
        const int64_t tile_lo = tile * kTile;
        const int64_t tile_hi = min(tile_lo + static_cast<int64_t>(kTile), d);
        if (pass == PASS_FUSED) {
            float s;
            if constexpr (QK == QK_SIGN) {
                DF acc{0.0f, 0.0f};
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    float uk[4];
                    src.get(k, uk);
#pragma unroll
                    for (int i = 0; i < 4; ++i) df_accumulate(acc, fabsf(uk[i]));  // invalid u are 0
                }
                s = block_sign_scale(acc, tile_hi - tile_lo, sm.red256, &sm.bcastf);
            } else {
                float mx = 0.0f;
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    float uk[4];
                    src.get(k, uk);
#pragma unroll
                    for (int i = 0; i < 4; ++i) mx = fmaxf(mx, fabsf(uk[i]));
                }
                s = block_max_all(mx, sm.redm);
            }
            if (threadIdx.x == 0) scales[tile] = s;
            // sm.qtab was filled by build_qtab before the reduction's barrier
            encode_store<QK, FULL, BALLOT>(src, s, tile, d, q, words, resid, ef, seed, id, t,
                                           (QK == QK_UNIF && q.bits <= 8) ? sm.qtab : nullptr);
            return;
        }
        if constexpr (PASS == PASS_LAZY_ONE && QK == QK_SIGN) {
            // u (with error feedback), the codes, and the one group's partial norm of the tile
            // (a compensated sum to ~2^-44, like the per-group loop below; one barrier)
            DF acc{0.0f, 0.0f};
#pragma unroll
            for (int k = 0; k < kSlots; ++k) {
                const int64_t qs = slot_of(tile, k);
                float uk[4];
                src.get(k, uk);
                if (ef && (FULL || 4 * qs < d)) store4<FULL>(resid, qs, d, uk);
                uint32_t c[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    float dec;
                    const uint32_t code = encode1<QK>(uk[i], 0.0f, q, 0.0f, 0, 0.0f, dec);
                    c[i] = (FULL || 4 * qs + i < d) ? code : 0u;
                    df_accumulate(acc, fabsf(uk[i]));  // u beyond d is 0
                }
                store_codes4<FULL, BALLOT>(words, qs, 1, c, 0, d);
            }
            const DF tot = block_sum_lane0(acc, sm.red256);
            if (threadIdx.x == 0) partials[part_idx] = static_cast<double>(tot.hi) + static_cast<double>(tot.lo);
            return;
        }
        // PASS_STASH: u into resid for encode_kernel.  PASS_LAZY (scaled sign): u into resid, where
        // the residual is formed from it and the scale later (lazy_residual; without error feedback
        // the residual stays 0), and the codes now: the sign of u needs no scale.
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int64_t qs = slot_of(tile, k);
            float uk[4];
            src.get(k, uk);
            if ((PASS != PASS_LAZY || ef) && (FULL || 4 * qs < d)) store4<FULL>(resid, qs, d, uk);
            if constexpr (PASS == PASS_LAZY && QK == QK_SIGN) {
                uint32_t c[4];
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    float dec;
                    const uint32_t code = encode1<QK>(uk[i], 0.0f, q, 0.0f, 0, 0.0f, dec);
                    c[i] = (FULL || 4 * qs + i < d) ? code : 0u;
                }
                store_codes4<FULL, BALLOT>(words, qs, 1, c, 0, d);
            }
        }
        const Grouping &G = q.grp;
        for (int64_t gi = first_group_of_tile(G, tile);; ++gi) {
            const int64_t gb = group_begin(G, gi, d), ge = group_end(G, gi, d);
            const int64_t lo = max(gb, tile_lo), hi = min(ge, tile_hi);
            double part;
            if constexpr (QK == QK_SIGN) {
                DF acc{0.0f, 0.0f};
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    const int64_t j0 = 4 * slot_of(tile, k);
                    float uk[4];
                    src.get(k, uk);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (j0 + i >= lo && j0 + i < hi) df_accumulate(acc, fabsf(uk[i]));
                }
                part = block_sum(acc, sm.red, &sm.bcast);
            } else {
                float mx = 0.0f;
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    const int64_t j0 = 4 * slot_of(tile, k);
                    float uk[4];
                    src.get(k, uk);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (j0 + i >= lo && j0 + i < hi) mx = fmaxf(mx, fabsf(uk[i]));
                }
                part = static_cast<double>(block_max(mx, sm.redm, &sm.bcastf));
            }
            if (threadIdx.x == 0) partials[G.pair_base[gi] + (tile - gb / kTile)] = part;
            if (ge >= tile_hi) break;
        }
    }
}

// PASS_LAZY (scaled sign): where the residual e = u - Q(u) of a kept u is formed -- u - (u >= 0 ? s
// : -s), s the scale of the coordinate's group in the previous message (scales).  This is
// e <- u - Q(u) of Algorithm 1 / Algorithm 2 with the same binary32 operations, evaluated where the
// residual is next read.  LazyScale holds a tile's scale when the tile lies in one group (loaded
// once, early), else the group to start the per-coordinate lookups from.
struct LazyScale {
    int64_t g1, hint;  // the tile's one group (-1: several), the tile's first group
    float s1;          // the scale of g1
};

__device__ __forceinline__ LazyScale lazy_scale_of_tile(const QParams &q, const float *scales, int64_t tile, int64_t d)
{
    LazyScale ls;
    ls.g1 = tile_single_group(q.grp, tile, d);
    ls.hint = first_group_of_tile(q.grp, tile);
    ls.s1 = ls.g1 >= 0 ? scales[ls.g1] : 0.0f;
    return ls;
}

// The residual of the kept u of coordinates j0 .. j0+3 (in place in e); coordinates >= d unchanged.
template <bool FULL>
__device__ __forceinline__ void lazy_residual4(const QParams &q, const float *scales, const LazyScale &ls, int64_t j0,
                                               int64_t d, float (&e)[4])
{
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        if (FULL || j0 + i < d) {
            const float s = ls.g1 >= 0 ? ls.s1 : scales[group_of(q.grp, j0 + i, ls.hint)];
            float dec;
            (void)encode1<QK_SIGN>(e[i], s, q, 0.0f, 0, 0.0f, dec);
            e[i] = __fsub_rn(e[i], dec);
        }
    }
}

// The same for all of this thread's slots of tile `tile`.
// The same for a tile inside one group, whose previous scale is s.
template <bool FULL>
__device__ __forceinline__ void lazy_residual_one(const QParams &q, float s, int64_t tile, int64_t d,
                                                  float (&e)[kSlots][4])
{
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t j0 = 4 * slot_of(tile, k);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (FULL || j0 + i < d) {
                float dec;
                (void)encode1<QK_SIGN>(e[k][i], s, q, 0.0f, 0, 0.0f, dec);
                e[k][i] = __fsub_rn(e[k][i], dec);
            }
        }
    }
}

template <bool FULL>
__device__ __forceinline__ void lazy_residual(const QParams &q, const float *scales, int64_t tile, int64_t d,
                                              float (&e)[kSlots][4])
{
    const LazyScale ls = lazy_scale_of_tile(q, scales, tile, d);
#pragma unroll
    for (int k = 0; k < kSlots; ++k) lazy_residual4<FULL>(q, scales, ls, 4 * slot_of(tile, k), d, e[k]);
}

}  // namespace ea
