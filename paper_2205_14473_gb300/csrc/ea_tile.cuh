// ea_tile.cuh -- the common end of a worker or server tile: given the residual-corrected input u
// of the tile's 4096 coordinates (held in registers, 16 per thread), form the group scale, encode
// and pack the message, and keep the residual e = u - Q(u) (Algorithm 1 / Algorithm 2).
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

// Encode u (valid coordinates only) with scale s, store codes (all lanes) and the residual.
// FULL: the whole tile lies inside [0, d), so no coordinate needs a bounds check.
// Variants of the per-coordinate encode, chosen once per tile: the uniform grid's zero scale
// (every q = 0), deterministic or stochastic rounding, decode from the fl(i/L) table or by division.
enum EncVar : int { ENC_PLAIN = 0, ENC_UZERO, ENC_UDET_TAB, ENC_UDET_DIV, ENC_USTO_TAB, ENC_USTO_DIV };

template <int QK, bool FULL, bool BALLOT, int VAR>
__device__ __forceinline__ void encode_store_v(float (&u)[kSlots][4], float s, int64_t tile, int64_t d,
                                               const QParams &q, uint32_t *words, float *resid, int ef,
                                               uint64_t seed, uint32_t id, uint32_t t, const float *qtab)
{
    constexpr bool STO = VAR == ENC_USTO_TAB || VAR == ENC_USTO_DIV;
    constexpr bool TAB = VAR == ENC_UDET_TAB || VAR == ENC_USTO_TAB;
    const int bits = code_bits<QK>(q);
    const int L = (QK == QK_UNIF) ? unif_L(bits) : 0;
    const float Lf = static_cast<float>(L);
    const int64_t n_words = (d * bits + 31) >> 5;
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t qs = slot_of(tile, k);
        const int64_t j0 = 4 * qs;
        float U[4] = {0.f, 0.f, 0.f, 0.f};
        if (STO && (FULL || j0 < d)) uniforms4(seed, id, t, j0, U);
        uint32_t c[4];
        float e[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float dec = 0.0f;
            uint32_t code = 0u;
            if (VAR == ENC_PLAIN) {
                code = encode1<QK>(u[k][i], s, q, Lf, L, U[i], dec, qtab);
            } else if (VAR == ENC_UZERO) {
                code = static_cast<uint32_t>(L);  // Example 1: Q = 0 when the scale is 0
            } else {
                // Example 1 with s > 0: z = u / s, y = z L, then the grid index (see unif_index)
                const float y = __fmul_rn(__fdiv_rn(u[k][i], s), Lf);
                int qi;
                if (STO) {
                    const float f = floorf(y);
                    qi = static_cast<int>(f) + (U[i] < __fsub_rn(y, f) ? 1 : 0);
                } else {
                    qi = __float2int_rn(y);
                }
                dec = __fmul_rn(s, TAB ? qtab[qi + L] : __fdiv_rn(static_cast<float>(qi), Lf));
                code = static_cast<uint32_t>(qi + L);
            }
            c[i] = (FULL || j0 + i < d) ? code : 0u;
            e[i] = ef ? __fsub_rn(u[k][i], dec) : 0.0f;
        }
        store_codes4<FULL, BALLOT>(words, qs, bits, c, n_words);
        if (ef && (FULL || j0 < d)) store4<FULL>(resid, qs, d, e);
    }
}

// Encode u (valid coordinates only) with scale s, store codes (all lanes) and the residual.
// FULL: the whole tile lies inside [0, d), so no coordinate needs a bounds check.
template <int QK, bool FULL, bool BALLOT = true>
__device__ __forceinline__ void encode_store(float (&u)[kSlots][4], float s, int64_t tile, int64_t d,
                                             const QParams &q, uint32_t *words, float *resid, int ef,
                                             uint64_t seed, uint32_t id, uint32_t t, const float *qtab)
{
    if constexpr (QK == QK_UNIF) {
        if (!(s > 0.0f))
            encode_store_v<QK, FULL, BALLOT, ENC_UZERO>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab);
        else if (q.stochastic && qtab)
            encode_store_v<QK, FULL, BALLOT, ENC_USTO_TAB>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab);
        else if (q.stochastic)
            encode_store_v<QK, FULL, BALLOT, ENC_USTO_DIV>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab);
        else if (qtab)
            encode_store_v<QK, FULL, BALLOT, ENC_UDET_TAB>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab);
        else
            encode_store_v<QK, FULL, BALLOT, ENC_UDET_DIV>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab);
    } else {
        encode_store_v<QK, FULL, BALLOT, ENC_PLAIN>(u, s, tile, d, q, words, resid, ef, seed, id, t, qtab);
    }
}

// The tile's end for a quantizer with scale groups.
//   PASS_FUSED: the tile is exactly one scale group (blocks of 4096): reduce, encode, store.
//   PASS_STASH: store u in resid and one partial norm per (tile, group) for finalize/encode.
// BALLOT: pack 1-bit codes with __ballot_sync (worker kernels) or with shuffles (the server, whose
// tile loop is instruction-bound).
template <int QK, bool FULL = false, bool BALLOT = true>
__device__ __forceinline__ void finish_tile(float (&u)[kSlots][4], int64_t tile, int64_t d, const QParams &q,
                                            uint32_t *words, float *scales, float *resid, int ef, int pass,
                                            uint64_t seed, uint32_t id, uint32_t t, double *partials,
                                            TileSmem &sm)
{
    if constexpr (!has_scale<QK>()) {
        encode_store<QK, FULL, BALLOT>(u, 0.0f, tile, d, q, words, resid, ef, seed, id, t, nullptr);
        return;
    } else {
        const int64_t tile_lo = tile * kTile;
        const int64_t tile_hi = min(tile_lo + static_cast<int64_t>(kTile), d);
        if (pass == PASS_FUSED) {
            float s;
            if constexpr (QK == QK_SIGN) {
                DF acc{0.0f, 0.0f};
#pragma unroll
                for (int k = 0; k < kSlots; ++k)
#pragma unroll
                    for (int i = 0; i < 4; ++i) df_accumulate(acc, fabsf(u[k][i]));  // invalid u are 0
                s = block_sign_scale(acc, tile_hi - tile_lo, sm.red256, &sm.bcastf);
            } else {
                float mx = 0.0f;
#pragma unroll
                for (int k = 0; k < kSlots; ++k)
#pragma unroll
                    for (int i = 0; i < 4; ++i) mx = fmaxf(mx, fabsf(u[k][i]));
                s = block_max_all(mx, sm.redm);
            }
            if (threadIdx.x == 0) scales[tile] = s;
            // sm.qtab was filled by build_qtab before the reduction's barrier
            encode_store<QK, FULL, BALLOT>(u, s, tile, d, q, words, resid, ef, seed, id, t,
                                           (QK == QK_UNIF && q.bits <= 8) ? sm.qtab : nullptr);
            return;
        }
        // PASS_STASH
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int64_t qs = slot_of(tile, k);
            if (FULL || 4 * qs < d) store4<FULL>(resid, qs, d, u[k]);
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
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (j0 + i >= lo && j0 + i < hi) df_accumulate(acc, fabsf(u[k][i]));
                }
                part = block_sum(acc, sm.red, &sm.bcast);
            } else {
                float mx = 0.0f;
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    const int64_t j0 = 4 * slot_of(tile, k);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        if (j0 + i >= lo && j0 + i < hi) mx = fmaxf(mx, fabsf(u[k][i]));
                }
                part = static_cast<double>(block_max(mx, sm.redm, &sm.bcastf));
            }
            if (threadIdx.x == 0) partials[G.pair_base[gi] + (tile - gb / kTile)] = part;
            if (ge >= tile_hi) break;
        }
    }
}

}  // namespace ea
