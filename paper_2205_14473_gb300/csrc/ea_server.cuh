// ea_server.cuh -- the server's round (Algorithm 1) on one 4096-coordinate tile.
#pragma once

#include <atomic>

#include "ea_async.cuh"
#include "ea_grouped.cuh"
#include "ea_tile.cuh"

namespace ea {

// The worker-order sum of the n decoded worker messages at this thread's 16 coordinates of tile
// `tile` (coordinates >= d give 0), read straight from global memory.  utab: fl(i / L) of the
// workers' uniform grid (b_w <= 8) or null; stab: 256 floats of shared memory for the sign table.
// Contains a CTA barrier (all threads call it; the caller orders stab's previous readers before it).
template <int QW>
__device__ __forceinline__ void decode_sum_direct(const ServerArgs &a, int64_t tile, const float *utab, float *stab,
                                                  TileGroups &tg, float (&acc)[kSlots][4])
{
    const int64_t d = a.d;
    const int Lw = (QW == QK_UNIF) ? unif_L(a.qw.bits) : 0;
    const float Lwf = static_cast<float>(Lw);
    // The workers' scale of a coordinate: one per worker for the whole tile when the tile lies
    // in one of Q_w's groups (always for 4096-blocks), else a per-coordinate group lookup.
    const Grouping &GW = a.qw.grp;
    const int64_t wg = has_scale<QW>() ? tile_single_group(GW, tile, d) : 0;
    const bool wtile = wg >= 0;
    const int64_t whint = first_group_of_tile(GW, tile);
#pragma unroll
    for (int k = 0; k < kSlots; ++k)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[k][i] = 0.0f;

    // Scaled-sign workers with one scale each for the tile: the worker-order sum of the first
    // m = min(n, 8) workers depends only on their m sign bits.  Thread p forms that sum for pattern
    // p (worker w's sign at bit pi(w), pi = (0, 4, 1, 5, 2, 6, 3, 7)) from 0, as the loop below
    // would; a coordinate's pattern is gathered from X (bit 4w + i = worker w's code of slot
    // coordinate i) by ((X >> i) & 0x11111111) * 0x01020408 >> 24, which carries no bits.  The
    // remaining workers are then added in order.
    int w_first = 0;
    if constexpr (QW == QK_SIGN) {
        if (wtile) {
            const int m = min(a.n, 8);
            constexpr uint32_t pi = 0x73625140u;  // pi(w) in nibble w
            float t = 0.0f;
            for (int w = 0; w < m; ++w) {
                const float sw = __ldg(a.wscales + static_cast<int64_t>(w) * a.wscales_stride + wg);
                t = __fadd_rn(t, ((threadIdx.x >> ((pi >> (4 * w)) & 7u)) & 1u) ? sw : -sw);
            }
            stab[threadIdx.x] = t;
            __syncthreads();
            const int sh = 4 * (threadIdx.x & 7);  // this thread's nibble in every code word
#pragma unroll
            for (int k = 0; k < kSlots; ++k) {
                const int64_t q = slot_of(tile, k);
                if (4 * q >= d) continue;
                uint32_t X = 0;
#pragma unroll
                for (int w = 0; w < 8; ++w) {
                    if (w < m) {
                        const uint32_t word = __ldg(a.wwords + static_cast<int64_t>(w) * a.wwords_stride + (q >> 3));
                        X |= __funnelshift_r(word, word, (sh - 4 * w) & 31) & (0xfu << (4 * w));
                    }
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[k][i] = stab[(((X >> i) & 0x11111111u) * 0x01020408u) >> 24];
            }
            w_first = m;
        }
    }

    // a tile over several groups: each coordinate's group, looked up once (segments from shared
    // memory), as an offset from the tile's first group (a tile of 4096 coordinates meets at most
    // 4096 groups: 16 bits per coordinate)
    const bool seg = has_scale<QW>() && !wtile && GW.gkind == GK_SEG;
    if (seg) {
        cache_tile_groups(GW, tile, d, tg);
        __syncthreads();
    }
    uint32_t gl[kSlots][2] = {{0u, 0u}, {0u, 0u}, {0u, 0u}, {0u, 0u}};
    if (has_scale<QW>() && !wtile) {
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int64_t j0 = 4 * slot_of(tile, k);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int64_t j = j0 + i < d ? j0 + i : d - 1;
                const int64_t g = (seg ? tile_group_of(GW, tg, tile, j) : group_of(GW, j, whint)) - whint;
                gl[k][i >> 1] |= static_cast<uint32_t>(g) << (16 * (i & 1));
            }
        }
    }
#pragma unroll 2
    for (int w = w_first; w < a.n; ++w) {
        const uint32_t *ww = a.wwords + static_cast<int64_t>(w) * a.wwords_stride;
        const float *wsc = a.wscales + static_cast<int64_t>(w) * a.wscales_stride;
        const float s_tile = (has_scale<QW>() && wtile) ? __ldg(wsc + wg) : 0.0f;
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int64_t q = slot_of(tile, k);
            const int64_t j0 = 4 * q;
            if (j0 >= d) continue;
            uint32_t c[4];
            load_codes4(ww, q, code_bits<QW>(a.qw), c);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                if (j0 + i < d) {
                    float s = 0.0f;
                    if (has_scale<QW>())
                        s = wtile ? s_tile : __ldg(wsc + whint + ((gl[k][i >> 1] >> (16 * (i & 1))) & 0xffffu));
                    acc[k][i] = __fadd_rn(acc[k][i], decode1<QW>(c[i], s, a.qw, Lwf, Lw, utab));
                }
            }
        }
    }
}

// The workers' uniform grid's fl(i / L), i = -L .. L, into utab (b_w <= 8; no barrier).
template <int QW>
__device__ __forceinline__ const float *build_worker_utab(const ServerArgs &a, float *utab)
{
    if (QW != QK_UNIF || a.qw.bits > 8) return nullptr;
    const int Lw = unif_L(a.qw.bits);
    for (int i = threadIdx.x; i <= 2 * Lw; i += blockDim.x)
        utab[i] = __fdiv_rn(static_cast<float>(i - Lw), static_cast<float>(Lw));
    return utab;
}

// Decode the n worker messages of this tile, average them (summed in worker order, one division
// by n), add the server residual (and, with Adam at the server, take the Adam step on the
// average first), then Q_s and e_s <- w - Q_s(w) (finish_tile).
// HBM traffic per coordinate: n b_w/8 B of worker codes + 4 B e_s read + 4 B e_s written + b_s/8 B
// of broadcast code (+ 16 B for m, v with Adam at the server).
template <int MODE, int QW, int QS>
__global__ void __launch_bounds__(kThreads, 2) server_kernel(const ServerArgs a)
{
    __shared__ TileSmem sm;
    __shared__ float utab_s[256];  // fl(i / L) for the workers' uniform grid, i = -L..L (b_w <= 8)
    __shared__ float stab[256];
    __shared__ TileGroups tg;
    const int64_t tile = blockIdx.x;
    const int64_t d = a.d;

    pdl_trigger();
    build_qtab<QS>(a.qs, sm.qtab);  // read after the scale reduction's barrier
    const float *utab = build_worker_utab<QW>(a, utab_s);
    if (utab) __syncthreads();
    pdl_wait();

    float es[kSlots][4], ms[kSlots][4], vs[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        load4(a.es, q, d, es[k]);
        if (MODE == MODE_S) {
            load4(a.ms, q, d, ms[k]);
            load4(a.vs, q, d, vs[k]);
        }
    }
    float acc[kSlots][4];
    decode_sum_direct<QW>(a, tile, utab, stab, tg, acc);

    const float nf = static_cast<float>(a.n);
    const bool pow2n = (a.n & (a.n - 1)) == 0;
    const float inv_n = __frcp_rn(nf);  // exact when n is a power of two
    float u[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float step = pow2n ? __fmul_rn(acc[k][i], inv_n) : __fdiv_rn(acc[k][i], nf);
            if (MODE == MODE_S) step = adam_step(step, ms[k][i], vs[k][i], a.hp);
            u[k][i] = (j0 + i < d) ? __fadd_rn(step, es[k][i]) : 0.0f;
        }
        if (MODE == MODE_S && j0 < d) {
            store4(a.ms, q, d, ms[k]);
            store4(a.vs, q, d, vs[k]);
        }
    }
    finish_tile<QS>(URegs{u}, tile, d, a.qs, a.words, a.scales, a.es, a.ef, a.pass, a.seed,
                    static_cast<uint32_t>(a.n), a.t, a.partials, sm);
}

// Phase one of a grouped server tile: w (the average, after the Adam step with Adam at the server,
// plus e_s) of the coordinate range [lo, hi) of tile `tile` (0 elsewhere) into ub; m_s and v_s
// updated and stored in the range.  FULL: the range is the whole tile.
template <int MODE, int QW, bool FULL, bool LAZY = false>
__device__ __forceinline__ void server_u_range(const ServerArgs &a, int64_t tile, int64_t lo, int64_t hi, float4 *ub,
                                               const float *utab, float *stab, TileGroups &tg)
{
    LazyScale lzs{};
    if (LAZY && a.lazy_in) lzs = lazy_scale_of_tile(a.qs, a.scales, tile, a.d);
    float acc[kSlots][4];
    decode_sum_direct<QW>(a, tile, utab, stab, tg, acc);
    const float nf = static_cast<float>(a.n);
    const bool pow2n = (a.n & (a.n - 1)) == 0;
    const float inv_n = __frcp_rn(nf);  // exact when n is a power of two
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
        const bool in = FULL || (j0 >= lo && j0 < hi);
        float es[4] = {0.f, 0.f, 0.f, 0.f}, ms[4] = {0.f, 0.f, 0.f, 0.f}, vs[4] = {1.f, 1.f, 1.f, 1.f}, u[4];
        if (in) {
            load4<FULL>(a.es, q, hi, es);
            if (MODE == MODE_S) {
                load4<FULL>(a.ms, q, hi, ms);
                load4<FULL>(a.vs, q, hi, vs);
            }
            if (LAZY && a.lazy_in) lazy_residual4<FULL>(a.qs, a.scales, lzs, j0, hi, es);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float step = pow2n ? __fmul_rn(acc[k][i], inv_n) : __fdiv_rn(acc[k][i], nf);
            if (MODE == MODE_S) step = adam_step(step, ms[i], vs[i], a.hp);
            u[i] = (in && (FULL || j0 + i < hi)) ? __fadd_rn(step, es[i]) : 0.0f;
        }
        ub[k * kThreads + threadIdx.x] = make_float4(u[0], u[1], u[2], u[3]);
        if (MODE == MODE_S && in) {
            store4<FULL>(a.ms, q, hi, ms);
            store4<FULL>(a.vs, q, hi, vs);
        }
    }
}

// Load the four codes of local slot ls (0 .. 1023) of a tile's code chunk held in shared memory.
__device__ __forceinline__ void load_codes4_smem(const uint32_t *words, int ls, int bits, uint32_t c[4])
{
    if (bits <= 8) {
        const uint32_t w = words[(ls * bits) >> 3];
        const int sh = ((ls * bits) & 7) * 4;
        const uint32_t mask = (1u << bits) - 1u;
#pragma unroll
        for (int i = 0; i < 4; ++i) c[i] = (w >> (sh + i * bits)) & mask;
    } else if (bits == 16) {
        const uint2 w = reinterpret_cast<const uint2 *>(words)[ls];
        c[0] = w.x & 0xffffu;
        c[1] = w.x >> 16;
        c[2] = w.y & 0xffffu;
        c[3] = w.y >> 16;
    } else {
        const uint4 w = reinterpret_cast<const uint4 *>(words)[ls];
        c[0] = w.x;
        c[1] = w.y;
        c[2] = w.z;
        c[3] = w.w;
    }
}


// Whether the grouped server stages a tile's worker codes in shared memory: all n chunks must fit
// in the tile's slot (4096 b_w / 8 bytes each, 16 KB in all).
__device__ __forceinline__ bool server_codes_fit(const ServerArgs &a, int bw) { return a.n * bw <= 32; }

// The worker-order sum of the n decoded worker messages at this thread's 16 coordinates of tile
// `tile`, from the tile's code chunks staged in shared memory (cw: worker w's chunk at
// w * chunk_words) and the workers' scales of the tile's groups (wsc: worker w's scale of the
// tile's group gw0 + g at w * ngw + g).  seg: the tile holds several of Q_w's segments (tg holds
// them); ngw > 1 without seg: several blocks (looked up arithmetically).  Contains a CTA barrier.
template <int QW>
__device__ __forceinline__ void decode_sum_staged(const ServerArgs &a, int64_t tile, const uint32_t *cw,
                                                  int chunk_words, const float *wsc, int ngw, int64_t gw0, bool seg,
                                                  const TileGroups &tg, float *stab, const float *utab,
                                                  float (&acc)[kSlots][4])
{
    const int n = a.n;
    const int bw = code_bits<QW>(a.qw);
    const int Lw = (QW == QK_UNIF) ? unif_L(a.qw.bits) : 0;
    const float Lwf = static_cast<float>(Lw);
    const Grouping &GW = a.qw.grp;
#pragma unroll
    for (int k = 0; k < kSlots; ++k)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[k][i] = 0.0f;
    int w_first = 0;
    if constexpr (QW == QK_SIGN) {
        if (ngw == 1) {
            // the worker-order sum of the first m = min(n, 8) workers by sign pattern (worker w's
            // code at bit pi(w), pi = (0, 4, 1, 5, 2, 6, 3, 7)), thread p forming pattern p's sum as
            // the loop below would
            const int m = min(n, 8);
            constexpr uint32_t pi = 0x73625140u;  // pi(w) in nibble w
            float t = 0.0f;
            for (int w = 0; w < m; ++w)
                t = __fadd_rn(t, ((threadIdx.x >> ((pi >> (4 * w)) & 7u)) & 1u) ? wsc[w] : -wsc[w]);
            stab[threadIdx.x] = t;
            compute_sync();
            const int sh = 4 * (threadIdx.x & 7);  // this thread's nibble in every code word
#pragma unroll
            for (int k = 0; k < kSlots; ++k) {
                const int ls = k * kThreads + threadIdx.x;
                uint32_t X = 0;  // bit 4w + i: worker w's code of the slot's coordinate i
#pragma unroll
                for (int w = 0; w < 8; ++w)
                    if (w < m) X |= ((cw[w * chunk_words + (ls >> 3)] >> sh) & 0xfu) << (4 * w);
                // bits 4w of X >> i times 0x01020408 land, without carries, at 24 + pi(w)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[k][i] = stab[(((X >> i) & 0x11111111u) * 0x01020408u) >> 24];
            }
            w_first = m;
        }
    }
    // each coordinate's group within the tile (0 .. ngw - 1 <= 255: the caller's table bound),
    // looked up once, one byte per coordinate of a slot
    uint32_t gl[kSlots] = {0u, 0u, 0u, 0u};
    if (has_scale<QW>() && ngw > 1) {
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int64_t j0 = 4 * slot_of(tile, k);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int64_t j = j0 + i < a.d ? j0 + i : a.d - 1;
                const int64_t g = (seg ? tile_group_of(GW, tg, tile, j) : group_of(GW, j, gw0)) - gw0;
                gl[k] |= static_cast<uint32_t>(g) << (8 * i);
            }
        }
    }
    if constexpr (QW == QK_SIGN) {
        if (ngw == 1) {
            // the workers past the table, in order: each one's sign nibble of the slot, then a
            // select of +-s_w and one addition per coordinate
#pragma unroll 1
            for (int w = w_first; w < n; ++w) {
                const uint32_t *ww = cw + w * chunk_words;
                const float sw = wsc[w], nsw = -sw;
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    const int ls = k * kThreads + threadIdx.x;
                    const uint32_t nib = ww[ls >> 3] >> (4 * (ls & 7));
#pragma unroll
                    for (int i = 0; i < 4; ++i) acc[k][i] = __fadd_rn(acc[k][i], ((nib >> i) & 1u) ? sw : nsw);
                }
            }
            return;
        }
    }
#pragma unroll 1
    for (int w = w_first; w < n; ++w) {
        const uint32_t *ww = cw + w * chunk_words;
        const float *ws = wsc + w * ngw;
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int ls = k * kThreads + threadIdx.x;
            uint32_t c[4];
            load_codes4_smem(ww, ls, bw, c);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float s = has_scale<QW>() ? ws[(gl[k] >> (8 * i)) & 0xffu] : 0.0f;
                acc[k][i] = __fadd_rn(acc[k][i], decode1<QW>(c[i], s, a.qw, Lwf, Lw, utab));
            }
        }
    }
}

// Phase one of a grouped server tile, inputs staged in shared memory: the tile's worker code
// chunks go into the tile's own slot ub (free until w lands in it) and the workers' scales of its
// groups into wsc, all loads issued at once; then the decode reads shared memory only.  w (the
// average, after the Adam step with Adam at the server, plus e_s) of the range [lo, hi) then
// replaces the codes in ub (0 outside the range); m_s, v_s are updated and stored in the range.
// Returns false, having done nothing, when the tile's scale table would not fit (the caller then
// takes server_u_range).
template <int MODE, int QW, bool FULL, bool LAZY = false>
__device__ __forceinline__ bool server_u_staged(const ServerArgs &a, int64_t tile, int64_t lo, int64_t hi, float4 *ub,
                                                const float *utab, float *stab, float *wsc, GroupSmem &gs)
{
    const int64_t d = a.d;
    const int n = a.n;
    const int bw = code_bits<QW>(a.qw);
    const Grouping &GW = a.qw.grp;
    int64_t gw0 = 0;
    int ngw = 1;
    if (has_scale<QW>()) {
        gw0 = first_group_of_tile(GW, tile);
        const int64_t last = min(tile * kTile + static_cast<int64_t>(kTile), d) - 1;
        ngw = static_cast<int>(group_of(GW, last, gw0) - gw0 + 1);
        if (n * ngw > kWorkerScales || ngw > kStagedTileGroups) return false;
    }
    const bool seg = has_scale<QW>() && ngw > 1 && GW.gkind == GK_SEG;
    float es[kSlots][4], ms[kSlots][4], vs[kSlots][4];
    bool in[kSlots];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        in[k] = FULL || (4 * q >= lo && 4 * q < hi);
#pragma unroll
        for (int i = 0; i < 4; ++i) es[k][i] = ms[k][i] = 0.0f, vs[k][i] = 1.0f;
        if (in[k]) {
            load4<FULL>(a.es, q, hi, es[k]);
            if (MODE == MODE_S) {
                load4<FULL>(a.ms, q, hi, ms[k]);
                load4<FULL>(a.vs, q, hi, vs[k]);
            }
        }
    }
    compute_sync();  // the slot's and the tables' previous readers are done
    const int chunk_words = kTile * bw / 32;
    uint32_t *cw = reinterpret_cast<uint32_t *>(ub);
    {
        const int64_t cbase = tile * chunk_words;          // the tile's chunk in every code stream
        const int64_t avail = a.wcode_bytes / 4 - cbase;   // words of the (padded) stream from there
        const int nvec = n * chunk_words / 4;
        // every copy issued at once (cp.async: no register round trip), then one wait
        for (int v = threadIdx.x; v < nvec; v += kThreads) {
            const int w = (4 * v) / chunk_words, o = (4 * v) % chunk_words;
            uint4 *dst = reinterpret_cast<uint4 *>(cw) + v;
            if (o + 4 <= avail) cp_async16(dst, a.wwords + static_cast<int64_t>(w) * a.wwords_stride + cbase + o);
            else *dst = make_uint4(0u, 0u, 0u, 0u);
        }
        if (has_scale<QW>())
            for (int i = threadIdx.x; i < n * ngw; i += kThreads)
                cp_async4(wsc + i, a.wscales + static_cast<int64_t>(i / ngw) * a.wscales_stride + gw0 + i % ngw);
        if (seg) cache_tile_groups(GW, tile, d, gs.tg);
        cp_async_wait_all();
    }
    compute_sync();
    float acc[kSlots][4];
    decode_sum_staged<QW>(a, tile, cw, chunk_words, wsc, ngw, gw0, seg, gs.tg, stab, utab, acc);
    compute_sync();  // every thread has read the staged codes
    if constexpr (LAZY) {
        if (a.lazy_in) {  // es holds the previous round's w: its residual (lo is the tile's start)
            const LazyScale lzs = lazy_scale_of_tile(a.qs, a.scales, tile, d);
#pragma unroll
            for (int k = 0; k < kSlots; ++k)
                if (in[k]) lazy_residual4<FULL>(a.qs, a.scales, lzs, 4 * slot_of(tile, k), hi, es[k]);
        }
    }
    const float nf = static_cast<float>(n);
    const bool pow2n = (n & (n - 1)) == 0;
    const float inv_n = __frcp_rn(nf);  // exact when n is a power of two
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
        float u[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float step = pow2n ? __fmul_rn(acc[k][i], inv_n) : __fdiv_rn(acc[k][i], nf);
            if (MODE == MODE_S) step = adam_step(step, ms[k][i], vs[k][i], a.hp);
            u[i] = (in[k] && (FULL || j0 + i < hi)) ? __fadd_rn(step, es[k][i]) : 0.0f;
        }
        ub[k * kThreads + threadIdx.x] = make_float4(u[0], u[1], u[2], u[3]);
        if (MODE == MODE_S && in[k]) {
            store4<FULL>(a.ms, q, hi, ms[k]);
            store4<FULL>(a.vs, q, hi, vs[k]);
        }
    }
    return true;
}

// Algorithm 1 for Q_s scale groups that span tiles, in one cooperative pass (PASS_GROUPED; see
// GroupPlan and worker_grouped_kernel): phase one decodes, averages and parks w of the CTA's
// tiles of a wave in shared memory and queues the partial norms, published once per wave; phase
// two encodes Q_s(w) and stores e_s <- w - Q_s(w).
template <int MODE, int QW, int QS>
__global__ void __launch_bounds__(kThreads, MODE == MODE_S ? 2 : 3) server_grouped_kernel(const ServerArgs a)
{
    extern __shared__ __align__(16) float4 uslot[];  // a.gp.slots tiles of w
    __shared__ GroupSmem gs;
    __shared__ float utab_s[256];
    __shared__ float stab[256];
    __shared__ float wsc[kWorkerScales];
    build_qtab<QS>(a.qs, gs.qtab);
    const float *utab = build_worker_utab<QW>(a, utab_s);
    __syncthreads();
    const bool staged = server_codes_fit(a, code_bits<QW>(a.qw));
    const GroupPlan &gp = a.gp;
    int turn = 0;  // reductions so far (the same count in every thread)
    for (int w = 0; w < static_cast<int>(gp.n_waves); ++w) {
        const int64_t c0 = gp.cuts[w], c1 = gp.cuts[w + 1];
        const int t0 = static_cast<int>(c0 / kTile) + blockIdx.x;   // tiles < 2^28 (d <= 2^40)
        const int t_end = static_cast<int>((c1 - 1) / kTile) + 1;
        int k = 0;
        for (int tile = t0; tile < t_end; tile += gridDim.x, ++k) {
            float4 *ub = uslot + k * (kThreads * kSlots);
            const int64_t tl = static_cast<int64_t>(tile) * kTile, lo = max(c0, tl), hi = min(c1, tl + kTile);
            const bool full = lo == tl && hi == tl + kTile;
            bool done = false;
            if (staged)
                done = full ? server_u_staged<MODE, QW, true>(a, tile, lo, hi, ub, utab, stab, wsc, gs)
                            : server_u_staged<MODE, QW, false>(a, tile, lo, hi, ub, utab, stab, wsc, gs);
            if (!done) {
                compute_sync();  // stab's and tg's previous readers are done
                if (full) server_u_range<MODE, QW, true>(a, tile, lo, hi, ub, utab, stab, gs.tg);
                else server_u_range<MODE, QW, false>(a, tile, lo, hi, ub, utab, stab, gs.tg);
            }
            range_partials<QS>(ub, tile, lo, hi, a.d, a.qs, a.partials, gs, turn);
        }
        if (!wave_barrier(gp, w, a.status, gs)) return;
        encode_wave<QS>(uslot, t0, t_end, c0, c1, a.d, a.qs, a.words, a.partials, a.scales, a.es, a.ef, a.seed,
                        static_cast<uint32_t>(a.n), a.t, gs);
    }
}


// PASS_LAZY for a scaled-sign broadcast whose groups span tiles, one CTA per tile.  w (the average,
// after the Adam step with Adam at the server, plus the residual formed from the previous round's
// kept w) is stored as the broadcast's signs, which need no scale, and in es as the kept w, with the
// groups' partial norms; finalize_kernel then forms the broadcast scales.  No CTA waits for another.
// STAGED: every tile's worker codes and scales fit the shared-memory staging (the host checks
// server_codes_fit and the groups per tile), and only that path is compiled in; else direct loads.
template <int MODE, int QW, bool STAGED>
__global__ void __launch_bounds__(kThreads, MODE == MODE_S ? 2 : 3) server_lazy_kernel(const ServerArgs a)
{
    __shared__ float4 ub[kSlots * kThreads];
    __shared__ GroupSmem gs;
    __shared__ float utab_s[256];
    __shared__ float stab[256];
    __shared__ float wsc[kWorkerScales];
    pdl_trigger();
    const float *utab = build_worker_utab<QW>(a, utab_s);
    __syncthreads();
    pdl_wait();
    const int64_t tile = blockIdx.x;
    const int64_t d = a.d, lo = tile * kTile, hi = min(lo + static_cast<int64_t>(kTile), d);
    const bool full = hi == lo + kTile;
    if constexpr (STAGED) {
        const bool done = full ? server_u_staged<MODE, QW, true, true>(a, tile, lo, hi, ub, utab, stab, wsc, gs)
                               : server_u_staged<MODE, QW, false, true>(a, tile, lo, hi, ub, utab, stab, wsc, gs);
        if (!done) {  // outside what the host checked: report it, store nothing
            if (threadIdx.x == 0) report_status(a.status, kStatusCheck);
            return;
        }
    } else {
        if (full) server_u_range<MODE, QW, true, true>(a, tile, lo, hi, ub, utab, stab, gs.tg);
        else server_u_range<MODE, QW, false, true>(a, tile, lo, hi, ub, utab, stab, gs.tg);
    }
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t qs = slot_of(tile, k);
        const float4 v = ub[k * kThreads + threadIdx.x];
        const float w[4] = {v.x, v.y, v.z, v.w};
        uint32_t c[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float dec;
            const uint32_t code = encode1<QK_SIGN>(w[i], 0.0f, a.qs, 0.0f, 0, 0.0f, dec);
            c[i] = (4 * qs + i < d) ? code : 0u;
        }
        store_codes4<false, false>(a.words, qs, 1, c, 0, d);
        if (a.ef && 4 * qs < d) store4(a.es, qs, d, w);
    }
    int turn = 0;
    range_partials<QK_SIGN>(ub, tile, lo, hi, d, a.qs, a.partials, gs, turn);
}

template <int MODE, bool STAGED>
static cudaError_t launch_server_lazy_st(const ServerArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>(a.n_tiles)), block(kThreads);
    switch (a.qw.kind) {
    case QK_SIGN: return launch_pdl(server_lazy_kernel<MODE, QK_SIGN, STAGED>, grid, block, 0, s, a);
    case QK_UNIF: return launch_pdl(server_lazy_kernel<MODE, QK_UNIF, STAGED>, grid, block, 0, s, a);
    case QK_POW2: return launch_pdl(server_lazy_kernel<MODE, QK_POW2, STAGED>, grid, block, 0, s, a);
    default: return launch_pdl(server_lazy_kernel<MODE, QK_IDENT, STAGED>, grid, block, 0, s, a);
    }
}

template <int MODE>
cudaError_t launch_server_lazy(const ServerArgs &a, bool staged, cudaStream_t s)
{
    return staged ? launch_server_lazy_st<MODE, true>(a, s) : launch_server_lazy_st<MODE, false>(a, s);
}

constexpr int kWorkerTab = 1024;  // floats of the staged server's per-tile worker table

// Bits 0, 4, ..., 28 of x moved to bits 0 .. 7 (the inverse of spread8_by4).
__device__ __forceinline__ uint32_t gather_every4(uint32_t x)
{
    x &= 0x11111111u;
    x = (x | (x >> 3)) & 0x03030303u;
    x = (x | (x >> 6)) & 0x000f000fu;
    x = (x | (x >> 12)) & 0x000000ffu;
    return x;
}

// All 256 compute threads agree on `ok` (named barrier 1 with an AND reduction).
__device__ __forceinline__ bool compute_all(bool ok)
{
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "bar.red.and.pred q, 1, %2, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(ok ? 1u : 0u), "n"(kThreads)
        : "memory");
    return r != 0;
}

// Transpose the 8x8 bit matrix whose bit 8r + c is row r, column c (rows 0-3 in lo, 4-7 in hi):
// three delta swaps of 1-, 2- and 4-bit blocks (Hacker's Delight, section 7-3).
__device__ __forceinline__ void transpose8x8(uint32_t &lo, uint32_t &hi)
{
    uint32_t t;
    t = ((lo >> 7) ^ lo) & 0x00aa00aau, lo ^= t ^ (t << 7);
    t = ((hi >> 7) ^ hi) & 0x00aa00aau, hi ^= t ^ (t << 7);
    t = ((lo >> 14) ^ lo) & 0x0000ccccu, lo ^= t ^ (t << 14);
    t = ((hi >> 14) ^ hi) & 0x0000ccccu, hi ^= t ^ (t << 14);
    t = ((hi << 4) ^ lo) & 0xf0f0f0f0u, lo ^= t, hi ^= t >> 4;
}

// Sum, in worker order, the decoded values of n workers' B-bit uniform-grid codes of this thread's
// four slots, reading each decoded value from the per-tile table wtab (worker w's 2^B - 1 values
// from w * 2^B); a tile's chunk holds kTile * B / 8 bytes per worker.  The worker loop is
// kept rolled (two workers per iteration) so that the hot loop stays small in the instruction
// cache; the slots and coordinates inside it are unrolled.
// PAIRS (B = 4): the thread-pair decode below (used with Adam at the workers; with Adam at the
// server the per-thread form measured faster, the Adam step leaving fewer registers).
// NW > 0: the worker count n is NW, known at compile time (the worker loop is then unrolled).
template <int B, bool PAIRS, int NW = 0>
__device__ __forceinline__ void unif_decode_sum(const unsigned char *codes, int n_rt, const float *wtab,
                                                float (&acc)[kSlots][4])
{
    const int n = NW ? NW : n_rt;
    constexpr int chunk_words = kTile * B / 32;
    constexpr uint32_t mask = (1u << B) - 1u;
    // the slot's 4B bits start at bit 4 B ls of the chunk, ls = k * kThreads + threadIdx.x
    if constexpr (B == 4 && PAIRS) {
        // 4-bit codes, thread pairs: a code word holds the 8 coordinates of a pair (2q, 2q+1) in
        // one slot.  The even thread decodes the pair's word in slots 0, 2, the odd one in slots 1,
        // 3; two shift-and-masks put every code times 4 in a byte (even coordinates in a, odd in
        // b), one byte permute per coordinate takes it out, and at the end one shuffle per
        // coordinate hands each thread the half that is its own.
        static_assert(kSlots % 2 == 0, "slots are taken in pairs");
        const bool odd = threadIdx.x & 1;
        const uint32_t *pw = reinterpret_cast<const uint32_t *>(codes) + (threadIdx.x >> 1) + (odd ? kThreads / 2 : 0);
        const unsigned char *tb = reinterpret_cast<const unsigned char *>(wtab);
        float blk[kSlots / 2][8];
#pragma unroll
        for (int h = 0; h < kSlots / 2; ++h)
#pragma unroll
            for (int j = 0; j < 8; ++j) blk[h][j] = 0.0f;
#pragma unroll(NW ? NW : 2)
        for (int w = 0; w < n; ++w, pw += chunk_words, tb += 4 << B) {
#pragma unroll
            for (int h = 0; h < kSlots / 2; ++h) {
                const uint32_t word = pw[h * kThreads];  // slot 2h (+1 for the odd thread), word q
                const uint32_t ev = (word << 2) & 0x3c3c3c3cu, od = (word >> 2) & 0x3c3c3c3cu;
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint32_t o0 = __byte_perm(ev, 0u, 0x4440u | j), o1 = __byte_perm(od, 0u, 0x4440u | j);
                    blk[h][2 * j] = __fadd_rn(blk[h][2 * j], *reinterpret_cast<const float *>(tb + o0));
                    blk[h][2 * j + 1] = __fadd_rn(blk[h][2 * j + 1], *reinterpret_cast<const float *>(tb + o1));
                }
            }
        }
#pragma unroll
        for (int h = 0; h < kSlots / 2; ++h)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float recv = __shfl_xor_sync(0xffffffffu, odd ? blk[h][i] : blk[h][4 + i], 1);
                acc[2 * h][i] = odd ? recv : blk[h][i];
                acc[2 * h + 1][i] = odd ? blk[h][4 + i] : recv;
            }
        return;
    }
    const int sh = ((static_cast<int>(threadIdx.x) * B) & 7) * 4;
    const uint32_t *cw = reinterpret_cast<const uint32_t *>(codes) + ((static_cast<int>(threadIdx.x) * B) >> 3);
    const unsigned char *tb = reinterpret_cast<const unsigned char *>(wtab);
#pragma unroll(NW ? NW : 2)
    for (int w = 0; w < n; ++w, cw += chunk_words, tb += 4 << B) {
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const uint32_t word = cw[(k * kThreads * B) >> 3];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                // rotating right by (position - 2) mod 32 puts the field, times 4 (a byte offset
                // into worker w's table), at bits 2 .. B+1: one shift and one mask
                const uint32_t off = __funnelshift_r(word, word, (sh + i * B - 2) & 31) & (mask << 2);
                acc[k][i] = __fadd_rn(acc[k][i], *reinterpret_cast<const float *>(tb + off));
            }
        }
    }
}

// One tile of the staged server on the compute warps: the stage `st` holds e_s (m_s, v_s), the
// workers' code chunks and scales.  The stage's e_s slots then hold u until the re-quantization
// has read it; the stage is released (arrive on `empty`) after that.
// NW: the worker count when it is 8, known at compile time (the per-worker bounds, the average's
// division and the decode loops then fold; for scaled-sign workers the table is the whole average
// and the per-worker path is not compiled in), or 0 for a count known at run time.
template <int MODE, int QW, int QS, bool FULL, int NW>
__device__ __forceinline__ bool server_staged_tile(const ServerArgs &a, int64_t tile, const unsigned char *st,
                                                   bool ok, uint64_t *empty, int Lw, float Lwf, const float *utab,
                                                   float *wtab, const uint32_t (&flip)[8], TileSmem &sm)
{
    static_assert(NW == 0 || NW == 8, "a compile-time worker count of 8");
    const StagePlan &P = a.plan;
    const int64_t d = a.d;
    const int bw = code_bits<QW>(a.qw);
    const int n = NW ? NW : a.n;
    const float nf = static_cast<float>(n);
    const bool pow2n = (n & (n - 1)) == 0;
    const float inv_n = NW ? 1.0f / NW : __frcp_rn(nf);  // exact when n is a power of two
    float acc[kSlots][4];  // the average of the decoded worker messages
    const float *sc = reinterpret_cast<const float *>(st + P.off_scales);
    bool done = false;
    // wtab is rebuilt below; the previous tile's reads of it end at its scale reduction's barrier,
    // which a Q_s without scales does not have
    if constexpr (!has_scale<QS>() && (QW == QK_SIGN || QW == QK_UNIF)) compute_sync();
    if constexpr (QW == QK_SIGN) {
      {
        done = NW == 8 || n <= 8;
        // Scaled-sign workers: the worker-order sum of the first m = min(n, 8) workers depends
        // only on their m sign bits.  Thread p forms it for sign pattern p (bit w = worker w's
        // code), exactly as the per-coordinate loop would; for n <= 8 it is divided by n and is
        // the average, for n > 8 the remaining workers are added after it in order.
        {
            float t = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; ++w)
                if (w < n) t = __fadd_rn(t, __uint_as_float(__float_as_uint(sc[w]) ^ flip[w]));
            wtab[threadIdx.x] = !done ? t : pow2n ? __fmul_rn(t, inv_n) : __fdiv_rn(t, nf);
        }
        // the table's barrier, and agreement on the stage wait: if any thread's wait ran out, the
        // entries just written may hold stale stage data and the tile is abandoned unread
        if (!compute_all(ok)) return false;
        // Patterns of eight consecutive coordinates at a time: byte b of every worker's code word
        // (8 coordinates x 8 workers) gathered into two registers, the 8x8 bit matrix transposed,
        // and byte j is then coordinate j's pattern.  Of a thread pair (2q, 2q+1), the even thread
        // transposes the pair's block in slot k and the odd one in slot k+1; one shuffle swaps
        // the halves that belong to the other thread.
        const uint32_t *c0 = reinterpret_cast<const uint32_t *>(st + P.off_codes);
        const unsigned char *tb = reinterpret_cast<const unsigned char *>(wtab);
        static_assert(kSlots % 2 == 0, "slots are taken in pairs");
        const bool odd = threadIdx.x & 1;
        const uint32_t bsel = (threadIdx.x >> 1) & 3;  // the block's byte in its word
        const uint32_t sel = bsel | ((bsel + 4) << 4);
#pragma unroll
        for (int k = 0; k < kSlots; k += 2) {
            const int word = 32 * (k + (odd ? 1 : 0)) + static_cast<int>(threadIdx.x >> 3);
            uint32_t wd[8];
#pragma unroll
            for (int w = 0; w < 8; ++w) wd[w] = w < n ? c0[w * (kTile / 32) + word] : 0u;
            uint32_t lo = __byte_perm(__byte_perm(wd[0], wd[1], sel), __byte_perm(wd[2], wd[3], sel), 0x5410);
            uint32_t hi = __byte_perm(__byte_perm(wd[4], wd[5], sel), __byte_perm(wd[6], wd[7], sel), 0x5410);
            transpose8x8(lo, hi);
            const uint32_t recv = __shfl_xor_sync(0xffffffffu, odd ? lo : hi, 1);
            const uint32_t pk = odd ? recv : lo, pk1 = odd ? hi : recv;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                // pattern byte i times 4: a byte offset into the table
                const uint32_t o0 = (i == 0 ? pk << 2 : pk >> (8 * i - 2)) & 0x3fcu;
                const uint32_t o1 = (i == 0 ? pk1 << 2 : pk1 >> (8 * i - 2)) & 0x3fcu;
                acc[k][i] = *reinterpret_cast<const float *>(tb + o0);
                acc[k + 1][i] = *reinterpret_cast<const float *>(tb + o1);
            }
        }
      }
    }
    if (!done) {
        // scaled-sign workers (n > 8): acc already holds the sum of workers 0..7
        constexpr bool partial = QW == QK_SIGN;
        if constexpr (!partial) {
#pragma unroll
            for (int k = 0; k < kSlots; ++k)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[k][i] = 0.0f;
        }
        // Uniform-grid workers: every worker's 2L+1 decoded values s_w * fl(i/L) for this tile, as
        // decode1 would form them, so that a coordinate's decode is one table read.
        // Worker w's table starts at w * 2^b; entries 0 .. 2L = 2^b - 2 are used.
        const int nL = 2 * Lw + 1;
        const bool dec_tab = QW == QK_UNIF && utab != nullptr && (n << bw) <= kWorkerTab;
        if (dec_tab) {
            for (int idx = threadIdx.x; idx < (n << bw); idx += kThreads) {
                const int i = idx & ((1 << bw) - 1);
                if (i < nL) wtab[idx] = __fmul_rn(sc[idx >> bw], utab[i]);
            }
        }
        if constexpr (!partial)
            if (!compute_all(ok)) return false;  // the table's barrier and agreement on the stage wait
        bool summed = false;
        if constexpr (QW == QK_UNIF) {
            if (dec_tab && bw == 4) {
                unif_decode_sum<4, MODE == MODE_W, NW>(st + P.off_codes, n, wtab, acc);
                summed = true;
            } else if (dec_tab && bw == 8) {
                unif_decode_sum<8, false, NW>(st + P.off_codes, n, wtab, acc);
                summed = true;
            }
        }
        if (!summed) {  // any worker count and code width; kept rolled (it is not the common case)
#pragma unroll 1
            for (int w = partial ? 8 : 0; w < n; ++w) {
                const uint32_t *cw = reinterpret_cast<const uint32_t *>(st + P.off_codes + static_cast<size_t>(w) * P.code_chunk);
                const float sw = has_scale<QW>() ? sc[w] : 0.0f;
                const float *dw = wtab + (w << bw);
#pragma unroll
                for (int k = 0; k < kSlots; ++k) {
                    uint32_t c[4];
                    load_codes4_smem(cw, k * kThreads + threadIdx.x, bw, c);
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        acc[k][i] = __fadd_rn(acc[k][i], dec_tab ? dw[c[i]] : decode1<QW>(c[i], sw, a.qw, Lwf, Lw, utab));
                }
            }
        }
        // the average: a multiplication by 1/n is exact for n a power of two (one branch per tile)
        if (pow2n) {
#pragma unroll
            for (int k = 0; k < kSlots; ++k)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[k][i] = __fmul_rn(acc[k][i], inv_n);
        } else {
#pragma unroll
            for (int k = 0; k < kSlots; ++k)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[k][i] = __fdiv_rn(acc[k][i], nf);
        }
    }
    // e_s (and m_s, v_s) are read from the stage only now, to keep registers for the sums.  Each
    // slot's u goes back into the stage over its e_s (only this thread reads it again), so that no
    // register holds u across the scale's reduction.
    float4 *ubuf = reinterpret_cast<float4 *>(const_cast<unsigned char *>(st) + P.off_a);
    DF l1{0.0f, 0.0f};
    float mx = 0.0f;
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int ls = k * kThreads + threadIdx.x;
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
        float es[4], ms[4], vs[4], u[4];
        to_arr(ubuf[ls], es);
        if (MODE == MODE_S) {
            to_arr(reinterpret_cast<const float4 *>(st + P.off_b)[ls], ms);
            to_arr(reinterpret_cast<const float4 *>(st + P.off_c)[ls], vs);
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float step = acc[k][i];
            if (MODE == MODE_S) step = adam_step(step, ms[i], vs[i], a.hp);
            u[i] = (FULL || j0 + i < d) ? __fadd_rn(step, es[i]) : 0.0f;  // invalid u are 0
            if constexpr (QS == QK_SIGN) df_accumulate(l1, fabsf(u[i]));
            else mx = fmaxf(mx, fabsf(u[i]));
        }
        ubuf[ls] = make_float4(u[0], u[1], u[2], u[3]);
        if (MODE == MODE_S && (FULL || j0 < d)) {
            store4<FULL>(a.ms, q, d, ms);
            store4<FULL>(a.vs, q, d, vs);
        }
    }
    finish_tile_smem<QS, FULL, false>(ubuf, l1, mx, tile, d, a.qs, a.words, a.scales, a.es, a.ef, a.seed,
                                      static_cast<uint32_t>(a.n), a.t, sm);
    // the stage is no longer read: hand it back to the producer
    __syncwarp();
    if ((threadIdx.x & 31) == 0) mbar_arrive(empty);
    return true;
}

// The server's round with its inputs staged through shared memory.  Persistent CTAs of 8 compute
// warps and 1 producer warp: the producer streams, for each of the CTA's tiles, the e_s tile (and
// m_s, v_s with Adam at the server) and the n workers' code chunks with bulk copies, and the n
// worker scales with 4-byte cp.async, into a ring of stages guarded by full/empty mbarriers; the
// compute warps decode, average, re-quantize and write e_s and the broadcast straight to HBM.
// Used when Q_s scales are per 4096-tile (or absent) and Q_w's are per 4096-tile (or absent).
template <int MODE, int QW, int QS>
__global__ void __launch_bounds__(kThreads + 32, server_ctas_per_sm(MODE, QW, QS)) server_staged_kernel(const ServerArgs a)
{
    extern __shared__ __align__(128) unsigned char dsm[];
    static_assert(sizeof(TileSmem) + sizeof(float) * (256 + kWorkerTab) + 128 <= kServerStaticSmem,
                  "the stage plan's bound on static shared memory");
    __shared__ TileSmem sm;
    __shared__ float utab[256];
    __shared__ float wtab[kWorkerTab];  // per tile: the average of every sign pattern (scaled-sign
                                        // workers) or every worker's decoded grid values (uniform)
    const StagePlan &P = a.plan;
    const int S = P.stages;
    uint64_t *full = reinterpret_cast<uint64_t *>(dsm);
    uint64_t *empty = full + S;
    unsigned char *stage0 = dsm + 128 * ((2 * S * 8 + 127) / 128);
    constexpr bool scaled_w = has_scale<QW>();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    pdl_trigger();

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&full[s], 1 + (scaled_w ? 32 : 0));
            mbar_init(&empty[s], kWarps);
        }
        mbar_init_fence();
    }
    const int Lw = (QW == QK_UNIF) ? unif_L(a.qw.bits) : 0;
    const float Lwf = static_cast<float>(Lw);
    const bool use_tab = QW == QK_UNIF && a.qw.bits <= 8;
    if (use_tab)
        for (int i = threadIdx.x; i <= 2 * Lw; i += blockDim.x) utab[i] = __fdiv_rn(static_cast<float>(i - Lw), Lwf);
    build_qtab<QS>(a.qs, sm.qtab);
    __syncthreads();
    pdl_wait();  // the workers' messages and e_s are written

    if (warp == kWarps) {  // ---------------------------------------------------------- producer
        int64_t it = 0;
        bool ok = true;
        for (int64_t tile = blockIdx.x; tile < a.n_tiles; tile += gridDim.x, ++it) {
            const int s = static_cast<int>(it % S);
            if (it >= S && !mbar_wait(&empty[s], static_cast<uint32_t>(((it / S) & 1) ^ 1))) {
                ok = false;
                break;
            }
            unsigned char *st = stage0 + static_cast<size_t>(s) * P.stage_bytes;
            const int64_t lo = tile * kTile;
            const uint32_t vb = static_cast<uint32_t>(min(static_cast<int64_t>(kTile), a.dpad - lo) * 4);
            const int64_t coff = tile * static_cast<int64_t>(P.code_chunk);
            const uint32_t cb = static_cast<uint32_t>(min(static_cast<int64_t>(P.code_chunk), a.wcode_bytes - coff));
            if (lane == 0) {
                mbar_arrive_expect_tx(&full[s], vb * (MODE == MODE_S ? 3u : 1u) + cb * static_cast<uint32_t>(a.n));
                bulk_g2s(st + P.off_a, a.es + lo, vb, &full[s]);
                if (MODE == MODE_S) {
                    bulk_g2s(st + P.off_b, a.ms + lo, vb, &full[s]);
                    bulk_g2s(st + P.off_c, a.vs + lo, vb, &full[s]);
                }
                const unsigned char *wb = reinterpret_cast<const unsigned char *>(a.wwords) + coff;
                for (int w = 0; w < a.n; ++w)
                    bulk_g2s(st + P.off_codes + static_cast<size_t>(w) * P.code_chunk, wb + w * a.wcode_bytes, cb,
                             &full[s]);
            }
            if (scaled_w) {
                float *sc = reinterpret_cast<float *>(st + P.off_scales);
                for (int w = lane; w < a.n; w += 32) cp_async4(sc + w, a.wscales + w * a.wscales_stride + tile);
                cp_async_arrive_noinc(&full[s]);
            }
        }
        // the copies of the last stages must land before the CTA may exit
        for (int64_t j = (it > S ? it - S : 0); j < it; ++j)
            if (!mbar_wait(&full[j % S], static_cast<uint32_t>((j / S) & 1))) ok = false;
        if (!ok && lane == 0) report_status(a.status, kStatusTimeout);
        return;
    }

    // ------------------------------------------------------------------------- compute warps
    const int64_t d = a.d;
    // sign-pattern table (scaled-sign workers): this thread's pattern p = threadIdx.x gives worker w
    // the sign of bit w of p, kept as a binary32 sign-bit mask
    uint32_t flip[8];
#pragma unroll
    for (int w = 0; w < 8; ++w) flip[w] = ((threadIdx.x >> w) & 1u) ? 0u : 0x80000000u;
    const bool n8 = a.n == 8;  // full tiles with eight workers: the compile-time count
    int64_t it = 0;
    for (int64_t tile = blockIdx.x; tile < a.n_tiles; tile += gridDim.x, ++it) {
        const int s = static_cast<int>(it % S);
        // bounded wait; the tile's first barrier makes every compute thread agree on the outcome
        const bool ok = mbar_wait(&full[s], static_cast<uint32_t>((it / S) & 1));
        const unsigned char *st = stage0 + static_cast<size_t>(s) * P.stage_bytes;
        const bool go = (tile + 1) * kTile <= d
            ? (n8 ? server_staged_tile<MODE, QW, QS, true, 8>(a, tile, st, ok, &empty[s], Lw, Lwf, use_tab ? utab : nullptr, wtab, flip, sm)
                  : server_staged_tile<MODE, QW, QS, true, 0>(a, tile, st, ok, &empty[s], Lw, Lwf, use_tab ? utab : nullptr, wtab, flip, sm))
            : server_staged_tile<MODE, QW, QS, false, 0>(a, tile, st, ok, &empty[s], Lw, Lwf, use_tab ? utab : nullptr, wtab, flip, sm);
        if (!go) {
            if (threadIdx.x == 0) report_status(a.status, kStatusTimeout);
            break;
        }
    }
}

template <int MODE, int QW, int QS>
static cudaError_t launch_server_staged(const ServerArgs &a, cudaStream_t s)
{
    // Function attributes are per device: one flag per device ordinal.  Two threads that race on a
    // first launch both set the same values, which is harmless.
    static std::atomic<bool> attr_set[kMaxDevices];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    if (!attr_set[dev].load(std::memory_order_acquire)) {
        e = cudaFuncSetAttribute(server_staged_kernel<MODE, QW, QS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kServerMaxDynSmem);
        if (e == cudaSuccess)  // all of the SM's unified L1 / shared memory as shared memory
            e = cudaFuncSetAttribute(server_staged_kernel<MODE, QW, QS>,
                                     cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        if (e != cudaSuccess) return e;
        attr_set[dev].store(true, std::memory_order_release);
    }
    return launch_pdl(server_staged_kernel<MODE, QW, QS>, dim3(a.plan.grid), dim3(kThreads + 32), a.plan.smem_bytes, s, a);
}


// The grouped server for one placement and broadcast kind (the uniform grid only).
template <int MODE, int QS>
cudaError_t server_grouped_shape_for_qs(int qw, GroupedShape *out)
{
    if constexpr (QS != QK_UNIF) {
        return cudaErrorNotSupported;
    } else {
        const int w = MODE == MODE_S ? 2 : 3;  // the kernel's launch bounds
        switch (qw) {
        case QK_SIGN: return grouped_shape(server_grouped_kernel<MODE, QK_SIGN, QS>, w, out);
        case QK_UNIF: return grouped_shape(server_grouped_kernel<MODE, QK_UNIF, QS>, w, out);
        case QK_POW2: return grouped_shape(server_grouped_kernel<MODE, QK_POW2, QS>, w, out);
        default: return grouped_shape(server_grouped_kernel<MODE, QK_IDENT, QS>, w, out);
        }
    }
}

template <int MODE, int QS>
cudaError_t launch_server_grouped_for_qs(const ServerArgs &a, int grid, cudaStream_t s)
{
    if constexpr (QS != QK_UNIF) {
        return cudaErrorNotSupported;
    } else {
        const int slots = a.gp.slots;
        switch (a.qw.kind) {
        case QK_SIGN: return grouped_launch(server_grouped_kernel<MODE, QK_SIGN, QS>, a, grid, slots, s);
        case QK_UNIF: return grouped_launch(server_grouped_kernel<MODE, QK_UNIF, QS>, a, grid, slots, s);
        case QK_POW2: return grouped_launch(server_grouped_kernel<MODE, QK_POW2, QS>, a, grid, slots, s);
        default: return grouped_launch(server_grouped_kernel<MODE, QK_IDENT, QS>, a, grid, slots, s);
        }
    }
}

// Launch the server kernel for one placement and one broadcast quantizer kind (each (MODE, QS) pair
// is instantiated in a translation unit of its own, ea_server_<mode>_q<QS>.cu).
template <int MODE, int QS>
cudaError_t launch_server_for_qs(const ServerArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>(a.n_tiles)), block(kThreads);
    switch (a.qw.kind) {
    case QK_SIGN:
        if (a.plan.enabled) return launch_server_staged<MODE, QK_SIGN, QS>(a, s);
        return launch_pdl(server_kernel<MODE, QK_SIGN, QS>, grid, block, 0, s, a);
    case QK_UNIF:
        if (a.plan.enabled) return launch_server_staged<MODE, QK_UNIF, QS>(a, s);
        return launch_pdl(server_kernel<MODE, QK_UNIF, QS>, grid, block, 0, s, a);
    case QK_POW2:
        if (a.plan.enabled) return launch_server_staged<MODE, QK_POW2, QS>(a, s);
        return launch_pdl(server_kernel<MODE, QK_POW2, QS>, grid, block, 0, s, a);
    default:
        if (a.plan.enabled) return launch_server_staged<MODE, QK_IDENT, QS>(a, s);
        return launch_pdl(server_kernel<MODE, QK_IDENT, QS>, grid, block, 0, s, a);
    }
    return cudaGetLastError();
}

}  // namespace ea
