// ea_worker.cu -- worker compress (Algorithm 2), the two-pass scale kernels, and x <- x - Q_s(w).
#include "ea_grouped.cuh"

namespace ea {

// One tile of worker_kernel; FULL: the tile lies inside [0, d) (every tile but a ragged last one).
// Each slot's u goes to ubuf (only this thread reads it again), so that no register holds u across
// the scale's reduction and more CTAs fit on an SM.
template <int MODE, int QK, bool FULL, int PASS>
__device__ __forceinline__ void worker_tile(const WorkerArgs &a, int64_t tile, float4 *ubuf, TileSmem &sm)
{
    const int64_t d = a.d;
    // PASS_LAZY_ONE: the tile's group, its previous scale and the slot of its partial norm, looked
    // up before the tile's loads so that these short dependent loads overlap them
    int64_t part_idx = 0;
    float s_prev = 0.0f;
    if constexpr (PASS == PASS_LAZY_ONE) {
        const Grouping &G = a.q.grp;
        const int64_t g1 = first_group_of_tile(G, tile);
        part_idx = G.pair_base[g1] + (tile - group_begin(G, g1, d) / kTile);
        if (a.lazy_in) s_prev = a.scales[g1];
    }
    float g[kSlots][4], e[kSlots][4], m[kSlots][4], v[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        load4<FULL>(a.g, q, d, g[k]);
        load4<FULL>(a.e, q, d, e[k]);
        if (MODE == MODE_W) {
            load4<FULL>(a.m, q, d, m[k]);
            load4<FULL>(a.v, q, d, v[k]);
        }
    }
    // the grid's fl(i/L) table, built while the loads are in flight (read after the scale
    // reduction's barrier)
    build_qtab<QK>(a.q, sm.qtab);
    if constexpr (PASS == PASS_LAZY) {
        // e holds the previous round's u: its residual is u - Q(u) with the previous scales
        if (a.lazy_in) lazy_residual<FULL>(a.q, a.scales, tile, d, e);
    } else if constexpr (PASS == PASS_LAZY_ONE) {
        if (a.lazy_in) lazy_residual_one<FULL>(a.q, s_prev, tile, d, e);
    }
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
        float u[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float step = g[k][i];
            if (MODE == MODE_W) step = adam_step(g[k][i], m[k][i], v[k][i], a.hp);
            u[i] = (FULL || j0 + i < d) ? __fadd_rn(step, e[k][i]) : 0.0f;
        }
        ubuf[k * kThreads + threadIdx.x] = make_float4(u[0], u[1], u[2], u[3]);
        if (MODE == MODE_W && (FULL || j0 < d)) {
            store4<FULL>(a.m, q, d, m[k]);
            store4<FULL>(a.v, q, d, v[k]);
        }
    }
    finish_tile<QK, FULL, true, PASS>(USmem{ubuf}, tile, d, a.q, a.words, a.scales, a.e, a.ef, a.pass, a.seed, a.id, a.t,
                                      a.partials, sm, part_idx);
}

// Algorithm 2 for one worker on one 4096-coordinate tile.  With Adam at the worker:
//   v <- beta2 v + (1-beta2) g^2, m <- beta1 m + (1-beta1) g, u = alpha m / sqrt(v) + e;
// with Adam at the server: u = g + e.  Then Q_w(u) and e <- u - Q_w(u) (finish_tile).
// HBM traffic per coordinate: 16 B read + 12 B written + b/8 B of code (Adam at the worker).
// Resident CTAs per SM the registers are sized for: four with Adam at the server (g and e per
// coordinate), three with Adam at the worker.  Measured: the server-side-Adam uniform grid runs
// faster at four CTAs with a few bytes of spill than at three without, and the worker-side-Adam
// uniform grid faster at three (80 registers, a few bytes of spill) than at two.
// PASS_LAZY for the scaled sign: the same tile, the codes stored with the partial norms and u kept
// in e (see lazy_residual); one launch per message plus finalize_kernel.
template <int MODE>
__global__ void __launch_bounds__(kThreads, MODE == MODE_S ? 4 : 3)
    worker_lazy_kernel(const WorkerArgs a)
{
    __shared__ TileSmem sm;
    __shared__ float4 ubuf[kSlots * kThreads];
    pdl_trigger();
    pdl_wait();
    const int64_t tile = blockIdx.x;
    if ((tile + 1) * kTile <= a.d) {
        if (tile_single_group(a.q.grp, tile, a.d) >= 0) worker_tile<MODE, QK_SIGN, true, PASS_LAZY_ONE>(a, tile, ubuf, sm);
        else worker_tile<MODE, QK_SIGN, true, PASS_LAZY>(a, tile, ubuf, sm);
    } else {
        worker_tile<MODE, QK_SIGN, false, PASS_LAZY>(a, tile, ubuf, sm);
    }
}

template <int MODE, int QK>
__global__ void __launch_bounds__(kThreads, MODE == MODE_S ? 4 : 3)
    worker_kernel(const WorkerArgs a)
{
    __shared__ TileSmem sm;
    __shared__ float4 ubuf[kSlots * kThreads];
    pdl_trigger();
    pdl_wait();
    const int64_t tile = blockIdx.x;
    // the scale pass as a compile-time constant: each instantiation carries only its own path
    const bool full = (tile + 1) * kTile <= a.d;
    if (a.pass == PASS_FUSED) {
        if (full) worker_tile<MODE, QK, true, PASS_FUSED>(a, tile, ubuf, sm);
        else worker_tile<MODE, QK, false, PASS_FUSED>(a, tile, ubuf, sm);
    } else {
        if (full) worker_tile<MODE, QK, true, PASS_STASH>(a, tile, ubuf, sm);
        else worker_tile<MODE, QK, false, PASS_STASH>(a, tile, ubuf, sm);
    }
}

// Phase one of a grouped worker tile: u of the coordinate range [lo, hi) of tile `tile` (0
// elsewhere) into ub, with m and v updated and stored in the range (Adam at the worker).
// FULL: the range is the whole tile.  All four slots' loads are issued at once (the kernel's
// register budget is sized for it), so that enough bytes are in flight per SM.
template <int MODE, bool FULL>
__device__ __forceinline__ void worker_u_range(const WorkerArgs &a, int64_t tile, int64_t lo, int64_t hi, float4 *ub)
{
    constexpr int H = kSlots;
#pragma unroll
    for (int h = 0; h < kSlots; h += H) {
        float g[H][4], e[H][4], m[H][4], v[H][4];
        bool in[H];
#pragma unroll
        for (int k = 0; k < H; ++k) {
            const int64_t q = slot_of(tile, h + k);
            in[k] = FULL || (4 * q >= lo && 4 * q < hi);
#pragma unroll
            for (int i = 0; i < 4; ++i) g[k][i] = e[k][i] = m[k][i] = 0.0f, v[k][i] = 1.0f;
            if (in[k]) {
                load4<FULL>(a.g, q, hi, g[k]);
                load4<FULL>(a.e, q, hi, e[k]);
                if (MODE == MODE_W) {
                    load4<FULL>(a.m, q, hi, m[k]);
                    load4<FULL>(a.v, q, hi, v[k]);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < H; ++k) {
            const int64_t q = slot_of(tile, h + k);
            const int64_t j0 = 4 * q;
            float u[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float step = g[k][i];
                if (MODE == MODE_W) step = adam_step(g[k][i], m[k][i], v[k][i], a.hp);
                u[i] = (in[k] && (FULL || j0 + i < hi)) ? __fadd_rn(step, e[k][i]) : 0.0f;
            }
            ub[(h + k) * kThreads + threadIdx.x] = make_float4(u[0], u[1], u[2], u[3]);
            if (MODE == MODE_W && in[k]) {
                store4<FULL>(a.m, q, hi, m[k]);
                store4<FULL>(a.v, q, hi, v[k]);
            }
        }
    }
}

// Algorithm 2 for scale groups that span tiles, in one cooperative pass (PASS_GROUPED; see
// GroupPlan): for each wave, every CTA computes u of its tiles into shared memory (phase one) and
// publishes the partial norms; once a group's scale is ready, the tiles are encoded from shared
// memory and e <- u - Q_w(u) stored (phase two).  HBM traffic per coordinate as worker_kernel's:
// no second read of u.
template <int MODE, int QK>
__global__ void __launch_bounds__(kThreads, MODE == MODE_S ? 4 : 2) worker_grouped_kernel(const WorkerArgs a)
{
    extern __shared__ __align__(16) float4 uslot[];  // a.gp.slots tiles of u
    __shared__ GroupSmem gs;
    build_qtab<QK>(a.q, gs.qtab);
    __syncthreads();
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
            if (lo == tl && hi == tl + kTile) worker_u_range<MODE, true>(a, tile, lo, hi, ub);
            else worker_u_range<MODE, false>(a, tile, lo, hi, ub);
            range_partials<QK>(ub, tile, lo, hi, a.d, a.q, a.partials, gs, turn);
        }
        if (!wave_barrier(gp, w, a.status, gs)) return;
        encode_wave<QK>(uslot, t0, t_end, c0, c1, a.d, a.q, a.words, a.partials, a.scales, a.e, a.ef, a.seed, a.id,
                        a.t, gs);
    }
}

// One CTA per scale group (blockIdx.x) and message (blockIdx.y): combine the group's per-tile
// partial norms in a fixed order and write the group scale (Example 1: ||.||_inf; scaled sign:
// ||.||_1 / |group|).
template <int QK>
__global__ void __launch_bounds__(kThreads) finalize_kernel(const FinalizeArgs a)
{
    __shared__ double red[kWarps];
    pdl_trigger();
    pdl_wait();
    const int64_t gi = blockIdx.x;
    const double *partials = a.partials + static_cast<int64_t>(blockIdx.y) * a.partials_stride;
    float *scales = a.scales + static_cast<int64_t>(blockIdx.y) * a.scales_stride;
    const int64_t pb = a.q.grp.pair_base[gi], pe = a.q.grp.pair_base[gi + 1];
    double acc = 0.0;
    for (int64_t p = pb + threadIdx.x; p < pe; p += kThreads)
        acc = (QK == QK_SIGN) ? __dadd_rn(acc, partials[p]) : fmax(acc, partials[p]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const double w = __shfl_down_sync(0xffffffffu, acc, o);
        acc = (QK == QK_SIGN) ? __dadd_rn(acc, w) : fmax(acc, w);
    }
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = red[0];
        for (int w = 1; w < kWarps; ++w) t = (QK == QK_SIGN) ? __dadd_rn(t, red[w]) : fmax(t, red[w]);
        const int64_t len = group_end(a.q.grp, gi, a.d) - group_begin(a.q.grp, gi, a.d);
        scales[gi] = (QK == QK_SIGN) ? sign_scale(t, len) : static_cast<float>(t);
    }
}

// Second pass, one CTA per tile: encode the stashed input with its group's scale and leave the
// residual u - Q(u) in its place.
template <int QK>
__global__ void __launch_bounds__(kThreads, 2) encode_kernel(const EncodeArgs a)
{
    __shared__ float qtab_s[256];
    pdl_trigger();
    const float *qtab = build_qtab<QK>(a.q, qtab_s);
    __syncthreads();
    pdl_wait();
    const int64_t tile = blockIdx.x;
    const int64_t d = a.d;
    const Grouping &G = a.q.grp;
    const int L = (QK == QK_UNIF) ? unif_L(a.q.bits) : 0;
    const float Lf = static_cast<float>(L);
    const int64_t hint = first_group_of_tile(G, tile);
    float u[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) load4(a.buf, slot_of(tile, k), d, u[k]);
    // a tile inside one group (the common case) has one scale: the fused tile encode
    const int64_t g1 = tile_single_group(G, tile, d);
    if (g1 >= 0) {
        const float s = a.scales[g1];
        if ((tile + 1) * kTile <= d)
            encode_store<QK, true, true>(URegs{u}, s, tile, d, a.q, a.words, a.buf, a.ef, a.seed, a.id, a.t, qtab);
        else
            encode_store<QK, false, true>(URegs{u}, s, tile, d, a.q, a.words, a.buf, a.ef, a.seed, a.id, a.t, qtab);
        if (!a.ef) {  // without error feedback the residual is 0: clear the stash of u
            const float z[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int k = 0; k < kSlots; ++k)
                if (4 * slot_of(tile, k) < d) store4(a.buf, slot_of(tile, k), d, z);
        }
        return;
    }
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t qs = slot_of(tile, k);
        const int64_t j0 = 4 * qs;
        float U[4] = {0.f, 0.f, 0.f, 0.f};
        if (QK == QK_UNIF && a.q.stochastic && j0 < d) uniforms4(a.seed, a.id, a.t, j0, U);
        uint32_t c[4];
        float e[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float dec = 0.0f;
            c[i] = 0u;
            if (j0 + i < d) {
                const float s = a.scales[group_of(G, j0 + i, hint)];
                c[i] = encode1<QK>(u[k][i], s, a.q, Lf, L, U[i], dec, qtab);
            }
            e[i] = a.ef ? __fsub_rn(u[k][i], dec) : 0.0f;
        }
        store_codes4(a.words, qs, a.q.bits, c, 0, d);
        if (j0 < d) store4(a.buf, qs, d, e);
    }
}

// x <- x - dec(Q_s message) on one tile (Algorithm 1 and Algorithm 2); HBM traffic per coordinate:
// 4 B read + 4 B written + b/8 B of code.  BITS: the code width as a compile-time constant.  The
// loads of x and of the raw code words are issued first; the fl(i/L) table of the uniform grid
// (b <= 8) is built while they are in flight, and the codes are unpacked after its barrier.
// TILE_SCALE: the scales are 4096-blocks, one per tile (then no group lookup is compiled in; that
// instantiation measured 4% faster than one carrying the lookup as well).
template <int QK, bool FULL, int BITS, bool TILE_SCALE>
__device__ __forceinline__ void apply_tile(const ApplyArgs &a, int64_t tile, float *qtab_s)
{
    const int64_t d = a.d;
    const Grouping &G = a.q.grp;
    constexpr int bits = BITS;
    const int L = (QK == QK_UNIF) ? unif_L(bits) : 0;
    const float Lf = static_cast<float>(L);
    float x[kSlots][4];
    uint4 raw[kSlots];  // the slot's code bits: .x for b <= 8, .x .y for b = 16, all four for b = 32
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        load4<FULL>(a.x, q, d, x[k]);
        raw[k] = make_uint4(0u, 0u, 0u, 0u);
        if (FULL || 4 * q < d) {
            if constexpr (bits <= 8) {
                raw[k].x = __ldg(a.words + ((q * bits) >> 3));
            } else if constexpr (bits == 16) {
                const uint2 w = __ldg(reinterpret_cast<const uint2 *>(a.words) + q);
                raw[k].x = w.x, raw[k].y = w.y;
            } else {
                raw[k] = __ldg(reinterpret_cast<const uint4 *>(a.words) + q);
            }
        }
    }
    const float *qtab = nullptr;
    if constexpr (QK == QK_UNIF && bits <= 8) {
        qtab = build_qtab<QK>(a.q, qtab_s);
        __syncthreads();
    }
    // one scale for the whole tile: 4096-blocks, or a tile inside one group
    const int64_t g1 = !has_scale<QK>() ? 0 : TILE_SCALE ? tile : tile_single_group(G, tile, d);
    const bool tile_scale = TILE_SCALE || g1 >= 0;
    const float s_tile = (has_scale<QK>() && tile_scale) ? __ldg(a.scales + g1) : 0.0f;
    const int64_t hint = first_group_of_tile(G, tile);
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
        if (!FULL && j0 >= d) continue;
        uint32_t c[4];
        if constexpr (bits <= 8) {
            const int sh = static_cast<int>((q * bits) & 7) * 4;
#pragma unroll
            for (int i = 0; i < 4; ++i) c[i] = (raw[k].x >> (sh + i * bits)) & ((1u << bits) - 1u);
        } else if constexpr (bits == 16) {
            c[0] = raw[k].x & 0xffffu, c[1] = raw[k].x >> 16, c[2] = raw[k].y & 0xffffu, c[3] = raw[k].y >> 16;
        } else {
            c[0] = raw[k].x, c[1] = raw[k].y, c[2] = raw[k].z, c[3] = raw[k].w;
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if (FULL || j0 + i < d) {
                float s = s_tile;
                if (has_scale<QK>() && !tile_scale) s = __ldg(a.scales + group_of(G, j0 + i, hint));
                x[k][i] = __fsub_rn(x[k][i], decode1<QK>(c[i], s, a.q, Lf, L, qtab));
            }
        }
        store4<FULL>(a.x, q, d, x[k]);
    }
}

template <int QK, int BITS>
__device__ __forceinline__ void apply_body(const ApplyArgs &a, float *qtab_s)
{
    const int64_t tile = blockIdx.x;
    const bool full = (tile + 1) * kTile <= a.d;
    if (a.q.grp.gkind == GK_BLOCK && a.q.grp.G == kTile) {
        if (full) apply_tile<QK, true, BITS, true>(a, tile, qtab_s);
        else apply_tile<QK, false, BITS, true>(a, tile, qtab_s);
    } else {
        if (full) apply_tile<QK, true, BITS, false>(a, tile, qtab_s);
        else apply_tile<QK, false, BITS, false>(a, tile, qtab_s);
    }
}

// One CTA per 4096-tile; the code width is dispatched once per CTA.
template <int QK>
__global__ void __launch_bounds__(kThreads) apply_kernel(const ApplyArgs a)
{
    __shared__ float qtab_s[256];
    pdl_trigger();
    pdl_wait();
    if constexpr (QK == QK_UNIF) {
        switch (a.q.bits) {  // the widths ea_init accepts
        case 2: apply_body<QK, 2>(a, qtab_s); break;
        case 4: apply_body<QK, 4>(a, qtab_s); break;
        case 8: apply_body<QK, 8>(a, qtab_s); break;
        default: apply_body<QK, 16>(a, qtab_s); break;
        }
    } else if constexpr (QK == QK_POW2) {
        if (a.q.bits == 4) apply_body<QK, 4>(a, qtab_s);
        else apply_body<QK, 8>(a, qtab_s);
    } else {
        apply_body<QK, QK == QK_SIGN ? 1 : 32>(a, qtab_s);
    }
}

__global__ void fill_kernel(float *p, int64_t count, float value)
{
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x)
        p[i] = value;
}

// ------------------------------------------------------------------------------- launchers

template <int MODE>
static cudaError_t launch_worker_mode(const WorkerArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>(a.n_tiles)), block(kThreads);
    if (a.pass == PASS_LAZY)
        return a.q.kind == QK_SIGN ? launch_pdl(worker_lazy_kernel<MODE>, grid, block, 0, s, a) : cudaErrorNotSupported;
    switch (a.q.kind) {
    case QK_SIGN: return launch_pdl(worker_kernel<MODE, QK_SIGN>, grid, block, 0, s, a);
    case QK_UNIF: return launch_pdl(worker_kernel<MODE, QK_UNIF>, grid, block, 0, s, a);
    case QK_POW2: return launch_pdl(worker_kernel<MODE, QK_POW2>, grid, block, 0, s, a);
    default: return launch_pdl(worker_kernel<MODE, QK_IDENT>, grid, block, 0, s, a);
    }
}

cudaError_t launch_worker(int mode, const WorkerArgs &a, cudaStream_t s)
{
    return mode == MODE_W ? launch_worker_mode<MODE_W>(a, s) : launch_worker_mode<MODE_S>(a, s);
}

// The grouped kernel exists for the uniform grid (a scaled-sign message takes PASS_LAZY).
cudaError_t worker_grouped_shape(int mode, int qk, GroupedShape *out)
{
    const int w = mode == MODE_W ? 2 : 4;  // the kernels' launch bounds
    if (qk != QK_UNIF) return cudaErrorNotSupported;
    return mode == MODE_W ? grouped_shape(worker_grouped_kernel<MODE_W, QK_UNIF>, w, out)
                          : grouped_shape(worker_grouped_kernel<MODE_S, QK_UNIF>, w, out);
}

cudaError_t launch_worker_grouped(int mode, const WorkerArgs &a, int grid, cudaStream_t s)
{
    const int slots = a.gp.slots;
    if (a.q.kind != QK_UNIF) return cudaErrorNotSupported;
    return mode == MODE_W ? grouped_launch(worker_grouped_kernel<MODE_W, QK_UNIF>, a, grid, slots, s)
                          : grouped_launch(worker_grouped_kernel<MODE_S, QK_UNIF>, a, grid, slots, s);
}

cudaError_t launch_finalize(const FinalizeArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>(a.q.grp.n_groups), static_cast<unsigned>(a.n_msgs > 1 ? a.n_msgs : 1)),
        block(kThreads);
    if (a.q.kind == QK_SIGN) return launch_pdl(finalize_kernel<QK_SIGN>, grid, block, 0, s, a);
    return launch_pdl(finalize_kernel<QK_UNIF>, grid, block, 0, s, a);
}

cudaError_t launch_encode(const EncodeArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>(a.n_tiles)), block(kThreads);
    if (a.q.kind == QK_SIGN) return launch_pdl(encode_kernel<QK_SIGN>, grid, block, 0, s, a);
    return launch_pdl(encode_kernel<QK_UNIF>, grid, block, 0, s, a);
}

// The residual u - Q(u) of the u kept by PASS_LAZY, into a.out, one CTA per tile (a view of it).
__global__ void __launch_bounds__(kThreads) lazy_resid_kernel(const ResidArgs a)
{
    pdl_trigger();
    pdl_wait();
    const int64_t tile = blockIdx.x;
    const bool full = (tile + 1) * kTile <= a.d;
    float u[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) load4(a.u, slot_of(tile, k), a.d, u[k]);
    if (full) lazy_residual<true>(a.q, a.scales, tile, a.d, u);
    else lazy_residual<false>(a.q, a.scales, tile, a.d, u);
#pragma unroll
    for (int k = 0; k < kSlots; ++k)
        if (4 * slot_of(tile, k) < a.d) store4(a.out, slot_of(tile, k), a.d, u[k]);
}

cudaError_t launch_lazy_resid(const ResidArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>((a.d + kTile - 1) / kTile)), block(kThreads);
    if (a.q.kind != QK_SIGN) return cudaErrorNotSupported;
    return launch_pdl(lazy_resid_kernel, grid, block, 0, s, a);
}

cudaError_t launch_apply(const ApplyArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>((a.d + kTile - 1) / kTile)), block(kThreads);
    switch (a.q.kind) {
    case QK_SIGN: return launch_pdl(apply_kernel<QK_SIGN>, grid, block, 0, s, a);
    case QK_UNIF: return launch_pdl(apply_kernel<QK_UNIF>, grid, block, 0, s, a);
    case QK_POW2: return launch_pdl(apply_kernel<QK_POW2>, grid, block, 0, s, a);
    default: return launch_pdl(apply_kernel<QK_IDENT>, grid, block, 0, s, a);
    }
}

cudaError_t launch_fill(float *p, int64_t count, float value, cudaStream_t s)
{
    if (count <= 0) return cudaSuccess;
    const int64_t want = (count + 255) / 256;
    fill_kernel<<<static_cast<unsigned>(want < 152 * 64 ? want : 152 * 64), 256, 0, s>>>(p, count, value);
    return cudaGetLastError();
}

}  // namespace ea
