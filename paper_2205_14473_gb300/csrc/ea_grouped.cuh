// ea_grouped.cuh -- the one-pass scale of groups that span tiles (PASS_GROUPED; see GroupPlan):
// per-(group, tile) partial norms stored in global memory, a bounded grid-wide barrier per wave,
// every group's scale combined from its partials in one fixed order, and the encode of a tile's
// coordinate range [lo, hi) from the input parked in shared memory.
//
// A tile may hold several groups (their boundaries need not be tile-aligned), and a wave cut may
// fall inside a tile: the tile's coordinates before the cut belong to one wave and the rest to the
// next.  Cuts start a code word and a float4 slot, so two ranges never write the same word.
//
// Synchronisation is one counter per plan: each CTA adds one arrival per wave and waits until all
// gridDim.x CTAs of this wave (of this launch) have arrived; no per-group counters or flags, whose
// updates and polls would all land on a few L2 lines at the end of every wave.
#pragma once

#include <algorithm>

#include "ea_async.cuh"
#include "ea_tile.cuh"

namespace ea {

__device__ __forceinline__ unsigned long long ld_acquire_gpu_u64(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

constexpr int kRangeScales = kGroupedScales;  // scales of the groups a CTA encodes in one wave

// Per-CTA shared state of the grouped kernels.
struct GroupSmem {
    DF red[2][kWarps];            // per-warp partial sums, by parity of the reduction's turn
    uint32_t redm[2][kWarps];     // per-warp partial maxima, likewise
    float qtab[256];              // the message's uniform grid fl(i / L) (build_qtab)
    int abort;                    // the wave barrier ran out of time: the CTA stops
    float gsc[kRangeScales];      // scales of the groups of the CTA's ranges in this wave, in order
    TileGroups tg;                // segments of a tile that holds several
};

// For every group of Q that meets [lo, hi) (a range of tile `tile`), reduce this CTA's part of it
// -- |u| summed (compensated, to ~2^-44) for the scaled sign, max |u| for Example 1's grid -- over
// u in ub and store it as the group's partial for this tile.  One barrier per group: the warps'
// results go to red[turn & 1] and thread 0 combines them in warp order.  All threads call it.
template <int QK>
__device__ __forceinline__ void range_partials(const float4 *ub, int64_t tile, int64_t lo, int64_t hi, int64_t d,
                                               const QParams &q, double *partials, GroupSmem &gs, int &turn)
{
    const Grouping &G = q.grp;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int64_t gi = group_of(G, lo, first_group_of_tile(G, tile));; ++gi, ++turn) {
        const int64_t gb = group_begin(G, gi, d), ge = group_end(G, gi, d);
        const int64_t a = max(gb, lo), b = min(ge, hi);
        const int par = turn & 1;
        if constexpr (QK == QK_SIGN) {
            DF acc{0.0f, 0.0f};
#pragma unroll
            for (int k = 0; k < kSlots; ++k) {
                const int64_t j0 = 4 * slot_of(tile, k);
                const float4 v = ub[k * kThreads + threadIdx.x];
                const float u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (j0 + i >= a && j0 + i < b) df_accumulate(acc, fabsf(u[i]));
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                const DF w{__shfl_down_sync(0xffffffffu, acc.hi, o), __shfl_down_sync(0xffffffffu, acc.lo, o)};
                acc = df_add(acc, w);
            }
            if (lane == 0) gs.red[par][warp] = acc;
            compute_sync();
            if (threadIdx.x == 0) {
                DF t = gs.red[par][0];
#pragma unroll
                for (int w = 1; w < kWarps; ++w) t = df_add(t, gs.red[par][w]);
                partials[G.pair_base[gi] + (tile - gb / kTile)] = static_cast<double>(t.hi) + static_cast<double>(t.lo);
            }
        } else {
            float mx = 0.0f;
#pragma unroll
            for (int k = 0; k < kSlots; ++k) {
                const int64_t j0 = 4 * slot_of(tile, k);
                const float4 v = ub[k * kThreads + threadIdx.x];
                const float u[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    if (j0 + i >= a && j0 + i < b) mx = fmaxf(mx, fabsf(u[i]));
            }
            const uint32_t m = __reduce_max_sync(0xffffffffu, __float_as_uint(mx));  // exact on bit patterns
            if (lane == 0) gs.redm[par][warp] = m;
            compute_sync();
            if (threadIdx.x == 0) {
                uint32_t t = gs.redm[par][0];
#pragma unroll
                for (int w = 1; w < kWarps; ++w) t = max(t, gs.redm[par][w]);
                partials[G.pair_base[gi] + (tile - gb / kTile)] = static_cast<double>(__uint_as_float(t));
            }
        }
        if (ge >= hi) break;
    }
}

// The wave barrier: every CTA's partials of wave w are stored once all gridDim.x CTAs have arrived
// (arrivals count across waves and launches: this one completes at (epoch * n_waves + w + 1) *
// gridDim.x).  Thread 0 fences, arrives and polls with exponential backoff (256 ns doubling to
// 2 us); after ~2 s it records kStatusTimeout and every thread returns false.  All threads call it.
__device__ __forceinline__ bool wave_barrier(const GroupPlan &gp, int w, uint32_t *status, GroupSmem &gs)
{
    compute_sync();  // this CTA's partials are stored
    if (threadIdx.x == 0) {
        const unsigned long long target =
            (gp.epoch * static_cast<unsigned long long>(gp.n_waves) + static_cast<unsigned long long>(w) + 1ull) *
            gridDim.x;
        __threadfence();
        atomicAdd(gp.arrive, 1ull);
        bool ok = true;
        if (ld_acquire_gpu_u64(gp.arrive) < target) {
            const long long t0 = clock64();
            uint32_t ns = 256;
            while (ld_acquire_gpu_u64(gp.arrive) < target) {
                if (clock64() - t0 > kWaitLimitCycles) {
                    ok = false;
                    break;
                }
                __nanosleep(ns);
                ns = ns < 2048 ? 2 * ns : ns;
            }
        }
        if (!ok) report_status(status, kStatusTimeout);
        gs.abort = ok ? 0 : 1;
    }
    compute_sync();
    return gs.abort == 0;
}

// The groups of the range [lo, hi) of tile `tile`: the first one and how many.
__device__ __forceinline__ void range_groups(const Grouping &G, int64_t tile, int64_t lo, int64_t hi, int64_t &g0,
                                             int &ng)
{
    g0 = group_of(G, lo, first_group_of_tile(G, tile));
    ng = static_cast<int>(group_of(G, hi - 1, g0) - g0 + 1);
}

// Phase two for the CTA's tiles of one wave (tiles t0, t0 + gridDim.x, ... below t_end, u in
// uslot), after the wave barrier.  First the scale of every group of the CTA's ranges: one warp per
// group combines the group's partials in a fixed order -- lane strides, then a shuffle tree, in
// binary64 -- so every CTA that needs a group forms the same scale (||u||_1 / |group| rounded once,
// or the maximum); the CTA whose tile holds the group's first coordinate stores it in the message.
// Then each range is encoded -- one group takes the tile encode with its scale, several look each
// coordinate's group up -- storing the codes (words whose first coordinate lies in the range) and,
// with error feedback, the residual.  All threads call it.
template <int QK>
__device__ __forceinline__ void encode_wave(const float4 *uslot, int t0, int t_end, int64_t c0, int64_t c1, int64_t d,
                                            const QParams &q, uint32_t *words, const double *partials, float *scales,
                                            float *resid, int ef, uint64_t seed, uint32_t id, uint32_t t,
                                            GroupSmem &gs)
{
    const Grouping &G = q.grp;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    {
        int idx = 0;
        for (int tile = t0; tile < t_end; tile += gridDim.x) {
            const int64_t tl = static_cast<int64_t>(tile) * kTile, lo = max(c0, tl), hi = min(c1, tl + kTile);
            int64_t g0;
            int ng;
            range_groups(G, tile, lo, hi, g0, ng);
            for (int i = 0; i < ng; ++i, ++idx) {
                if ((idx & (kWarps - 1)) != warp) continue;
                const int64_t gi = g0 + i;
                const int64_t pb = G.pair_base[gi], pe = G.pair_base[gi + 1];
                double s = 0.0;
                for (int64_t p = pb + lane; p < pe; p += 32) {
                    const double v = __ldcg(partials + p);
                    s = (QK == QK_SIGN) ? __dadd_rn(s, v) : fmax(s, v);
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) {
                    const double w = __shfl_down_sync(0xffffffffu, s, o);
                    s = (QK == QK_SIGN) ? __dadd_rn(s, w) : fmax(s, w);
                }
                if (lane == 0) {
                    const int64_t gb = group_begin(G, gi, d);
                    const float sf = (QK == QK_SIGN) ? sign_scale(s, group_end(G, gi, d) - gb) : static_cast<float>(s);
                    if (idx < kRangeScales) gs.gsc[idx] = sf;
                    if (gb >= lo) scales[gi] = sf;  // the group's first coordinate is in this range
                }
            }
        }
    }
    compute_sync();  // the scales are in shared memory
    const float *qtab = (QK == QK_UNIF && q.bits <= 8) ? gs.qtab : nullptr;
    const int bits = code_bits<QK>(q);
    const int L = (QK == QK_UNIF) ? unif_L(bits) : 0;
    const float Lf = static_cast<float>(L);
    int k = 0, idx = 0;
    for (int tile = t0; tile < t_end; tile += gridDim.x, ++k) {
        const float4 *ub = uslot + k * (kThreads * kSlots);
        const int64_t tl = static_cast<int64_t>(tile) * kTile, lo = max(c0, tl), hi = min(c1, tl + kTile);
        int64_t g0;
        int ng;
        range_groups(G, tile, lo, hi, g0, ng);
        const int base = idx;
        idx += ng;
        if (ng == 1) {
            const float s = gs.gsc[base];
            if (lo == tl && hi == tl + kTile)
                encode_store<QK, true, true>(USmem{ub}, s, tile, hi, q, words, resid, ef, seed, id, t, qtab, lo);
            else
                encode_store<QK, false, true>(USmem{ub}, s, tile, hi, q, words, resid, ef, seed, id, t, qtab, lo);
            continue;
        }
        const bool seg = G.gkind == GK_SEG;  // several segments: look them up in shared memory
        if (seg) {
            compute_sync();  // the previous range's readers of tg are done
            cache_tile_groups(G, tile, d, gs.tg);
            compute_sync();
        }
#pragma unroll
        for (int kk = 0; kk < kSlots; ++kk) {
            const int64_t qs = slot_of(tile, kk);
            const int64_t j0 = 4 * qs;
            const bool in = j0 >= lo && j0 < hi;
            float U[4] = {0.f, 0.f, 0.f, 0.f};
            if (QK == QK_UNIF && q.stochastic && in) uniforms4(seed, id, t, j0, U);
            const float4 v = ub[kk * kThreads + threadIdx.x];
            const float u[4] = {v.x, v.y, v.z, v.w};
            uint32_t c[4];
            float e[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                float dec = 0.0f;
                c[i] = 0u;
                if (in && j0 + i < hi) {
                    const int64_t gi = seg ? tile_group_of(G, gs.tg, tile, j0 + i) : group_of(G, j0 + i, g0);
                    c[i] = encode1<QK>(u[i], gs.gsc[base + (gi - g0)], q, Lf, L, U[i], dec, qtab);
                }
                e[i] = ef ? __fsub_rn(u[i], dec) : 0.0f;
            }
            store_codes4<false, true>(words, qs, bits, c, lo, hi);
            if (ef && in) store4(resid, qs, hi, e);
        }
    }
    compute_sync();  // gsc and tg are rewritten in the next wave
}

// ---------------------------------------------------------------------------- host helpers

// Shape of a grouped kernel on the current device: as many tile slots of shared memory as fit
// beside its static shared memory when `reg_ctas` CTAs (the register budget of its launch bounds)
// share an SM, at most 8; then the resident CTAs per SM with that much dynamic shared memory.
// Sets the kernel's dynamic shared-memory limit on the current device.
template <class Kernel>
cudaError_t grouped_shape(Kernel kernel, int reg_ctas, GroupedShape *out)
{
    cudaFuncAttributes fa{};
    cudaError_t e = cudaFuncGetAttributes(&fa, kernel);
    if (e != cudaSuccess) return e;
    const size_t per_cta = kSmemPerSm / static_cast<size_t>(reg_ctas);
    const size_t fixed = kSmemReservedPerCta + fa.sharedSizeBytes;
    const int slots = per_cta > fixed ? static_cast<int>(std::min<size_t>(8, (per_cta - fixed) / (kTile * 4))) : 0;
    if (slots < 1) return cudaErrorInvalidConfiguration;
    const int bytes = slots * kTile * 4;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    int occ = 0;
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, kernel, kThreads, bytes);
    if (e != cudaSuccess) return e;
    out->ctas_per_sm = occ;
    out->slots = slots;
    return occ > 0 ? cudaSuccess : cudaErrorInvalidConfiguration;
}

// Cooperative launch (every CTA resident at once, which the grouped kernels' waits rely on) of a
// grouped kernel taking one argument struct; `slots` tiles of dynamic shared memory per CTA.
template <class Kernel, class Args>
cudaError_t grouped_launch(Kernel kernel, const Args &a, int grid, int slots, cudaStream_t s)
{
    void *args[] = {const_cast<Args *>(&a)};
    return cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(kernel), dim3(grid), dim3(kThreads), args,
                                       static_cast<size_t>(slots) * kTile * 4, s);
}

}  // namespace ea
