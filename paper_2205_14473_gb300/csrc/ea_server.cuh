// ea_server.cuh -- the server's round (Algorithm 1) on one 4096-coordinate tile.
#pragma once

#include "ea_tile.cuh"

namespace ea {

// Decode the n worker messages of this tile, average them (summed in worker order, one division
// by n), add the server residual (and, with Adam at the server, take the Adam step on the
// average first), then Q_s and e_s <- w - Q_s(w) (finish_tile).
// HBM traffic per coordinate: n b_w/8 B of worker codes + 4 B e_s read + 4 B e_s written + b_s/8 B
// of broadcast code (+ 16 B for m, v with Adam at the server).
template <int MODE, int QW, int QS>
__global__ void __launch_bounds__(kThreads, 2) server_kernel(const ServerArgs a)
{
    __shared__ TileSmem sm;
    __shared__ float utab[256];  // fl(i / L) for the workers' uniform grid, i = -L..L (b_w <= 8)
    const int64_t tile = blockIdx.x;
    const int64_t d = a.d;

    const int Lw = (QW == QK_UNIF) ? unif_L(a.qw.bits) : 0;
    const float Lwf = static_cast<float>(Lw);
    const bool use_tab = QW == QK_UNIF && a.qw.bits <= 8;
    if (use_tab) {
        for (int i = threadIdx.x; i <= 2 * Lw; i += kThreads)
            utab[i] = __fdiv_rn(static_cast<float>(i - Lw), Lwf);
        __syncthreads();
    }

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

    // The workers' scale of a coordinate: one per worker for the whole tile when Q_w uses
    // 4096-blocks, else a per-coordinate group lookup.
    const Grouping &GW = a.qw.grp;
    const bool wtile = GW.gkind == GK_BLOCK && GW.G == kTile;
    const int64_t whint = first_group_of_tile(GW, tile);

    float acc[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[k][i] = 0.0f;

#pragma unroll 2
    for (int w = 0; w < a.n; ++w) {
        const uint32_t *ww = a.wwords + static_cast<int64_t>(w) * a.wwords_stride;
        const float *wsc = a.wscales + static_cast<int64_t>(w) * a.wscales_stride;
        const float s_tile = (has_scale<QW>() && wtile) ? __ldg(wsc + tile) : 0.0f;
#pragma unroll
        for (int k = 0; k < kSlots; ++k) {
            const int64_t q = slot_of(tile, k);
            const int64_t j0 = 4 * q;
            if (j0 >= d) continue;
            uint32_t c[4];
            load_codes4(ww, q, a.qw.bits, c);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                if (j0 + i < d) {
                    float s = 0.0f;
                    if (has_scale<QW>()) s = wtile ? s_tile : __ldg(wsc + group_of(GW, j0 + i, whint));
                    acc[k][i] = __fadd_rn(acc[k][i], decode1<QW>(c[i], s, a.qw, Lwf, Lw, use_tab ? utab : nullptr));
                }
            }
        }
    }

    const float nf = static_cast<float>(a.n);
    float u[kSlots][4];
#pragma unroll
    for (int k = 0; k < kSlots; ++k) {
        const int64_t q = slot_of(tile, k);
        const int64_t j0 = 4 * q;
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            float step = __fdiv_rn(acc[k][i], nf);
            if (MODE == MODE_S) step = adam_step(step, ms[k][i], vs[k][i], a.hp);
            u[k][i] = (j0 + i < d) ? __fadd_rn(step, es[k][i]) : 0.0f;
        }
        if (MODE == MODE_S && j0 < d) {
            store4(a.ms, q, d, ms[k]);
            store4(a.vs, q, d, vs[k]);
        }
    }
    finish_tile<QS>(u, tile, d, a.qs, a.words, a.scales, a.es, a.ef, a.pass, a.seed,
                    static_cast<uint32_t>(a.n), a.t, a.partials, sm);
}

template <int MODE, int QW>
static cudaError_t launch_server_qw(const ServerArgs &a, cudaStream_t s)
{
    const dim3 grid(static_cast<unsigned>(a.n_tiles)), block(kThreads);
    switch (a.qs.kind) {
    case QK_SIGN: server_kernel<MODE, QW, QK_SIGN><<<grid, block, 0, s>>>(a); break;
    case QK_UNIF: server_kernel<MODE, QW, QK_UNIF><<<grid, block, 0, s>>>(a); break;
    case QK_POW2: server_kernel<MODE, QW, QK_POW2><<<grid, block, 0, s>>>(a); break;
    default: server_kernel<MODE, QW, QK_IDENT><<<grid, block, 0, s>>>(a); break;
    }
    return cudaGetLastError();
}

template <int MODE>
static cudaError_t launch_server_mode(const ServerArgs &a, cudaStream_t s)
{
    switch (a.qw.kind) {
    case QK_SIGN: return launch_server_qw<MODE, QK_SIGN>(a, s);
    case QK_UNIF: return launch_server_qw<MODE, QK_UNIF>(a, s);
    case QK_POW2: return launch_server_qw<MODE, QK_POW2>(a, s);
    default: return launch_server_qw<MODE, QK_IDENT>(a, s);
    }
}

}  // namespace ea
