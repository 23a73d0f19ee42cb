// ea_api.cu -- host side of the C ABI in include/ea.h: configuration checks, workspace layout,
// the round protocol of Algorithms 1-2, kernel launches and the bits ledger of Corollary 1.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <string>
#include <vector>

#include "ea.h"
#include "ea_internal.h"

using namespace ea;

namespace {

thread_local std::string g_last_error;  // failures that have no handle yet

constexpr size_t kAlign = 256;
constexpr uint32_t kStatusTimeoutBit = 1u;  // set by kernels whose bounded waits gave up

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct QHost {
    int kind = 0, bits = 0, stochastic = 0, k = 0, K = 0;
    int gkind = GK_WHOLE, log2G = -1, pass = PASS_FUSED;
    int64_t G = 0, n_groups = 1, n_words = 0, n_pairs = 0;
    bool has_scales = false;
    std::vector<int64_t> offsets;     // GK_SEG
    std::vector<int32_t> tile_group;  // GK_SEG
    std::vector<int64_t> pair_base;   // PASS_STASH, PASS_GROUPED
    std::vector<int64_t> cuts;        // PASS_GROUPED: the waves
    int grid = 0, slots = 0;          // PASS_GROUPED: persistent CTAs and tile slots per CTA
    // device copies (inside the workspace)
    int64_t *d_offsets = nullptr, *d_pair_base = nullptr, *d_cuts = nullptr;
    int32_t *d_tile_group = nullptr;
    unsigned long long *d_arrive = nullptr;  // PASS_GROUPED: the wave barrier's counter
};

// Sizes of every workspace buffer, in the order they are carved.
struct Layout {
    size_t e_w, m_w, v_w, e_s, m_s, v_s, codes_w, scales_w, codes_s, scales_s, partials;
    size_t off_w, tg_w, pb_w, off_s, tg_s, pb_s, status;
    size_t cuts_w, arr_w, cuts_s, arr_s;  // the grouped pass (groups that span tiles)
    size_t rview;                         // PASS_LAZY: where a residual view is formed
    int64_t dpad, wcode_stride, wscale_stride;
};

}  // namespace

struct ea_handle {
    ea_config cfg{};
    QHost qw, qs;
    Layout lay{};
    cudaStream_t stream = nullptr;
    int64_t n_tiles = 0;
    float *m = nullptr, *v = nullptr, *e = nullptr, *es = nullptr, *ms = nullptr, *vs = nullptr;
    uint32_t *wcodes = nullptr, *scodes = nullptr;
    float *wscales = nullptr, *sscales = nullptr;
    double *partials = nullptr;   // the worker messages' partial norms (one set each when lazy)
    double *spartials = nullptr;  // the broadcast's
    uint32_t *status = nullptr;
    float *rview = nullptr;  // PASS_LAZY: the residual views are formed here
    StagePlan splan{};
    Hyper hp{};
    int64_t t = 0;
    uint64_t epoch_w = 0, epoch_s = 0;  // grouped launches so far (worker messages, broadcasts)
    std::vector<unsigned char> compressed;
    std::vector<unsigned char> lazy_w;  // PASS_LAZY: worker i's e holds its last u (see lazy_residual)
    bool lazy_s = false;                // PASS_LAZY: e_s holds the last w
    bool lazy_staged = false;           // PASS_LAZY broadcast: every tile's worker messages fit the staging
    bool wscales_pending = false;       // PASS_LAZY workers: a message's scales are not formed yet
    int n_compressed = 0;
    bool has_message = false;
    uint64_t up_bits = 0, down_bits = 0;
    std::string err;
};

namespace {

int fail(ea_handle *h, int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    if (h) h->err = buf;
    else g_last_error = buf;
    return code;
}

int check_cuda(ea_handle *h, cudaError_t e, const char *what)
{
    if (e == cudaSuccess) return EA_OK;
    return fail(h, EA_E_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

int ilog2_exact(int64_t x)
{
    if (x <= 0 || (x & (x - 1))) return -1;
    int r = 0;
    while ((int64_t{1} << r) < x) ++r;
    return r;
}

// Validate one quantizer and derive its groups, tables and pass.
int setup_quant(const ea_quantizer &q, int64_t d, const char *name, QHost &out)
{
    out = QHost{};
    out.kind = q.kind;
    out.bits = q.bits;
    out.stochastic = q.stochastic;
    out.k = q.pow2_k;
    out.K = q.pow2_K;
    switch (q.kind) {
    case EA_Q_IDENTITY:
        if (q.bits != 32) return fail(nullptr, EA_E_INVAL, "%s: the identity quantizer has 32 bits", name);
        break;
    case EA_Q_SIGN_L1:
        if (q.bits != 1) return fail(nullptr, EA_E_INVAL, "%s: the scaled sign has 1 bit", name);
        break;
    case EA_Q_UNIFORM_MAX:
        if (q.bits != 2 && q.bits != 4 && q.bits != 8 && q.bits != 16)
            return fail(nullptr, EA_E_UNSUPPORTED, "%s: uniform grids of 2, 4, 8 or 16 bits only", name);
        break;
    case EA_Q_POW2:
        if (q.bits != 4 && q.bits != 8)
            return fail(nullptr, EA_E_UNSUPPORTED, "%s: power-of-two codes of 4 or 8 bits only", name);
        if (q.pow2_k < -126 || q.pow2_K > 127 || q.pow2_k >= q.pow2_K)
            return fail(nullptr, EA_E_INVAL, "%s: need -126 <= k < K <= 127", name);
        if (static_cast<int64_t>(q.pow2_K) - q.pow2_k + 2 > (int64_t{1} << (q.bits - 1)))
            return fail(nullptr, EA_E_INVAL, "%s: K - k + 1 levels and the zero code need more than %d bits",
                        name, q.bits);
        break;
    default:
        return fail(nullptr, EA_E_INVAL, "%s: unknown quantizer kind %d", name, q.kind);
    }
    if (q.stochastic != 0 && q.stochastic != 1) return fail(nullptr, EA_E_INVAL, "%s: stochastic is 0 or 1", name);
    if (q.stochastic && q.kind != EA_Q_UNIFORM_MAX)
        return fail(nullptr, EA_E_INVAL, "%s: stochastic rounding applies to the uniform grid only", name);
    out.has_scales = q.kind == EA_Q_SIGN_L1 || q.kind == EA_Q_UNIFORM_MAX;
    out.n_words = (d * q.bits + 31) / 32;

    const int64_t n_tiles = (d + kTile - 1) / kTile;
    if (!out.has_scales) {
        out.gkind = GK_WHOLE;
        out.n_groups = 0;
        out.pass = PASS_FUSED;
        return EA_OK;
    }
    if (q.group == 0) {
        out.gkind = GK_WHOLE;
        out.n_groups = 1;
    } else if (q.group > 0) {
        out.gkind = GK_BLOCK;
        out.G = q.group;
        out.log2G = ilog2_exact(q.group);
        out.n_groups = (d + q.group - 1) / q.group;
    } else {
        if (!q.seg_lengths || q.n_seg < 1) return fail(nullptr, EA_E_INVAL, "%s: segments need lengths", name);
        out.gkind = GK_SEG;
        out.n_groups = q.n_seg;
        out.offsets.resize(q.n_seg + 1);
        out.offsets[0] = 0;
        for (int i = 0; i < q.n_seg; ++i) {
            if (q.seg_lengths[i] <= 0) return fail(nullptr, EA_E_INVAL, "%s: segment %d is empty", name, i);
            out.offsets[i + 1] = out.offsets[i] + q.seg_lengths[i];
        }
        if (out.offsets.back() != d)
            return fail(nullptr, EA_E_INVAL, "%s: segment lengths sum to %lld, not d = %lld", name,
                        static_cast<long long>(out.offsets.back()), static_cast<long long>(d));
        out.tile_group.resize(n_tiles);
        int64_t gi = 0;
        for (int64_t t = 0; t < n_tiles; ++t) {
            while (out.offsets[gi + 1] <= t * kTile) ++gi;
            out.tile_group[t] = static_cast<int32_t>(gi);
        }
    }
    // One pass when every group is exactly one tile; otherwise partial norms per (tile, group).
    const bool block_tiles = out.gkind == GK_BLOCK && out.G == kTile;
    const bool single_tile = out.n_groups == 1 && d <= kTile;
    if (block_tiles || single_tile) {
        out.pass = PASS_FUSED;
    } else {
        out.pass = PASS_STASH;
        out.pair_base.resize(out.n_groups + 1);
        out.pair_base[0] = 0;
        for (int64_t gi = 0; gi < out.n_groups; ++gi) {
            int64_t b, e;
            if (out.gkind == GK_WHOLE) { b = 0; e = d; }
            else if (out.gkind == GK_BLOCK) { b = gi * out.G; e = std::min(d, (gi + 1) * out.G); }
            else { b = out.offsets[gi]; e = out.offsets[gi + 1]; }
            out.pair_base[gi + 1] = out.pair_base[gi] + ((e - 1) / kTile - b / kTile + 1);
        }
        out.n_pairs = out.pair_base.back();
    }
    return EA_OK;
}

int validate(const ea_config *cfg, QHost &qw, QHost &qs)
{
    if (!cfg) return fail(nullptr, EA_E_INVAL, "config is NULL");
    if (cfg->d < 1) return fail(nullptr, EA_E_INVAL, "d must be >= 1");
    if (cfg->d > (int64_t{1} << 40)) return fail(nullptr, EA_E_UNSUPPORTED, "d above 2^40");
    if (cfg->n < 1 || cfg->n > 1024) return fail(nullptr, EA_E_INVAL, "n must be in [1, 1024]");
    if (cfg->placement != EA_ADAM_AT_WORKER && cfg->placement != EA_ADAM_AT_SERVER)
        return fail(nullptr, EA_E_INVAL, "unknown placement %d", cfg->placement);
    if (cfg->error_feedback != 0 && cfg->error_feedback != 1)
        return fail(nullptr, EA_E_INVAL, "error_feedback is 0 or 1");
    if (cfg->adam_form != 0 && cfg->adam_form != 1) return fail(nullptr, EA_E_INVAL, "adam_form is 0 or 1");
    if (!std::isfinite(cfg->alpha)) return fail(nullptr, EA_E_INVAL, "alpha must be finite");
    if (!(cfg->beta1 >= 0.0f && cfg->beta1 < 1.0f)) return fail(nullptr, EA_E_INVAL, "beta1 must be in [0, 1)");
    if (!(cfg->beta2 >= 0.0f && cfg->beta2 < 1.0f)) return fail(nullptr, EA_E_INVAL, "beta2 must be in [0, 1)");
    if (!(cfg->eps > 0.0f) || !std::isfinite(cfg->eps)) return fail(nullptr, EA_E_INVAL, "eps (= v_0) must be > 0");
    int r = setup_quant(cfg->qw, cfg->d, "Q_w", qw);
    if (r != EA_OK) return r;
    return setup_quant(cfg->qs, cfg->d, "Q_s", qs);
}

Layout make_layout(const ea_config &c, const QHost &qw, const QHost &qs)
{
    Layout L{};
    const bool W = c.placement == EA_ADAM_AT_WORKER;
    const int64_t n_tiles = (c.d + kTile - 1) / kTile;
    L.dpad = static_cast<int64_t>(align_up(static_cast<size_t>(c.d), 64));
    const size_t vec = static_cast<size_t>(L.dpad) * sizeof(float);
    L.e_w = vec * c.n;
    L.m_w = W ? vec * c.n : 0;
    L.v_w = W ? vec * c.n : 0;
    L.e_s = vec;
    L.m_s = W ? 0 : vec;
    L.v_s = W ? 0 : vec;
    // code buffers padded to 256 bytes so that 8- and 16-byte code stores of the last slot stay inside
    L.wcode_stride = static_cast<int64_t>(align_up(static_cast<size_t>(qw.n_words), 64));
    L.wscale_stride = static_cast<int64_t>(align_up(static_cast<size_t>(std::max<int64_t>(qw.n_groups, 1)), 64));
    L.codes_w = static_cast<size_t>(L.wcode_stride) * 4 * c.n;
    L.scales_w = static_cast<size_t>(L.wscale_stride) * 4 * c.n;
    L.codes_s = align_up(static_cast<size_t>(qs.n_words) * 4, kAlign);
    L.scales_s = align_up(static_cast<size_t>(std::max<int64_t>(qs.n_groups, 1)) * 4, kAlign);
    // partial norms: shared by the messages one after another, except that lazy scaled-sign worker
    // messages keep one set each (their scales are formed together before the server step) and the
    // broadcast then has its own
    const bool lazy_w = qw.pass == PASS_STASH && qw.kind == EA_Q_SIGN_L1;
    L.partials = (lazy_w ? static_cast<size_t>(c.n) * qw.n_pairs + qs.n_pairs
                         : static_cast<size_t>(std::max(qw.n_pairs, qs.n_pairs))) * sizeof(double);
    L.off_w = qw.gkind == GK_SEG ? qw.offsets.size() * 8 : 0;
    L.tg_w = qw.gkind == GK_SEG ? static_cast<size_t>(n_tiles) * 4 : 0;
    L.pb_w = qw.pass == PASS_STASH ? qw.pair_base.size() * 8 : 0;
    L.off_s = qs.gkind == GK_SEG ? qs.offsets.size() * 8 : 0;
    L.tg_s = qs.gkind == GK_SEG ? static_cast<size_t>(n_tiles) * 4 : 0;
    L.pb_s = qs.pass == PASS_STASH ? qs.pair_base.size() * 8 : 0;
    L.status = 4;
    // the grouped pass, whenever groups span tiles (ea_init picks it when its waves fit)
    const bool gw = qw.pass == PASS_STASH, gs = qs.pass == PASS_STASH;
    L.cuts_w = gw ? static_cast<size_t>(qw.n_groups + 1) * 8 : 0;
    L.arr_w = gw ? 8 : 0;
    L.cuts_s = gs ? static_cast<size_t>(qs.n_groups + 1) * 8 : 0;
    L.arr_s = gs ? 8 : 0;
    L.rview = ((gw && qw.kind == EA_Q_SIGN_L1) || (gs && qs.kind == EA_Q_SIGN_L1)) ? vec : 0;
    return L;
}

size_t layout_bytes(const Layout &L)
{
    const size_t parts[] = {L.e_w, L.m_w, L.v_w, L.e_s, L.m_s, L.v_s, L.codes_w, L.scales_w, L.codes_s,
                            L.scales_s, L.partials, L.off_w, L.tg_w, L.pb_w, L.off_s, L.tg_s, L.pb_s, L.status,
                            L.cuts_w, L.arr_w, L.cuts_s, L.arr_s, L.rview};
    size_t total = 0;
    for (size_t p : parts) total += align_up(p, kAlign);
    return total;
}

Grouping device_grouping(const QHost &q)
{
    Grouping g{};
    g.gkind = q.gkind;
    g.log2G = q.log2G;
    g.G = q.G;
    g.n_groups = q.n_groups;
    g.offsets = q.d_offsets;
    g.tile_group = q.d_tile_group;
    g.pair_base = q.d_pair_base;
    return g;
}

// The waves of PASS_GROUPED for q's groups: cuts at group boundaries that start a code word and a
// float4 slot (multiples of max(4, 32 / b)), each wave touching at most `cap` tiles, greedily as
// long as possible.  False when some run of groups between two usable cuts needs more tiles.
bool plan_waves(const QHost &q, int64_t d, int64_t cap, std::vector<int64_t> &cuts)
{
    const int64_t align = std::max<int64_t>(4, 32 / q.bits);
    std::vector<int64_t> cand;
    if (q.gkind == GK_BLOCK) {
        for (int64_t b = q.G; b < d; b += q.G)
            if (b % align == 0) cand.push_back(b);
    } else if (q.gkind == GK_SEG) {
        for (size_t i = 1; i + 1 < q.offsets.size(); ++i)
            if (q.offsets[i] % align == 0) cand.push_back(q.offsets[i]);
    }
    cand.push_back(d);
    auto tiles = [](int64_t a, int64_t b) { return (b - 1) / kTile - a / kTile + 1; };
    cuts.assign(1, 0);
    size_t i = 0;
    for (int64_t c = 0; c < d;) {
        int64_t best = -1;
        while (i < cand.size() && tiles(c, cand[i]) <= cap) best = cand[i++];
        if (best < 0) return false;
        cuts.push_back(best);
        c = best;
    }
    return true;
}

// Groups met by one CTA's tile ranges in wave [c0, c1) (tiles t0 + b, t0 + b + grid, ...).
int64_t cta_groups(const QHost &q, int64_t d, int64_t c0, int64_t c1, int64_t b, int64_t grid)
{
    auto group_at = [&](int64_t j) -> int64_t {
        if (q.gkind == GK_WHOLE) return 0;
        if (q.gkind == GK_BLOCK) return j / q.G;
        return std::upper_bound(q.offsets.begin(), q.offsets.end(), j) - q.offsets.begin() - 1;
    };
    int64_t total = 0;
    for (int64_t tile = c0 / kTile + b; tile * kTile < c1; tile += grid) {
        const int64_t lo = std::max(c0, tile * kTile), hi = std::min({c1, tile * kTile + kTile, d});
        total += group_at(hi - 1) - group_at(lo) + 1;
    }
    return total;
}

// Switch q from the two-pass scale to the grouped pass if its waves fit this device: `shape` is the
// grouped kernel's, `sms` the SM count.  max_tiles_per_cta > 0 bounds the tiles each CTA takes
// (measured on GB300: the grouped worker, whose CTAs run their tiles one after another, is faster
// than the two passes only while every CTA holds one tile; the grouped server is faster with
// several).
void try_grouped(QHost &q, int64_t d, int64_t n_tiles, const GroupedShape &shape, int sms, int max_tiles_per_cta)
{
    if (q.pass != PASS_STASH || shape.ctas_per_sm < 1 || shape.slots < 1 || sms < 1) return;
    const int64_t grid = std::min<int64_t>(static_cast<int64_t>(shape.ctas_per_sm) * sms, n_tiles);
    const int slots = max_tiles_per_cta > 0 ? std::min(shape.slots, max_tiles_per_cta) : shape.slots;
    std::vector<int64_t> cuts;
    if (!plan_waves(q, d, grid * slots, cuts)) return;
    if (max_tiles_per_cta > 0 && cuts.size() > 2) return;  // one wave only
    // every CTA's groups of a wave must fit its scale table
    for (size_t w = 0; w + 1 < cuts.size(); ++w)
        for (int64_t b = 0; b < grid; ++b)
            if (cta_groups(q, d, cuts[w], cuts[w + 1], b, grid) > kGroupedScales) return;
    q.cuts = std::move(cuts);
    q.grid = static_cast<int>(grid);
    q.slots = slots;
    q.pass = PASS_GROUPED;
}

// The most of q's scale groups that meet one 4096-tile.
int64_t max_groups_per_tile(const QHost &q, int64_t d, int64_t n_tiles)
{
    if (!q.has_scales || q.gkind == GK_WHOLE) return 1;
    if (q.gkind == GK_BLOCK) return (kTile - 1) / q.G + 2;  // a bound
    int64_t most = 1;
    for (int64_t t = 0; t < n_tiles; ++t) {
        const int64_t last = std::min((t + 1) * kTile, d) - 1;
        const int64_t g0 = q.tile_group[static_cast<size_t>(t)];
        int64_t g = g0;
        while (q.offsets[static_cast<size_t>(g + 1)] <= last) ++g;
        most = std::max(most, g - g0 + 1);
    }
    return most;
}

GroupPlan device_group_plan(const QHost &q, uint64_t epoch)
{
    GroupPlan g{};
    g.n_waves = static_cast<int64_t>(q.cuts.size()) - 1;
    g.cuts = q.d_cuts;
    g.arrive = q.d_arrive;
    g.epoch = epoch;
    g.slots = q.slots;
    return g;
}

QParams device_quant(const QHost &q)
{
    QParams p{};
    p.kind = q.kind;  // the EA_Q_* and QK_* enumerators coincide
    p.bits = q.bits;
    p.stochastic = q.stochastic;
    p.pow2_k = q.k;
    p.pow2_K = q.K;
    p.grp = device_grouping(q);
    return p;
}

uint64_t message_bits(const QHost &q, int64_t d)
{
    return static_cast<uint64_t>(d) * static_cast<uint64_t>(q.bits) +
           (q.has_scales ? 32ull * static_cast<uint64_t>(q.n_groups) : 0ull);
}

// Shared-memory staging of the server's inputs (see server_staged_kernel): one stage holds a
// tile's e_s (+ m_s, v_s) and the n workers' code chunks and scales.  Enabled when both messages
// have one scale per 4096-tile (or none) and two stages fit in 200 KB.
StagePlan make_server_plan(const ea_config &c, const QHost &qw, const QHost &qs, int64_t n_tiles, int sms)
{
    StagePlan P{};
    const bool qs_ok = !qs.has_scales || qs.pass == PASS_FUSED;
    const bool qw_ok = !qw.has_scales || qw.pass == PASS_FUSED;
    if (!qs_ok || !qw_ok || sms <= 0) return P;
    const bool server_adam = c.placement == EA_ADAM_AT_SERVER;
    uint32_t off = 0;
    P.off_a = off;
    off += 4 * kTile;
    if (server_adam) {
        P.off_b = off;
        off += 4 * kTile;
        P.off_c = off;
        off += 4 * kTile;
    }
    P.code_chunk = static_cast<uint32_t>(kTile / 8 * qw.bits);
    P.off_codes = off;
    const uint64_t codes = static_cast<uint64_t>(P.code_chunk) * c.n;
    if (codes > 100 * 1024) return P;
    off += static_cast<uint32_t>(codes);
    P.off_scales = off;
    off += static_cast<uint32_t>(align_up(4 * static_cast<size_t>(c.n), 16));
    P.stage_bytes = static_cast<uint32_t>(align_up(off, 128));
    // As many resident CTAs per SM as shared memory holds with one stage each (the kernel's
    // registers allow server_ctas_per_sm; the EA_Q_* kinds are the kernels' QK_* values), then as
    // many stages per CTA as fit, up to six.  The full/empty barriers of up to eight stages take
    // the first 128 bytes.
    const int max_ctas = server_ctas_per_sm(server_adam ? MODE_S : MODE_W, qw.kind, qs.kind);
    int per_sm = 0;
    for (int ctas = max_ctas; ctas >= 1 && per_sm == 0; --ctas) {
        const uint32_t room = std::min(kSmemPerSm / ctas - kServerStaticSmem - kSmemReservedPerCta, kServerMaxDynSmem);
        if (room < 128 + P.stage_bytes) continue;
        per_sm = ctas;
        P.stages = std::min(6, static_cast<int>((room - 128) / P.stage_bytes));
    }
    if (per_sm == 0) return P;
    P.smem_bytes = 128 + static_cast<uint32_t>(P.stages) * P.stage_bytes;
    P.grid = static_cast<int>(std::min<int64_t>(n_tiles, static_cast<int64_t>(sms) * per_sm));
    P.enabled = 1;
    return P;
}

// The hyper-parameters of the current round (1-based t = h->t + 1 for the bias corrections).
Hyper round_hyper(const ea_handle *h)
{
    Hyper hp = h->hp;
    if (hp.form == 1) {
        hp.bc1 = bias_correction(hp.beta1, h->t + 1);
        hp.bc2 = bias_correction(hp.beta2, h->t + 1);
    }
    return hp;
}

int check_hparams(float alpha, float beta1, float beta2)
{
    if (!std::isfinite(alpha)) return fail(nullptr, EA_E_INVAL, "alpha must be finite");
    if (!(beta1 >= 0.0f && beta1 < 1.0f)) return fail(nullptr, EA_E_INVAL, "beta1 must be in [0, 1)");
    if (!(beta2 >= 0.0f && beta2 < 1.0f)) return fail(nullptr, EA_E_INVAL, "beta2 must be in [0, 1)");
    return EA_OK;
}

int check_dev_ptr(ea_handle *h, const void *p, const char *what)
{
    if (!p) return fail(h, EA_E_INVAL, "%s is NULL", what);
    if (reinterpret_cast<uintptr_t>(p) % 16) return fail(h, EA_E_ALIGN, "%s is not 16-byte aligned", what);
    return EA_OK;
}

// Finish a message whose scale groups span tiles: scales from the partial norms, then encode.
// The group scales from the per-(tile, group) partial norms (PASS_STASH, PASS_LAZY).
int finalize_scales(ea_handle *h, const QHost &q, const double *partials, float *scales)
{
    FinalizeArgs f{};
    f.d = h->cfg.d;
    f.q = device_quant(q);
    f.partials = partials;
    f.scales = scales;
    return check_cuda(h, launch_finalize(f, h->stream), "finalize launch");
}

// PASS_LAZY worker messages: the scales of all n messages in one launch, from each worker's own
// partial norms (a message compressed in an earlier round gets the same scales again).
int finalize_worker_scales(ea_handle *h)
{
    if (!h->wscales_pending) return EA_OK;
    FinalizeArgs f{};
    f.d = h->cfg.d;
    f.q = device_quant(h->qw);
    f.partials = h->partials;
    f.scales = h->wscales;
    f.n_msgs = h->cfg.n;
    f.partials_stride = h->qw.n_pairs;
    f.scales_stride = h->lay.wscale_stride;
    const int r = check_cuda(h, launch_finalize(f, h->stream), "finalize launch");
    if (r == EA_OK) h->wscales_pending = false;
    return r;
}

int second_pass(ea_handle *h, const QHost &q, const double *partials, float *buf, uint32_t *words, float *scales,
                uint32_t id)
{
    int r = finalize_scales(h, q, partials, scales);
    if (r != EA_OK) return r;
    EncodeArgs e{};
    e.d = h->cfg.d;
    e.n_tiles = h->n_tiles;
    e.buf = buf;
    e.q = device_quant(q);
    e.words = words;
    e.scales = scales;
    e.ef = h->cfg.error_feedback;
    e.seed = h->cfg.seed;
    e.id = id;
    e.t = static_cast<uint32_t>(h->t);
    return check_cuda(h, launch_encode(e, h->stream), "encode launch");
}

}  // namespace

void ea::set_last_error(const char *msg) { g_last_error = msg; }

cudaError_t ea::launch_server(int mode, const ServerArgs &a, cudaStream_t s)
{
    if (mode == MODE_W) {
        switch (a.qs.kind) {
        case QK_SIGN: return launch_server_for_qs<MODE_W, QK_SIGN>(a, s);
        case QK_UNIF: return launch_server_for_qs<MODE_W, QK_UNIF>(a, s);
        case QK_POW2: return launch_server_for_qs<MODE_W, QK_POW2>(a, s);
        default: return launch_server_for_qs<MODE_W, QK_IDENT>(a, s);
        }
    }
    switch (a.qs.kind) {
    case QK_SIGN: return launch_server_for_qs<MODE_S, QK_SIGN>(a, s);
    case QK_UNIF: return launch_server_for_qs<MODE_S, QK_UNIF>(a, s);
    case QK_POW2: return launch_server_for_qs<MODE_S, QK_POW2>(a, s);
    default: return launch_server_for_qs<MODE_S, QK_IDENT>(a, s);
    }
}

// The grouped server exists for a uniform-grid broadcast (a scaled-sign one takes PASS_LAZY).
cudaError_t ea::launch_server_grouped(int mode, const ServerArgs &a, int grid, cudaStream_t s)
{
    if (a.qs.kind != QK_UNIF) return cudaErrorNotSupported;
    return mode == MODE_W ? launch_server_grouped_for_qs<MODE_W, QK_UNIF>(a, grid, s)
                          : launch_server_grouped_for_qs<MODE_S, QK_UNIF>(a, grid, s);
}

cudaError_t ea::server_grouped_shape(int mode, int qw, int qs, GroupedShape *out)
{
    if (qs != QK_UNIF) return cudaErrorNotSupported;
    return mode == MODE_W ? server_grouped_shape_for_qs<MODE_W, QK_UNIF>(qw, out)
                          : server_grouped_shape_for_qs<MODE_S, QK_UNIF>(qw, out);
}

extern "C" {

int ea_workspace_bytes(const ea_config *cfg, size_t *bytes)
{
    QHost qw, qs;
    if (!bytes) return fail(nullptr, EA_E_INVAL, "bytes is NULL");
    const int r = validate(cfg, qw, qs);
    if (r != EA_OK) return r;
    *bytes = layout_bytes(make_layout(*cfg, qw, qs));
    return EA_OK;
}

int ea_init(const ea_config *cfg, void *workspace, size_t workspace_bytes, void *stream, ea_handle **out)
{
    if (!out) return fail(nullptr, EA_E_INVAL, "out is NULL");
    *out = nullptr;
    QHost qw, qs;
    int r = validate(cfg, qw, qs);
    if (r != EA_OK) return r;
    const Layout L = make_layout(*cfg, qw, qs);
    const size_t need = layout_bytes(L);
    if (!workspace) return fail(nullptr, EA_E_WORKSPACE, "workspace is NULL");
    if (reinterpret_cast<uintptr_t>(workspace) % kAlign)
        return fail(nullptr, EA_E_WORKSPACE, "workspace is not 256-byte aligned");
    if (workspace_bytes < need)
        return fail(nullptr, EA_E_WORKSPACE, "workspace has %zu bytes, needs %zu", workspace_bytes, need);

    ea_handle *h = new (std::nothrow) ea_handle;
    if (!h) return fail(nullptr, EA_E_INVAL, "out of host memory");
    h->cfg = *cfg;
    h->cfg.qw.seg_lengths = nullptr;
    h->cfg.qs.seg_lengths = nullptr;
    h->qw = std::move(qw);
    h->qs = std::move(qs);
    h->lay = L;
    h->stream = static_cast<cudaStream_t>(stream);
    h->n_tiles = (cfg->d + kTile - 1) / kTile;
    h->compressed.assign(cfg->n, 0);
    h->lazy_w.assign(cfg->n, 0);
    h->hp.alpha = cfg->alpha;
    h->hp.beta1 = cfg->beta1;
    h->hp.beta2 = cfg->beta2;
    h->hp.c1 = 1.0f - cfg->beta1;
    h->hp.c2 = 1.0f - cfg->beta2;
    h->hp.form = cfg->adam_form;
    h->hp.eps = cfg->eps;

    char *p = static_cast<char *>(workspace);
    auto take = [&p](size_t n) {
        char *q = n ? p : nullptr;
        p += align_up(n, kAlign);
        return q;
    };
    h->e = reinterpret_cast<float *>(take(L.e_w));
    h->m = reinterpret_cast<float *>(take(L.m_w));
    h->v = reinterpret_cast<float *>(take(L.v_w));
    h->es = reinterpret_cast<float *>(take(L.e_s));
    h->ms = reinterpret_cast<float *>(take(L.m_s));
    h->vs = reinterpret_cast<float *>(take(L.v_s));
    h->wcodes = reinterpret_cast<uint32_t *>(take(L.codes_w));
    h->wscales = reinterpret_cast<float *>(take(L.scales_w));
    h->scodes = reinterpret_cast<uint32_t *>(take(L.codes_s));
    h->sscales = reinterpret_cast<float *>(take(L.scales_s));
    h->partials = reinterpret_cast<double *>(take(L.partials));
    h->spartials = h->partials;
    h->qw.d_offsets = reinterpret_cast<int64_t *>(take(L.off_w));
    h->qw.d_tile_group = reinterpret_cast<int32_t *>(take(L.tg_w));
    h->qw.d_pair_base = reinterpret_cast<int64_t *>(take(L.pb_w));
    h->qs.d_offsets = reinterpret_cast<int64_t *>(take(L.off_s));
    h->qs.d_tile_group = reinterpret_cast<int32_t *>(take(L.tg_s));
    h->qs.d_pair_base = reinterpret_cast<int64_t *>(take(L.pb_s));
    h->status = reinterpret_cast<uint32_t *>(take(L.status));
    h->qw.d_cuts = reinterpret_cast<int64_t *>(take(L.cuts_w));
    h->qw.d_arrive = reinterpret_cast<unsigned long long *>(take(L.arr_w));
    h->qs.d_cuts = reinterpret_cast<int64_t *>(take(L.cuts_s));
    h->qs.d_arrive = reinterpret_cast<unsigned long long *>(take(L.arr_s));
    h->rview = reinterpret_cast<float *>(take(L.rview));
    // scaled-sign messages whose groups span tiles: the sign codes need no scale, so one pass writes
    // them and keeps u (PASS_LAZY); its workspace is that of the two passes
    if (h->qw.pass == PASS_STASH && h->qw.kind == EA_Q_SIGN_L1) {
        h->qw.pass = PASS_LAZY;
        h->spartials = h->partials + static_cast<int64_t>(cfg->n) * h->qw.n_pairs;
    }
    if (h->qs.pass == PASS_STASH && h->qs.kind == EA_Q_SIGN_L1) {
        h->qs.pass = PASS_LAZY;
        // the server stages a tile's worker codes and scales in shared memory when they fit
        const int64_t g = max_groups_per_tile(h->qw, cfg->d, h->n_tiles);
        h->lazy_staged = static_cast<int64_t>(cfg->n) * h->qw.bits <= 32 &&
                         g <= kStagedTileGroups && cfg->n * g <= kWorkerScales;
    }
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) == cudaSuccess &&
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess) {
        h->splan = make_server_plan(*cfg, h->qw, h->qs, h->n_tiles, sms);
        // groups that span tiles: the one-pass grouped kernels when their waves fit, else two passes
        const int mode = cfg->placement == EA_ADAM_AT_WORKER ? MODE_W : MODE_S;
        int coop = 0;
        cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
        GroupedShape shw{}, shs{};
        if (coop && h->qw.pass == PASS_STASH && worker_grouped_shape(mode, h->qw.kind, &shw) == cudaSuccess)
            try_grouped(h->qw, cfg->d, h->n_tiles, shw, sms, 1);
        if (coop && h->qs.pass == PASS_STASH && server_grouped_shape(mode, h->qw.kind, h->qs.kind, &shs) == cudaSuccess)
            try_grouped(h->qs, cfg->d, h->n_tiles, shs, sms, 0);
        cudaGetLastError();  // a shape query that failed leaves the two-pass scale in place
    }

    // Algorithm 2: m_0 = 0, v_0 = eps (0 in the textbook form), e_1 = 0; Algorithm 1: e_1 = 0.
    // Messages start zeroed.
    cudaStream_t s = h->stream;
    const float v0 = cfg->adam_form == 0 ? cfg->eps : 0.0f;
    r = check_cuda(h, cudaMemsetAsync(workspace, 0, need, s), "workspace clear");
    if (r == EA_OK && cfg->placement == EA_ADAM_AT_WORKER)
        r = check_cuda(h, launch_fill(h->v, static_cast<int64_t>(cfg->n) * L.dpad, v0, s), "v_0 fill");
    if (r == EA_OK && cfg->placement == EA_ADAM_AT_SERVER)
        r = check_cuda(h, launch_fill(h->vs, L.dpad, v0, s), "v_0 fill");
    auto upload = [&](void *dst, const void *src, size_t n) {
        if (r == EA_OK && n) r = check_cuda(h, cudaMemcpyAsync(dst, src, n, cudaMemcpyHostToDevice, s), "table upload");
    };
    upload(h->qw.d_offsets, h->qw.offsets.data(), L.off_w);
    upload(h->qw.d_tile_group, h->qw.tile_group.data(), L.tg_w);
    upload(h->qw.d_pair_base, h->qw.pair_base.data(), L.pb_w);
    upload(h->qs.d_offsets, h->qs.offsets.data(), L.off_s);
    upload(h->qs.d_tile_group, h->qs.tile_group.data(), L.tg_s);
    upload(h->qs.d_pair_base, h->qs.pair_base.data(), L.pb_s);
    upload(h->qw.d_cuts, h->qw.cuts.data(), h->qw.cuts.size() * 8);
    upload(h->qs.d_cuts, h->qs.cuts.data(), h->qs.cuts.size() * 8);
    if (r != EA_OK) {
        g_last_error = h->err;
        delete h;
        return r;
    }
    *out = h;
    return EA_OK;
}

int ea_worker_compress(ea_handle *h, int32_t worker, const float *g)
{
    if (!h) return fail(nullptr, EA_E_INVAL, "handle is NULL");
    if (worker < 0 || worker >= h->cfg.n) return fail(h, EA_E_INVAL, "worker %d out of [0, %d)", worker, h->cfg.n);
    int r = check_dev_ptr(h, g, "g");
    if (r != EA_OK) return r;
    if (h->compressed[worker])
        return fail(h, EA_E_ORDER, "worker %d already compressed in round %lld", worker, static_cast<long long>(h->t));
    const int64_t dp = h->lay.dpad;
    WorkerArgs a{};
    a.d = h->cfg.d;
    a.n_tiles = h->n_tiles;
    a.g = g;
    const bool W = h->cfg.placement == EA_ADAM_AT_WORKER;
    a.m = W ? h->m + worker * dp : nullptr;
    a.v = W ? h->v + worker * dp : nullptr;
    a.e = h->e + worker * dp;
    a.q = device_quant(h->qw);
    a.words = h->wcodes + worker * h->lay.wcode_stride;
    a.scales = h->wscales + worker * h->lay.wscale_stride;
    a.hp = round_hyper(h);
    a.ef = h->cfg.error_feedback;
    a.pass = h->qw.pass;
    a.seed = h->cfg.seed;
    a.id = static_cast<uint32_t>(worker);
    a.t = static_cast<uint32_t>(h->t);
    a.partials = h->qw.pass == PASS_LAZY ? h->partials + static_cast<int64_t>(worker) * h->qw.n_pairs : h->partials;
    a.status = h->status;
    a.lazy_in = h->qw.pass == PASS_LAZY ? h->lazy_w[worker] : 0;
    if (h->qw.pass == PASS_GROUPED) {
        a.gp = device_group_plan(h->qw, h->epoch_w);
        r = check_cuda(h, launch_worker_grouped(W ? MODE_W : MODE_S, a, h->qw.grid, h->stream), "worker launch");
        if (r == EA_OK) ++h->epoch_w;
    } else {
        r = check_cuda(h, launch_worker(W ? MODE_W : MODE_S, a, h->stream), "worker launch");
    }
    if (r == EA_OK && h->qw.pass == PASS_STASH) r = second_pass(h, h->qw, a.partials, a.e, a.words, a.scales, a.id);
    if (r != EA_OK) return r;
    if (h->qw.pass == PASS_LAZY) {  // the scales are formed for all workers before the server step
        h->lazy_w[worker] = h->cfg.error_feedback ? 1 : 0;
        h->wscales_pending = true;
    }
    h->compressed[worker] = 1;
    ++h->n_compressed;
    return EA_OK;
}

int ea_server_step(ea_handle *h)
{
    if (!h) return fail(nullptr, EA_E_INVAL, "handle is NULL");
    if (h->n_compressed != h->cfg.n)
        return fail(h, EA_E_ORDER, "round %lld: %d of %d workers compressed", static_cast<long long>(h->t),
                    h->n_compressed, h->cfg.n);
    ServerArgs a{};
    a.d = h->cfg.d;
    a.n_tiles = h->n_tiles;
    a.n = h->cfg.n;
    a.wwords = h->wcodes;
    a.wwords_stride = h->lay.wcode_stride;
    a.wscales = h->wscales;
    a.wscales_stride = h->lay.wscale_stride;
    a.qw = device_quant(h->qw);
    a.qs = device_quant(h->qs);
    a.words = h->scodes;
    a.scales = h->sscales;
    a.es = h->es;
    a.ms = h->ms;
    a.vs = h->vs;
    a.hp = round_hyper(h);
    a.ef = h->cfg.error_feedback;
    a.pass = h->qs.pass;
    a.seed = h->cfg.seed;
    a.t = static_cast<uint32_t>(h->t);
    a.partials = h->spartials;
    a.dpad = h->lay.dpad;
    a.wcode_bytes = h->lay.wcode_stride * 4;
    a.status = h->status;
    a.plan = h->splan;
    a.lazy_in = h->qs.pass == PASS_LAZY && h->lazy_s ? 1 : 0;
    const bool W = h->cfg.placement == EA_ADAM_AT_WORKER;
    int r = finalize_worker_scales(h);
    if (r != EA_OK) return r;
    if (h->qs.pass == PASS_LAZY) {
        r = check_cuda(h, W ? launch_server_lazy<MODE_W>(a, h->lazy_staged, h->stream)
                            : launch_server_lazy<MODE_S>(a, h->lazy_staged, h->stream),
                       "server launch");
        if (r == EA_OK) r = finalize_scales(h, h->qs, h->spartials, h->sscales);
        if (r == EA_OK) h->lazy_s = h->cfg.error_feedback != 0;
    } else if (h->qs.pass == PASS_GROUPED) {
        a.gp = device_group_plan(h->qs, h->epoch_s);
        r = check_cuda(h, launch_server_grouped(W ? MODE_W : MODE_S, a, h->qs.grid, h->stream), "server launch");
        if (r == EA_OK) ++h->epoch_s;
    } else {
        r = check_cuda(h, launch_server(W ? MODE_W : MODE_S, a, h->stream), "server launch");
    }
    if (r == EA_OK && h->qs.pass == PASS_STASH)
        r = second_pass(h, h->qs, h->spartials, h->es, h->scodes, h->sscales, static_cast<uint32_t>(h->cfg.n));
    if (r != EA_OK) return r;
    h->up_bits += static_cast<uint64_t>(h->cfg.n) * message_bits(h->qw, h->cfg.d);
    h->down_bits += static_cast<uint64_t>(h->cfg.n) * message_bits(h->qs, h->cfg.d);
    ++h->t;
    h->compressed.assign(h->cfg.n, 0);
    h->n_compressed = 0;
    h->has_message = true;
    return EA_OK;
}

int ea_worker_apply(ea_handle *h, float *x)
{
    if (!h) return fail(nullptr, EA_E_INVAL, "handle is NULL");
    int r = check_dev_ptr(h, x, "x");
    if (r != EA_OK) return r;
    if (!h->has_message) return fail(h, EA_E_ORDER, "no broadcast yet: call ea_server_step first");
    ApplyArgs a{};
    a.d = h->cfg.d;
    a.x = x;
    a.q = device_quant(h->qs);
    a.words = h->scodes;
    a.scales = h->sscales;
    return check_cuda(h, launch_apply(a, h->stream), "apply launch");
}

int ea_set_hparams(ea_handle *h, float alpha, float beta1, float beta2)
{
    if (!h) return fail(nullptr, EA_E_INVAL, "handle is NULL");
    const int r = check_hparams(alpha, beta1, beta2);
    if (r != EA_OK) {
        h->err = ea_last_error(nullptr);
        return r;
    }
    h->hp.alpha = alpha;
    h->hp.beta1 = beta1;
    h->hp.beta2 = beta2;
    h->hp.c1 = 1.0f - beta1;
    h->hp.c2 = 1.0f - beta2;
    return EA_OK;
}

int ea_bits_sent(const ea_handle *h, uint64_t *up_bits, uint64_t *down_bits)
{
    if (!h || !up_bits || !down_bits) return fail(nullptr, EA_E_INVAL, "NULL argument");
    *up_bits = h->up_bits;
    *down_bits = h->down_bits;
    return EA_OK;
}

int ea_round_launches(const ea_handle *h, int32_t *launches)
{
    if (!h || !launches) return fail(nullptr, EA_E_INVAL, "NULL argument");
    auto per_message = [](const QHost &q) { return q.pass == PASS_STASH ? 3 : q.pass == PASS_LAZY ? 2 : 1; };
    // lazy worker messages: one pass each, and one finalize for all of them
    const int workers = h->qw.pass == PASS_LAZY ? h->cfg.n + 1 : h->cfg.n * per_message(h->qw);
    *launches = workers + per_message(h->qs) + 1;
    return EA_OK;
}

int ea_round_index(const ea_handle *h, int64_t *t)
{
    if (!h || !t) return fail(nullptr, EA_E_INVAL, "NULL argument");
    *t = h->t;
    return EA_OK;
}

int ea_get_view(const ea_handle *h, int32_t which, int32_t index, void **dev_ptr, size_t *bytes)
{
    if (!h || !dev_ptr || !bytes) return fail(nullptr, EA_E_INVAL, "NULL argument");
    ea_handle *hm = const_cast<ea_handle *>(h);
    const bool W = h->cfg.placement == EA_ADAM_AT_WORKER;
    const bool per_worker = which == EA_VIEW_M || which == EA_VIEW_V || which == EA_VIEW_E_WORKER ||
                            which == EA_VIEW_CODES_WORKER || which == EA_VIEW_SCALES_WORKER;
    if (per_worker && (index < 0 || index >= h->cfg.n))
        return fail(hm, EA_E_INVAL, "worker %d out of [0, %d)", index, h->cfg.n);
    const int64_t dp = h->lay.dpad;
    const size_t vec = static_cast<size_t>(h->cfg.d) * 4;
    if ((which == EA_VIEW_SCALES_WORKER || which == EA_VIEW_E_WORKER) && h->wscales_pending) {
        // lazy worker messages compressed this round: their scales first
        int r = finalize_worker_scales(hm);
        if (r == EA_OK) r = check_cuda(hm, cudaStreamSynchronize(h->stream), "stream synchronize");
        if (r != EA_OK) return r;
    }
    void *p = nullptr;
    size_t n = 0;
    switch (which) {
    case EA_VIEW_M: if (W) { p = h->m + index * dp; n = vec; } break;
    case EA_VIEW_V: if (W) { p = h->v + index * dp; n = vec; } break;
    case EA_VIEW_E_WORKER:
        p = h->e + index * dp;
        n = vec;
        if (h->qw.pass == PASS_LAZY && h->lazy_w[index]) {  // the residual, formed from the kept u
            ResidArgs ra{};
            ra.d = h->cfg.d;
            ra.u = h->e + index * dp;
            ra.out = h->rview;
            ra.q = device_quant(h->qw);
            ra.scales = h->wscales + index * h->lay.wscale_stride;
            int r = check_cuda(hm, launch_lazy_resid(ra, h->stream), "residual launch");
            if (r == EA_OK) r = check_cuda(hm, cudaStreamSynchronize(h->stream), "stream synchronize");
            if (r != EA_OK) return r;
            p = h->rview;
        }
        break;
    case EA_VIEW_E_SERVER:
        p = h->es;
        n = vec;
        if (h->qs.pass == PASS_LAZY && h->lazy_s) {  // the residual, formed from the kept w
            ResidArgs ra{};
            ra.d = h->cfg.d;
            ra.u = h->es;
            ra.out = h->rview;
            ra.q = device_quant(h->qs);
            ra.scales = h->sscales;
            int r = check_cuda(hm, launch_lazy_resid(ra, h->stream), "residual launch");
            if (r == EA_OK) r = check_cuda(hm, cudaStreamSynchronize(h->stream), "stream synchronize");
            if (r != EA_OK) return r;
            p = h->rview;
        }
        break;
    case EA_VIEW_M_SERVER: if (!W) { p = h->ms; n = vec; } break;
    case EA_VIEW_V_SERVER: if (!W) { p = h->vs; n = vec; } break;
    case EA_VIEW_CODES_WORKER: p = h->wcodes + index * h->lay.wcode_stride; n = h->qw.n_words * 4; break;
    case EA_VIEW_SCALES_WORKER: p = h->wscales + index * h->lay.wscale_stride; n = h->qw.n_groups * 4; break;
    case EA_VIEW_CODES_SERVER: p = h->scodes; n = h->qs.n_words * 4; break;
    case EA_VIEW_SCALES_SERVER: p = h->sscales; n = h->qs.n_groups * 4; break;
    default: return fail(hm, EA_E_INVAL, "unknown view %d", which);
    }
    if (!p && !(which == EA_VIEW_SCALES_WORKER || which == EA_VIEW_SCALES_SERVER))
        return fail(hm, EA_E_INVAL, "view %d does not exist in this placement", which);
    *dev_ptr = p;
    *bytes = n;
    return EA_OK;
}

int ea_sync_status(ea_handle *h)
{
    if (!h) return fail(nullptr, EA_E_INVAL, "handle is NULL");
    int r = check_cuda(h, cudaStreamSynchronize(h->stream), "stream synchronize");
    if (r != EA_OK) return r;
    r = check_cuda(h, cudaGetLastError(), "pending error");
    if (r != EA_OK) return r;
    uint32_t st = 0;
    r = check_cuda(h, cudaMemcpy(&st, h->status, sizeof st, cudaMemcpyDeviceToHost), "status read");
    if (r != EA_OK) return r;
    if (st) {
        cudaMemset(h->status, 0, sizeof st);
        if (st & kStatusTimeoutBit)
            return fail(h, EA_E_TIMEOUT, "a device-side wait exceeded its time limit (status 0x%x)", st);
        return fail(h, EA_E_DEVICE_CHECK, "device status 0x%x", st);
    }
    return EA_OK;
}

const char *ea_last_error(const ea_handle *h)
{
    return h ? h->err.c_str() : g_last_error.c_str();
}

int ea_destroy(ea_handle *h)
{
    delete h;
    return EA_OK;
}

}  // extern "C"
