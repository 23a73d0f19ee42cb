// ea_noalloc.cu -- ea_worker_compress_noalloc: the worker compress of a message with one scale
// for the whole vector, for callers that cannot allocate device memory.
//
// Who needs it: code that runs where no device allocation may happen -- inside a framework whose
// caching allocator has already reserved the GPU's memory, in a latency-critical path where the
// implicit synchronisation of cudaMalloc/cudaFree is not acceptable, or in a plug-in that is
// handed only the buffers it works on.  Such a caller owns g, m, v, e and the message buffers but
// cannot provide the scratch that the two-pass scale needs (one partial l1/l_inf norm per
// 4096-coordinate tile).  Here that scratch is a fixed array in device global memory, compiled
// into the library: every GPU that loads the library holds it (128 KB + 256 B) until the process
// exits, whether or not the function is called.
//
// The kernels are those of the two-pass scale that ea_worker_compress also launches (for the
// uniform grid; a scaled-sign message there takes the lazy pass, with the same results); only where
// their scratch lives differs.
#include <cmath>
#include <cstdarg>
#include <cstdio>

#include "ea.h"
#include "ea_internal.h"

namespace {

using namespace ea;

constexpr int64_t kMaxTiles = EA_NOALLOC_MAX_D / kTile;
// [0, 16): the two offsets of the single scale group's partial norms; [256, ...): the partials.
__device__ __align__(256) unsigned char g_scratch[256 + kMaxTiles * sizeof(double)];

__global__ void write_group_offsets(int64_t *pair_base, int64_t n_tiles)
{
    if (threadIdx.x == 0) {
        pair_base[0] = 0;
        pair_base[1] = n_tiles;
    }
}

int fail(int code, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    set_last_error(buf);
    return code;
}

// The device address of g_scratch in the current context, looked up on every call: the lookup
// allocates nothing, and a cached address would go stale after cudaDeviceReset or when another
// context is made current on the same device.
int scratch_address(unsigned char **out)
{
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return fail(EA_E_CUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    *out = static_cast<unsigned char *>(p);
    return EA_OK;
}

bool aligned16(const void *p) { return p && (reinterpret_cast<uintptr_t>(p) % 16) == 0; }

}  // namespace

extern "C" int ea_worker_compress_noalloc(const ea_config *cfg, int32_t worker, int64_t round, const float *g,
                                          float *m, float *v, float *e, uint32_t *codes, float *scales,
                                          void *stream)
{
    if (!cfg) return fail(EA_E_INVAL, "config is NULL");
    const ea_quantizer &q = cfg->qw;
    const int64_t d = cfg->d;
    if (d < 1) return fail(EA_E_INVAL, "d must be >= 1");
    if (d > EA_NOALLOC_MAX_D)
        return fail(EA_E_INVAL, "d = %lld exceeds the allocation-free limit of %lld coordinates",
                    static_cast<long long>(d), static_cast<long long>(EA_NOALLOC_MAX_D));
    if (cfg->n < 1 || worker < 0 || worker >= cfg->n) return fail(EA_E_INVAL, "worker %d out of [0, %d)", worker, cfg->n);
    if (round < 0 || round > 0xffffffffLL) return fail(EA_E_INVAL, "round out of [0, 2^32)");
    if (cfg->placement != EA_ADAM_AT_WORKER && cfg->placement != EA_ADAM_AT_SERVER)
        return fail(EA_E_INVAL, "unknown placement %d", cfg->placement);
    if (cfg->error_feedback != 0 && cfg->error_feedback != 1) return fail(EA_E_INVAL, "error_feedback is 0 or 1");
    if (cfg->adam_form != 0 && cfg->adam_form != 1) return fail(EA_E_INVAL, "adam_form is 0 or 1");
    if (!std::isfinite(cfg->alpha) || !(cfg->beta1 >= 0.0f && cfg->beta1 < 1.0f) ||
        !(cfg->beta2 >= 0.0f && cfg->beta2 < 1.0f) || !(cfg->eps > 0.0f))
        return fail(EA_E_INVAL, "hyper-parameters out of range");
    const bool sign = q.kind == EA_Q_SIGN_L1 && q.bits == 1;
    const bool unif = q.kind == EA_Q_UNIFORM_MAX && (q.bits == 2 || q.bits == 4 || q.bits == 8 || q.bits == 16);
    if (!sign && !unif)
        return fail(EA_E_UNSUPPORTED, "the allocation-free compress takes Q_w = scaled sign or uniform grid");
    if (q.group != 0) return fail(EA_E_UNSUPPORTED, "the allocation-free compress takes one scale for the whole vector");
    if (q.stochastic != 0 && !(unif && q.stochastic == 1)) return fail(EA_E_INVAL, "stochastic is 0, or 1 for the uniform grid");
    const bool W = cfg->placement == EA_ADAM_AT_WORKER;
    if (!aligned16(g) || !aligned16(e) || !aligned16(codes) || !scales || (W && (!aligned16(m) || !aligned16(v))))
        return fail(EA_E_ALIGN, "g, e, codes (and m, v with Adam at the worker) must be 16-byte aligned, scales non-NULL");

    unsigned char *scratch = nullptr;
    int r = scratch_address(&scratch);
    if (r != EA_OK) return r;
    int64_t *pair_base = reinterpret_cast<int64_t *>(scratch);
    double *partials = reinterpret_cast<double *>(scratch + 256);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int64_t n_tiles = (d + kTile - 1) / kTile;

    QParams qp{};
    qp.kind = q.kind;
    qp.bits = q.bits;
    qp.stochastic = q.stochastic;
    qp.grp.gkind = GK_WHOLE;
    qp.grp.log2G = -1;
    qp.grp.n_groups = 1;
    qp.grp.pair_base = pair_base;

    WorkerArgs a{};
    a.d = d;
    a.n_tiles = n_tiles;
    a.g = g;
    a.m = W ? m : nullptr;
    a.v = W ? v : nullptr;
    a.e = e;
    a.q = qp;
    a.words = codes;
    a.scales = scales;
    a.hp.alpha = cfg->alpha;
    a.hp.beta1 = cfg->beta1;
    a.hp.beta2 = cfg->beta2;
    a.hp.c1 = 1.0f - cfg->beta1;
    a.hp.c2 = 1.0f - cfg->beta2;
    a.hp.form = cfg->adam_form;
    a.hp.eps = cfg->eps;
    if (cfg->adam_form == 1) {
        a.hp.bc1 = bias_correction(cfg->beta1, round + 1);
        a.hp.bc2 = bias_correction(cfg->beta2, round + 1);
    }
    a.ef = cfg->error_feedback;
    a.pass = d <= kTile ? PASS_FUSED : PASS_STASH;
    a.seed = cfg->seed;
    a.id = static_cast<uint32_t>(worker);
    a.t = static_cast<uint32_t>(round);
    a.partials = partials;

    cudaError_t ce = cudaSuccess;
    if (a.pass == PASS_STASH) {
        write_group_offsets<<<1, 32, 0, s>>>(pair_base, n_tiles);
        ce = cudaGetLastError();
    }
    if (ce == cudaSuccess) ce = launch_worker(W ? MODE_W : MODE_S, a, s);
    if (ce == cudaSuccess && a.pass == PASS_STASH) {
        FinalizeArgs f{};
        f.d = d;
        f.q = qp;
        f.partials = partials;
        f.scales = scales;
        ce = launch_finalize(f, s);
        if (ce == cudaSuccess) {
            EncodeArgs en{};
            en.d = d;
            en.n_tiles = n_tiles;
            en.buf = e;
            en.q = qp;
            en.words = codes;
            en.scales = scales;
            en.ef = cfg->error_feedback;
            en.seed = cfg->seed;
            en.id = a.id;
            en.t = a.t;
            ce = launch_encode(en, s);
        }
    }
    if (ce != cudaSuccess) return fail(EA_E_CUDA, "launch: %s", cudaGetErrorString(ce));
    return EA_OK;
}
