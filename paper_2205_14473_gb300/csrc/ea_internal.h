// ea_internal.h -- launch parameters shared by the host API (ea_api.cu) and the kernel units.
// Not installed; the public interface is include/ea.h.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace ea {

// One CTA tile: 256 threads x 4 float4 slots = 4096 coordinates.  Tiles are aligned to multiples
// of 4096 in the flat vector, so for every code width b a tile owns whole 32-bit code words.
constexpr int kThreads = 256;
constexpr int kSlots = 4;
constexpr int kTile = kThreads * kSlots * 4;
// The staged server: CTAs of kThreads compute threads and one producer warp, built for up to
// server_ctas_per_sm resident CTAs per SM; each holds at most kServerStaticSmem bytes of static
// shared memory (checked where the kernel is defined) and up to kServerMaxDynSmem of stages.  An
// SM has kSmemPerSm bytes, of which every resident CTA takes kSmemReservedPerCta for the system.
constexpr uint32_t kServerStaticSmem = 9 * 1024;
constexpr uint32_t kServerMaxDynSmem = 200 * 1024;
constexpr uint32_t kSmemPerSm = 228 * 1024;
constexpr uint32_t kSmemReservedPerCta = 1024;
constexpr int kWarps = kThreads / 32;
// Shared-memory staging of a server tile's worker scales: at most kStagedTileGroups of Q_w's groups
// meet one tile, and n times that many scales fit in kWorkerScales.
constexpr int kWorkerScales = 512;
constexpr int kStagedTileGroups = 256;
// Device ordinals for which per-device host state (kernel attributes) is kept.
constexpr int kMaxDevices = 64;

enum QKind : int { QK_IDENT = 0, QK_SIGN = 1, QK_UNIF = 2, QK_POW2 = 3 };
enum GKind : int { GK_WHOLE = 0, GK_BLOCK = 1, GK_SEG = 2 };
enum Mode : int { MODE_W = 0, MODE_S = 1 };  // Adam at the workers (the paper) / at the server

// Resident CTAs per SM a staged server kernel's registers are sized for (its __launch_bounds__, and
// the stage plan's limit): four (56 registers) for scaled-sign workers and broadcast with Adam at
// the workers, whose tile needs the fewest live values; three (72 registers) otherwise.
constexpr int server_ctas_per_sm(int mode, int qw, int qs)
{
    return (mode == MODE_W && qw == QK_SIGN && qs == QK_SIGN) ? 4 : 3;
}

// How a message's scale groups tile the vector.
struct Grouping {
    int gkind;
    int log2G;                  // GK_BLOCK: log2 of G when G is a power of two, else -1
    int64_t G;                  // GK_BLOCK: block length
    int64_t n_groups;
    const int64_t *offsets;     // GK_SEG: n_groups + 1 offsets (device)
    const int32_t *tile_group;  // GK_SEG: first group that intersects each 4096-tile (device)
    const int64_t *pair_base;   // n_groups + 1: first partial-sum slot of each group (device)
};

struct QParams {
    int kind, bits, stochastic, pow2_k, pow2_K;
    Grouping grp;
};

struct Hyper {
    float alpha, beta1, beta2, c1, c2;  // c1 = 1 - beta1, c2 = 1 - beta2, rounded to binary32
    int form;                           // 0: the paper's Adam (Algorithm 2); 1: the textbook form
    float eps, bc1, bc2;                // textbook form: eps in the denominator, 1 - beta1^t, 1 - beta2^t
};

// 1 - beta^t for the 1-based round t: beta^t by t binary64 multiplications, rounded once.
inline float bias_correction(float beta, int64_t t1)
{
    double p = 1.0;
    for (int64_t k = 0; k < t1; ++k) p *= static_cast<double>(beta);
    return static_cast<float>(1.0 - p);
}

// How the scale of a message is formed.
enum Pass : int {
    PASS_FUSED = 0,   // every group lies inside one tile: reduce, encode and store in one pass
    PASS_STASH = 1,   // groups span tiles: store the input in the residual buffer plus one
                      // partial norm per (tile, group); finalize_kernel and encode_kernel finish
    PASS_GROUPED = 2, // groups span tiles, one cooperative pass: the input stays in shared memory
                      // while the group's partial norms are combined (GroupPlan)
    PASS_LAZY = 3     // scaled sign, groups span tiles: the codes (signs) need no scale, so one pass
                      // writes them with the partial norms and keeps u itself in the residual
                      // buffer; finalize_kernel forms the scales, and e = u - Q(u) is formed from
                      // (u, s) where it is next needed (the next round's pass, or a view)
};

// The one-pass plan for scale groups that span tiles.  The vector is cut into waves, coordinate
// ranges [cuts[w], cuts[w+1]) of whole groups whose tiles fit in shared memory at once (every cut
// starts a code word and a float4 slot).  A persistent CTA takes the wave's tiles blockIdx.x,
// blockIdx.x + gridDim.x, ... (at most `slots`), parks each tile's input in shared memory and
// stores one partial norm per (group, tile); after a grid-wide barrier every CTA combines, in a
// fixed order, the partials of the groups its tiles need, and encodes its tiles.  The launch is
// cooperative (all CTAs resident), so the barrier completes; its wait is still bounded and
// reports EA_E_TIMEOUT.
struct GroupPlan {
    int64_t n_waves;
    const int64_t *cuts;         // n_waves + 1 coordinate offsets (device)
    unsigned long long *arrive;  // CTAs arrived at the wave barriers, over all launches
    uint64_t epoch;              // launches made with this counter before this one
    int slots;                   // tiles of input a CTA holds in shared memory
};

// Scales of groups a grouped CTA holds in shared memory for one wave (the plan keeps the grouped
// pass off when some CTA's tiles of a wave meet more groups).
constexpr int kGroupedScales = 256;

// Shape of a grouped kernel on this device: CTAs per SM and tile slots per CTA.
struct GroupedShape {
    int ctas_per_sm, slots;
};

struct WorkerArgs {
    int64_t d, n_tiles;
    const float *g;
    float *m, *v, *e;
    QParams q;
    uint32_t *words;
    float *scales;
    Hyper hp;
    int ef, pass;
    uint64_t seed;
    uint32_t id, t;
    double *partials;
    GroupPlan gp;             // PASS_GROUPED
    uint32_t *status;         // device status word (timeouts); may be null outside a handle
    int lazy_in;              // PASS_LAZY: e holds the previous round's u, scales its scales
};

// Shared-memory staging plan of the pipelined (persistent, bulk-copy) kernels.  A stage holds one
// tile's inputs; byte offsets are relative to the stage start and 128-byte aligned.
struct StagePlan {
    int enabled;               // 0: use the direct-load kernel
    int stages;                // pipeline depth
    int grid;                  // persistent CTAs
    uint32_t stage_bytes;      // bytes of one stage
    uint32_t smem_bytes;       // dynamic shared memory per CTA (barriers + stages)
    uint32_t off_a, off_b, off_c, off_d;  // up to four 16 KB state tiles (kernel-specific meaning)
    uint32_t off_codes;        // n code chunks of code_chunk bytes
    uint32_t code_chunk;       // bytes of one worker's codes for one tile (4096 b / 8)
    uint32_t off_scales;       // n worker scales (binary32)
};

struct ServerArgs {
    int64_t d, n_tiles;
    int n;
    const uint32_t *wwords;   // worker i's codes at wwords + i * wwords_stride
    int64_t wwords_stride;
    const float *wscales;     // worker i's scales at wscales + i * wscales_stride
    int64_t wscales_stride;
    QParams qw, qs;
    uint32_t *words;          // the broadcast
    float *scales;
    float *es, *ms, *vs;
    Hyper hp;
    int ef, pass;
    uint64_t seed;
    uint32_t t;
    double *partials;
    int64_t dpad;             // padded length of e_s, m_s, v_s (multiple of 64)
    int64_t wcode_bytes;      // padded bytes of one worker's code stream (multiple of 256)
    uint32_t *status;         // device status word (timeouts)
    StagePlan plan;
    GroupPlan gp;             // PASS_GROUPED (Q_s's groups)
    int lazy_in;              // PASS_LAZY: es holds the previous round's w, scales its scales
};

// Second pass of PASS_STASH: encode the stashed input in buf, leave the residual in buf.
struct EncodeArgs {
    int64_t d, n_tiles;
    float *buf;
    QParams q;
    uint32_t *words;
    const float *scales;
    int ef;
    uint64_t seed;
    uint32_t id, t;
};

// The scales of n_msgs messages (blockIdx.y; 0 counts as 1), message y's partials at
// partials + y * partials_stride and its scales at scales + y * scales_stride.
struct FinalizeArgs {
    int64_t d;
    QParams q;
    const double *partials;
    float *scales;
    int n_msgs;
    int64_t partials_stride, scales_stride;
};

// PASS_LAZY: the residual u - Q(u) of the u kept in `u`, with the scales of its message, into out.
struct ResidArgs {
    int64_t d;
    const float *u;
    float *out;
    QParams q;
    const float *scales;
};

struct ApplyArgs {
    int64_t d;
    float *x;
    QParams q;
    const uint32_t *words;
    const float *scales;
};

cudaError_t launch_worker(int mode, const WorkerArgs &a, cudaStream_t s);
// The one-pass kernels of PASS_GROUPED (cooperative launches of `grid` CTAs) and their shapes.
cudaError_t launch_worker_grouped(int mode, const WorkerArgs &a, int grid, cudaStream_t s);
cudaError_t worker_grouped_shape(int mode, int qk, GroupedShape *out);
template <int MODE, int QS>
cudaError_t launch_server_grouped_for_qs(const ServerArgs &a, int grid, cudaStream_t s);
template <int MODE, int QS>
cudaError_t server_grouped_shape_for_qs(int qw, GroupedShape *out);
cudaError_t launch_server_grouped(int mode, const ServerArgs &a, int grid, cudaStream_t s);
// PASS_LAZY for a scaled-sign broadcast (instantiated with the QS = QK_SIGN server kernels).
// staged: every tile's worker codes and scales fit the shared-memory staging (lazy_server_staged).
template <int MODE>
cudaError_t launch_server_lazy(const ServerArgs &a, bool staged, cudaStream_t s);
cudaError_t server_grouped_shape(int mode, int qw, int qs, GroupedShape *out);
// The server kernel for one placement and broadcast quantizer kind; each (MODE, QS) pair is
// instantiated only in its own translation unit, ea_server_<mode>_q<QS>.cu.
template <int MODE, int QS>
cudaError_t launch_server_for_qs(const ServerArgs &a, cudaStream_t s);

// The server kernel for the placement and the broadcast quantizer kind of `a` (ea_api.cu).
cudaError_t launch_server(int mode, const ServerArgs &a, cudaStream_t s);
cudaError_t launch_finalize(const FinalizeArgs &a, cudaStream_t s);
cudaError_t launch_encode(const EncodeArgs &a, cudaStream_t s);
cudaError_t launch_lazy_resid(const ResidArgs &a, cudaStream_t s);
cudaError_t launch_apply(const ApplyArgs &a, cudaStream_t s);
cudaError_t launch_fill(float *p, int64_t count, float value, cudaStream_t s);

// Record the text that ea_last_error(NULL) reports for a failure that has no handle.
void set_last_error(const char *msg);

}  // namespace ea
