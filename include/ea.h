/*
 * ea.h -- C ABI of the GB300 (sm_103a) implementation of one round of Efficient-Adam's two-way
 * quantized, two-way error-feedback pipeline (Chen, Shen, Liu, Luo, arxiv 2205.14473).
 *
 * The n workers and the server of the parameter-server model (Figure 1) are simulated as separate
 * buffers on one GPU.  One round t is:
 *   ea_worker_compress(h, i, g_i)  for every worker i   -- Algorithm 2, the worker's message
 *   ea_server_step(h)                                   -- Algorithm 1, the server's broadcast
 *   ea_worker_apply(h, x)          for every replica    -- Algorithms 1-2, x <- x - Q_s(...)
 * Every call is asynchronous on the stream given to ea_init and never synchronizes, except
 * ea_sync_status.  The library allocates no device memory: the caller passes one workspace of
 * ea_workspace_bytes() bytes, and owns it, the stream, the gradients and x.
 *
 * Precision and formats (shared with the test oracle by specification, not by code):
 *   - every per-coordinate expression is evaluated in binary32 with round-to-nearest-even, one
 *     rounding per operation, in the order Algorithms 1-2 write it;
 *   - a message is a packed code stream (coordinate j at bits [j*b, j*b + b) of little-endian
 *     32-bit words, least significant bit first) plus one binary32 scale per scale group;
 *   - the l1 norm of a scale group is formed to better than 1e-10 relative and rounded once.
 *
 * Return values: EA_OK (0) or a negative EA_E_* code; ea_last_error() describes the last failure.
 */
#ifndef EA_H
#define EA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define EA_OK 0
#define EA_E_INVAL (-1)        /* a bad argument or configuration */
#define EA_E_ALIGN (-2)        /* a device pointer that is not 16-byte aligned */
#define EA_E_WORKSPACE (-3)    /* workspace missing, misaligned (256 B) or too small */
#define EA_E_ORDER (-4)        /* a call out of the round protocol */
#define EA_E_CUDA (-5)         /* a CUDA runtime error (launch or stream) */
#define EA_E_TIMEOUT (-6)      /* a bounded device-side wait gave up */
#define EA_E_DEVICE_CHECK (-7) /* a device-side consistency check failed */
#define EA_E_UNSUPPORTED (-8)  /* a valid configuration this build does not implement */

/* Quantization mappings (Definition 1) and compressors (Definition 3) of the paper. */
typedef enum {
    EA_Q_IDENTITY = 0,     /* 32-bit float, "Ours_full" of Table 2; 32 bits, no scale */
    EA_Q_SIGN_L1 = 1,      /* scaled sign, scale = ||u_group||_1 / |group|, sign(0) = +1; 1 bit */
    EA_Q_UNIFORM_MAX = 2,  /* Example 1: Q1(||u||_inf) * nearest point of {i/(2^k-1)}, k = bits-1 */
    EA_Q_POW2 = 3          /* Example 2: sign(u) * nearest of {2^k, ..., 2^K}; no scale */
} ea_qkind;

/* Where the Adam moments live.  The paper (Algorithm 2) keeps them on every worker; the second
 * placement keeps them on the server (workers send Q_w(g + e)). */
typedef enum { EA_ADAM_AT_WORKER = 0, EA_ADAM_AT_SERVER = 1 } ea_placement;

typedef struct ea_quantizer {
    int32_t kind;        /* ea_qkind */
    int32_t bits;        /* SIGN_L1: 1; UNIFORM_MAX: 2, 4, 8 or 16; POW2: 4 or 8; IDENTITY: 32 */
    int32_t stochastic;  /* UNIFORM_MAX only: round up with probability frac(y), Philox4x32-10 */
    int32_t pow2_k;      /* POW2: smallest exponent k (>= -126) */
    int32_t pow2_K;      /* POW2: largest exponent K, k < K, K - k + 2 <= 2^(bits-1) */
    int32_t n_seg;       /* number of segments when group < 0 */
    int64_t group;       /* scale groups: 0 whole vector, > 0 blocks of this length (last one
                            ragged), < 0 the explicit segments below */
    const int64_t *seg_lengths; /* host memory, n_seg positive lengths summing to d; copied */
} ea_quantizer;

typedef struct ea_config {
    int64_t d;            /* dimension, >= 1 */
    int32_t n;            /* workers N, 1 <= n <= 1024 */
    int32_t placement;    /* ea_placement */
    ea_quantizer qw;      /* Q_w, the workers' mapping (Algorithm 2) */
    ea_quantizer qs;      /* Q_s, the server's mapping (Algorithm 1) */
    float alpha;          /* alpha_t (ea_set_hparams changes it between rounds) */
    float beta1;          /* beta, the first-moment coefficient, 0 <= beta1 < 1 */
    float beta2;          /* theta_t, the second-moment coefficient, 0 <= beta2 < 1 */
    float eps;            /* adam_form 0: v_0 = eps (Algorithm 2), no eps in the denominator, no bias
                             correction; adam_form 1: v_0 = 0 and eps added to the denominator */
    int32_t error_feedback; /* 1 = the paper; 0 = the "_err" ablation of Table 2 */
    int32_t adam_form;    /* 0 = the paper's Adam (Algorithm 2); 1 = the textbook form, step
                             alpha (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps), t 1-based */
    uint64_t seed;        /* Philox key for stochastic rounding */
} ea_config;

typedef struct ea_handle ea_handle;

/* Bytes of workspace ea_init needs for cfg (Algorithms 1-2 state: m, v, e per worker, e_s (and
 * m, v on the server in EA_ADAM_AT_SERVER), the n + 1 messages and small tables).
 * Returns EA_E_INVAL for an invalid cfg, EA_E_UNSUPPORTED for one this build does not run. */
int ea_workspace_bytes(const ea_config *cfg, size_t *bytes);

/* Validate cfg, carve the caller's device workspace (256-byte aligned, >= ea_workspace_bytes,
 * owned by the caller and untouched by anyone else until ea_destroy) and initialise the state of
 * Algorithms 1-2 on `stream` (a cudaStream_t; NULL = the legacy default stream): m = 0, v = eps,
 * every residual e = 0.  x_1 is the caller's.  *out receives a host handle. */
int ea_init(const ea_config *cfg, void *workspace, size_t workspace_bytes, void *stream, ea_handle **out);

/* Algorithm 2 for worker `worker` in the current round: with Adam at the worker,
 *   v <- theta v + (1-theta) g^2;  m <- beta m + (1-beta) g;  u = alpha m / sqrt(v) + e;
 * with Adam at the server, u = g + e.  Then send Q_w(u) (into the worker's message buffer) and
 * keep e <- u - Q_w(u).  g: d binary32 values, 16-byte aligned, read only, not retained; device
 * memory, or pinned host memory mapped into the device's address space (the kernel then reads it
 * over the host link, with no staging copy).  Each worker compresses once per round; EA_E_ORDER
 * otherwise.  A scaled-sign message whose scale groups span 4096-coordinate tiles has its codes when
 * this returns; its scales are formed, with those of the other workers' messages, by the next
 * ea_server_step (or by a view of them, see ea_get_view), and e is kept as u (see ea_get_view). */
int ea_worker_compress(ea_handle *h, int32_t worker, const float *g);

/* Algorithm 1: average the n decoded worker messages (summed in worker order, then divided by
 * n), w = avg + e_s (with Adam at the server: Adam on avg with the server's m, v, then
 * w = alpha m / sqrt(v) + e_s), broadcast Q_s(w), keep e_s <- w - Q_s(w), add the round's bits
 * to the ledger and advance the round.  EA_E_ORDER unless all n workers compressed this round. */
int ea_server_step(ea_handle *h);

/* x <- x - Q_s(w) from the latest broadcast (Algorithm 1's and Algorithm 2's parameter update).
 * x: device, d binary32 values, 16-byte aligned, updated in place.  Call once per replica of x.
 * EA_E_ORDER before the first ea_server_step. */
int ea_worker_apply(ea_handle *h, float *x);

/* alpha_t, beta and theta_t (= beta2) for the calls that follow, e.g. between rounds: Assumption 2
 * sets theta_t = 1 - theta/T and alpha_t = alpha/sqrt(T) from the horizon T; the experiments decay
 * alpha in steps.  Same ranges as ea_config; EA_E_INVAL otherwise (nothing changed). */
int ea_set_hparams(ea_handle *h, float alpha, float beta1, float beta2);

/* Cumulative bits sent (Corollary 1's accounting): up = per round n messages of d*b_w bits plus
 * 32 per scale word of Q_w; down = the broadcast counted once per receiving worker, n messages of
 * d*b_s bits plus Q_s's scale words.  Padding bits of the last word are not counted. */
int ea_bits_sent(const ea_handle *h, uint64_t *up_bits, uint64_t *down_bits);

/* Rounds completed (ea_server_step calls). */
int ea_round_index(const ea_handle *h, int64_t *t);

/* Kernel launches that one round makes on the stream: n worker compresses, one server step and one
 * apply.  A message whose scale groups lie inside 4096-coordinate tiles takes one launch.  When the
 * groups span tiles:
 *   - a scaled-sign message takes one pass, which writes the codes (the signs, which need no scale)
 *     with the groups' partial norms, and a finalize forms the scales: one finalize for all worker
 *     messages (at the server step, or at a view of a worker's scales or residual), one for the
 *     broadcast (the residual is formed from the kept input where it is next read; see the views);
 *   - another message takes one launch in the grouped kernel, which holds u in shared memory while
 *     the partial norms are combined, when its waves fit: for the broadcast, groups of up to ~7.5
 *     million coordinates on a GB300; for a worker message, no more 4096-tiles than the grouped
 *     kernel has resident CTAs;
 *   - otherwise three: the two-pass scale (stash, finalize, encode). */
int ea_round_launches(const ea_handle *h, int32_t *launches);

/* Device views into the workspace (for inspection and checkpoints); index = worker for per-worker
 * views, ignored otherwise.  *bytes receives the view's size.  A view that does not exist in the
 * configured placement returns EA_E_INVAL.
 * A scaled-sign message whose groups span tiles keeps its quantizer's input (u of a worker, w of
 * the server) in place of the residual, which is formed from that input and the message's scales,
 * e = u - Q(u), where it is next needed.  EA_VIEW_E_WORKER and EA_VIEW_E_SERVER then form it, on the
 * handle's stream, into one workspace buffer shared by these views, and synchronize the stream
 * before returning: such a view is a snapshot, valid until the next residual view or the next
 * round; the kept state is unchanged.  Every other view aliases the live state. */
enum {
    EA_VIEW_M = 0,             /* worker m (float[d]), Adam at the worker */
    EA_VIEW_V = 1,             /* worker v (float[d]), Adam at the worker */
    EA_VIEW_E_WORKER = 2,      /* worker residual e (float[d]) */
    EA_VIEW_E_SERVER = 3,      /* server residual e_s (float[d]) */
    EA_VIEW_M_SERVER = 4,      /* server m (float[d]), Adam at the server */
    EA_VIEW_V_SERVER = 5,      /* server v (float[d]), Adam at the server */
    EA_VIEW_CODES_WORKER = 6,  /* worker message codes (uint32[ceil(d*b_w/32)]) */
    EA_VIEW_SCALES_WORKER = 7, /* worker message scales (float[groups of Q_w]) */
    EA_VIEW_CODES_SERVER = 8,  /* broadcast codes (uint32[ceil(d*b_s/32)]) */
    EA_VIEW_SCALES_SERVER = 9  /* broadcast scales (float[groups of Q_s]) */
};
int ea_get_view(const ea_handle *h, int32_t which, int32_t index, void **dev_ptr, size_t *bytes);

/* Synchronize the stream and report any asynchronous CUDA error or device-side check. */
int ea_sync_status(ea_handle *h);

/* Largest d accepted by ea_worker_compress_noalloc. */
#define EA_NOALLOC_MAX_D ((int64_t)16384 * 4096)

/* The paper has no counterpart: this is a deployment convenience.  Worker compress (the same
 * computation as ea_worker_compress, with the same results; it always takes the two-pass scale --
 * stash, finalize, encode -- and leaves the residual e itself in its buffer) for callers that cannot allocate
 * device memory -- code running inside a framework whose caching allocator has already reserved
 * the GPU's memory, latency-critical paths that must not take cudaMalloc's implicit
 * synchronisation, or plug-ins that are handed only the buffers they work on.  It needs no handle
 * and no workspace: the caller passes the worker's state and message buffers, and the scratch of
 * the two-pass scale (one partial norm per 4096-coordinate tile) is a fixed 128 KB array in device
 * memory compiled into the library, which every GPU that loads the library holds until the process
 * exits.  Nothing is allocated (no cudaMalloc/cudaFree, no library allocator).
 *   - Only Q_w = EA_Q_SIGN_L1 or EA_Q_UNIFORM_MAX with one scale for the whole vector (group 0);
 *     other quantizers return EA_E_UNSUPPORTED.  cfg->qs is ignored.
 *   - 1 <= d <= EA_NOALLOC_MAX_D (67,108,864); larger d returns EA_E_INVAL.
 *   - g (read), m and v (Adam at the worker; ignored, may be NULL, with Adam at the server) and e
 *     (read and written): device, d binary32 values, 16-byte aligned.  Start them at m = 0,
 *     v = eps (0 with adam_form 1), e = 0 as Algorithm 2 does.  codes: device, 16-byte aligned, room for
 *     4 * ceil(d * bits / 128) words; scales: device, one binary32.  round: the 0-based round,
 *     which with `worker` and cfg->seed keys the stochastic rounding.  stream: a cudaStream_t.
 *   - Every call looks up the scratch array's device address in the current device's context
 *     (cudaGetSymbolAddress, which allocates nothing); the first call on a device may also load
 *     the library's module there, so make that first call before any stream capture.
 *   - Every call shares the one array, which keeps the last call's contents; the calls rewrite all
 *     of it that they read.  Calls that overlap on the GPU race: order them on one stream or with
 *     events. */
int ea_worker_compress_noalloc(const ea_config *cfg, int32_t worker, int64_t round, const float *g, float *m,
                               float *v, float *e, uint32_t *codes, float *scales, void *stream);

/* Failure-detection check (no counterpart in the paper).  The staged server's waits on its
 * shared-memory stages are bounded: after the limit the kernel records EA_E_TIMEOUT in the
 * handle's status word, finishes its own copies and returns, and ea_sync_status reports it.  This
 * runs that wait and that report on their own: one CTA waits on an mbarrier that nothing arrives
 * on (arrive = 0), so the wait runs out after limit_cycles SM clock cycles, or on one that
 * completes first (arrive = 1).  No fault, trap or unbounded loop is involved.
 *   - limit_cycles: 1 .. 4,000,000,000 (the server's own limit, ~2 s); arrive: 0 or 1.
 *   - stream: a cudaStream_t; the call synchronizes it.
 *   - *timed_out: 1 if the kernel reported EA_E_TIMEOUT, else 0.
 *   - Returns EA_E_INVAL for out-of-range arguments, EA_E_CUDA if a CUDA call fails. */
int ea_selftest_bounded_wait(int64_t limit_cycles, int32_t arrive, void *stream, int32_t *timed_out);

/* Text of the last error on h (or of the last handle-less failure when h is NULL). */
const char *ea_last_error(const ea_handle *h);

/* Release the host handle.  The workspace stays the caller's.  h may be NULL. */
int ea_destroy(ea_handle *h);

#ifdef __cplusplus
}
#endif

#endif /* EA_H */
