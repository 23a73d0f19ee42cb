/*
 * ea_oracle.c -- plain, slow CPU oracle of one Efficient-Adam round.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg
 * and reference arm (--impl reference, the oracle timed on host cores) may load this file's library.  It shares no code, header, table or helper with the CUDA
 * library; it was written from the paper (Chen, Shen, Liu, Luo, "Efficient-Adam:
 * Communication-Efficient Distributed Adam", arxiv 2205.14473) and from the message format stated
 * below.
 *
 * What it computes
 *   - Algorithm 2 (the i-th worker): v <- theta v + (1-theta) g^2, m <- beta m + (1-beta) g,
 *     u = alpha m / sqrt(v) + e, send delta = Q_w(u), e <- u - delta.  Initial m = 0, v = eps, e = 0.
 *   - Algorithm 1 (the server): average the decoded deltas, w = avg + e_s, broadcast Q_s(w),
 *     e_s <- w - Q_s(w), x <- x - Q_s(w).
 *   - A second placement in which the Adam moments live on the server (workers send Q_w(g + e)),
 *     selected by `mode`; the paper itself uses the first.
 *   - alpha_t and theta_t may change between rounds (Assumption 2 sets them from T; the experiments
 *     decay alpha in steps): the caller updates the config before a round.  A textbook Adam form
 *     (bias correction, eps in the denominator, v_0 = 0) is selected by `adam_form`.
 *   - Quantizers: Example 1 (l_inf-scaled uniform grid, deterministic nearest point), the same grid
 *     with stochastic rounding driven by Philox4x32-10, Example 2 (nearest power of two), the scaled
 *     sign compressor of Definition 3 (scale = mean |u| of the group) and the 32-bit identity
 *     ("Ours_full" of Table 2).
 *
 * Precision.  The paper fixes binary32: Example 1 takes the scale from M_1, the 32-bit floats, and
 * the parameter, moment and residual vectors are 32-bit float vectors.  Every arithmetic step is
 * therefore evaluated in binary32 with IEEE round-to-nearest-even, one rounding per operation of
 * the paper's expression, in the order the paper writes it (build with -ffp-contract=off, no fast
 * math).  The l1 norm of a group is accumulated in binary64 in index order and rounded to binary32
 * once, after the division by the group length.
 *
 * Message format (shared by specification with the CUDA library, not by code).
 *   - A message is a packed code stream plus one binary32 scale per scale group (none for the
 *     identity and power-of-two quantizers).  Coordinate l occupies bits [l*b, l*b + b) of the
 *     stream, least significant bit first, in 32-bit words: word (l*b)/32, shift (l*b)%32.
 *   - sign:      b = 1, code 1 means u >= 0 (sign(0) = +1), decode +-s.
 *   - uniform:   b in {2,4,8,16}, L = 2^(b-1) - 1, q in [-L, L], code = q + L, decode s * (q / L).
 *   - pow2:      bit b-1 = sign (1 = negative), low b-1 bits = exponent index i = j - k in
 *                [0, K-k]; the all-ones index codes 0 (sign(0) = 0).  Decode +-2^(k+i).
 *   - identity:  b = 32, the code is the binary32 pattern itself.
 *
 * Stochastic rounding.  U_j = (w >> 8) * 2^-24 where w is word (j mod 4) of
 * Philox4x32-10(counter = (lo32(j/4), hi32(j/4), id, t), key = (lo32(seed), hi32(seed))), j the
 * global coordinate, id the worker index (the server uses id = n), t the 0-based round.  Round up
 * iff U_j < y - floor(y).  Philox4x32-10 is the counter-based generator of Salmon, Moraes, Dror and
 * Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3" (SC'11), written here from that definition.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

enum { ORA_Q_IDENTITY = 0, ORA_Q_SIGN_L1 = 1, ORA_Q_UNIFORM_MAX = 2, ORA_Q_POW2 = 3 };
enum { ORA_ADAM_AT_WORKER = 0, ORA_ADAM_AT_SERVER = 1 };

/* A quantizer and its scale groups: group g covers coordinates [offsets[g], offsets[g+1]). */
typedef struct {
    int32_t kind;
    int32_t bits;
    int32_t stochastic;
    int32_t pow2_k;
    int32_t pow2_K;
    int32_t reserved;
    int64_t n_groups;
    const int64_t *offsets;
} ora_quant;

/* ---------------------------------------------------------------- Philox4x32-10 (Salmon et al.) */

static void philox_one_round(uint32_t c[4], const uint32_t k[2])
{
    /* Two 32x32->64 products of the even counter words with the round multipliers; the odd
     * words and the key are mixed into the high halves (the Philox S-box for N = 4, W = 32). */
    const uint64_t prod0 = (uint64_t)0xD2511F53u * (uint64_t)c[0];
    const uint64_t prod1 = (uint64_t)0xCD9E8D57u * (uint64_t)c[2];
    const uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    const uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    const uint32_t n0 = hi1 ^ c[1] ^ k[0];
    const uint32_t n2 = hi0 ^ c[3] ^ k[1];
    c[0] = n0;
    c[1] = lo1;
    c[2] = n2;
    c[3] = lo0;
}

void ora_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    uint32_t c[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
    uint32_t k[2] = {key[0], key[1]};
    for (int r = 0; r < 10; ++r) {
        if (r > 0) { /* Weyl sequence key schedule between rounds */
            k[0] += 0x9E3779B9u;
            k[1] += 0xBB67AE85u;
        }
        philox_one_round(c, k);
    }
    for (int i = 0; i < 4; ++i) out[i] = c[i];
}

/* The uniform variate used to round coordinate j up or down (see the header). */
float ora_uniform(uint64_t seed, uint32_t id, uint32_t t, int64_t j)
{
    const uint64_t blk = (uint64_t)j >> 2;
    const uint32_t ctr[4] = {(uint32_t)blk, (uint32_t)(blk >> 32), id, t};
    const uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
    uint32_t w[4];
    ora_philox4x32_10(ctr, key, w);
    return (float)(w[j & 3] >> 8) * 0x1p-24f;
}

/* ------------------------------------------------------------------------------- code stream */

int64_t ora_code_words(int64_t d, int bits) { return (d * (int64_t)bits + 31) / 32; }

static void put_code(uint32_t *words, int64_t l, int bits, uint32_t code)
{
    const int64_t pos = l * (int64_t)bits;
    words[pos >> 5] |= code << (pos & 31);
}

static uint32_t get_code(const uint32_t *words, int64_t l, int bits)
{
    const int64_t pos = l * (int64_t)bits;
    const uint32_t w = words[pos >> 5];
    if (bits == 32) return w;
    return (w >> (pos & 31)) & ((1u << bits) - 1u);
}

/* ---------------------------------------------------------------------------------- quantizers */

static float f32_from_bits(uint32_t b) { float f; memcpy(&f, &b, 4); return f; }
static uint32_t bits_from_f32(float f) { uint32_t b; memcpy(&b, &f, 4); return b; }

/* Example 2: sign(x) times the element of {2^k, ..., 2^K} nearest to |x| (ties go up). */
static uint32_t pow2_encode(float x, int k, int K, int bits)
{
    const uint32_t zero_idx = (1u << (bits - 1)) - 1u;
    if (x == 0.0f) return zero_idx; /* sign(0) = 0, so Q(0) = 0 */
    const uint32_t sign = (x < 0.0f) ? (1u << (bits - 1)) : 0u;
    const float a = fabsf(x);
    int j;
    if (a <= ldexpf(1.0f, k)) {
        j = k;
    } else if (a >= ldexpf(1.0f, K)) {
        j = K;
    } else {
        int ex;
        frexpf(a, &ex);   /* a = f * 2^ex with f in [0.5, 1): 2^(ex-1) <= a < 2^ex */
        j = ex - 1;
        if (a >= 1.5f * ldexpf(1.0f, j)) j += 1; /* nearest in linear distance; midpoint rounds up */
    }
    return sign | (uint32_t)(j - k);
}

static float pow2_decode(uint32_t code, int k, int bits)
{
    const uint32_t zero_idx = (1u << (bits - 1)) - 1u;
    const uint32_t idx = code & zero_idx;
    if (idx == zero_idx) return 0.0f;
    const float mag = ldexpf(1.0f, k + (int)idx);
    return (code >> (bits - 1)) ? -mag : mag;
}

/* Decode coordinate l of a message whose group scale is s. */
static float decode_one(const ora_quant *q, uint32_t code, float s)
{
    switch (q->kind) {
    case ORA_Q_IDENTITY:
        return f32_from_bits(code);
    case ORA_Q_SIGN_L1:
        return code ? s : -s;
    case ORA_Q_UNIFORM_MAX: {
        const int L = (1 << (q->bits - 1)) - 1;
        const int qi = (int)code - L;
        return s * ((float)qi / (float)L);
    }
    case ORA_Q_POW2:
        return pow2_decode(code, q->pow2_k, q->bits);
    }
    return 0.0f;
}

int ora_has_scales(const ora_quant *q)
{
    return q->kind == ORA_Q_SIGN_L1 || q->kind == ORA_Q_UNIFORM_MAX;
}

/* Bits of one message: b per coordinate plus 32 per scale word. */
uint64_t ora_message_bits(const ora_quant *q, int64_t d)
{
    return (uint64_t)d * (uint64_t)q->bits + (ora_has_scales(q) ? 32ull * (uint64_t)q->n_groups : 0ull);
}

/*
 * Quantize u (length d) into a message: words (ora_code_words(d, bits) words, zeroed here), scales
 * (one per group when the quantizer has scales) and the decoded vector dec = Q(u).
 * gidx maps local coordinate l to its global index (NULL: identity); it only keys the Philox counter.
 */
int ora_quantize(const ora_quant *q, int64_t d, const float *u, const int64_t *gidx, uint64_t seed,
                 uint32_t id, uint32_t t, uint32_t *words, float *scales, float *dec)
{
    memset(words, 0, (size_t)ora_code_words(d, q->bits) * sizeof(uint32_t));
    if (q->kind == ORA_Q_IDENTITY) {
        for (int64_t l = 0; l < d; ++l) {
            put_code(words, l, 32, bits_from_f32(u[l]));
            dec[l] = u[l];
        }
        return 0;
    }
    if (q->kind == ORA_Q_POW2) {
        for (int64_t l = 0; l < d; ++l) {
            const uint32_t c = pow2_encode(u[l], q->pow2_k, q->pow2_K, q->bits);
            put_code(words, l, q->bits, c);
            dec[l] = pow2_decode(c, q->pow2_k, q->bits);
        }
        return 0;
    }
    for (int64_t g = 0; g < q->n_groups; ++g) {
        const int64_t a = q->offsets[g], b = q->offsets[g + 1];
        if (q->kind == ORA_Q_SIGN_L1) {
            /* scale = ||u_group||_1 / |group|: the l1 norm in binary64, one rounding to binary32 */
            double acc = 0.0;
            for (int64_t l = a; l < b; ++l) acc += fabs((double)u[l]);
            const float s = (b > a) ? (float)(acc / (double)(b - a)) : 0.0f;
            scales[g] = s;
            for (int64_t l = a; l < b; ++l) {
                const uint32_t c = (u[l] >= 0.0f) ? 1u : 0u;
                put_code(words, l, 1, c);
                dec[l] = c ? s : -s;
            }
        } else { /* Example 1: Q(x) = Q1(||x||_inf) * Q2(x / Q1(||x||_inf)), Q2 onto {i/L} */
            const int L = (1 << (q->bits - 1)) - 1;
            float s = 0.0f;
            for (int64_t l = a; l < b; ++l) {
                const float au = fabsf(u[l]);
                if (au > s) s = au;
            }
            scales[g] = s;
            for (int64_t l = a; l < b; ++l) {
                int qi = 0;
                if (s > 0.0f) {
                    const float z = u[l] / s;           /* x / Q1(||x||_inf), in [-1, 1] */
                    const float y = z * (float)L;       /* position on the grid, in [-L, L] */
                    if (q->stochastic) {
                        const float f = floorf(y);
                        const float frac = y - f;       /* exact: |y| < 2^23 */
                        const int64_t j = gidx ? gidx[l] : l;
                        const float U = ora_uniform(seed, id, t, j);
                        qi = (int)f + ((U < frac) ? 1 : 0);
                    } else {
                        qi = (int)rintf(y);             /* nearest grid point, ties to even */
                    }
                }
                const uint32_t c = (uint32_t)(qi + L);
                put_code(words, l, q->bits, c);
                dec[l] = s * ((float)qi / (float)L);
            }
        }
    }
    return 0;
}

/* Decode a whole message into dec (length d). */
void ora_decode(const ora_quant *q, int64_t d, const uint32_t *words, const float *scales, float *dec)
{
    if (!ora_has_scales(q)) {
        for (int64_t l = 0; l < d; ++l) dec[l] = decode_one(q, get_code(words, l, q->bits), 0.0f);
        return;
    }
    for (int64_t g = 0; g < q->n_groups; ++g)
        for (int64_t l = q->offsets[g]; l < q->offsets[g + 1]; ++l)
            dec[l] = decode_one(q, get_code(words, l, q->bits), scales[g]);
}

/* -------------------------------------------------------------------------------- round steps */

typedef struct {
    int64_t d;
    int32_t n;
    int32_t mode;            /* ORA_ADAM_AT_WORKER (the paper) or ORA_ADAM_AT_SERVER */
    int32_t error_feedback;  /* 1: the paper; 0: the "_err" ablation of Table 2 (residuals stay 0) */
    int32_t adam_form;       /* 0: the paper's Adam (Algorithm 2); 1: the textbook form below */
    float alpha, beta1, beta2, eps;
    uint64_t seed;
} ora_config;

/* 1 - beta^t for the 1-based round t, with beta^t formed by t binary64 multiplications and
 * rounded once to binary32. */
float ora_bias_correction(float beta, uint32_t t1)
{
    double p = 1.0;
    for (uint32_t k = 0; k < t1; ++k) p *= (double)beta;
    return (float)(1.0 - p);
}

/* One Adam moment update and step at the 1-based round t1.
 * Form 0, the paper's (Algorithm 2): v = theta v + (1-theta) g^2, m = beta m + (1-beta) g, step
 *   alpha m / sqrt(v); no bias correction, eps only as v_0.
 * Form 1, the textbook form of Kingma and Ba: the same moments from v_0 = 0, step
 *   alpha (m / (1 - beta^t)) / (sqrt(v / (1 - theta^t)) + eps). */
static float adam_step(const ora_config *c, uint32_t t1, float g, float *m, float *v)
{
    const float c1 = 1.0f - c->beta1, c2 = 1.0f - c->beta2;
    *v = c->beta2 * *v + c2 * (g * g);
    *m = c->beta1 * *m + c1 * g;
    if (c->adam_form == 0) return (c->alpha * *m) / sqrtf(*v);
    const float bc1 = ora_bias_correction(c->beta1, t1), bc2 = ora_bias_correction(c->beta2, t1);
    return (c->alpha * (*m / bc1)) / (sqrtf(*v / bc2) + c->eps);
}

/*
 * Worker i, round t (0-based): Algorithm 2's moment updates (W-mode) or the raw gradient (S-mode),
 * the residual-corrected input u, the message Q_w(u) and the new residual.  u and dec are caller
 * scratch of length d.  m and v are unused in S-mode.
 */
void ora_worker_step(const ora_config *cfg, const ora_quant *qw, const int64_t *gidx, int32_t worker,
                     uint32_t t, const float *g, float *m, float *v, float *e, float *u, float *dec,
                     uint32_t *words, float *scales)
{
    const int64_t d = cfg->d;
    for (int64_t l = 0; l < d; ++l) {
        const float step = (cfg->mode == ORA_ADAM_AT_WORKER) ? adam_step(cfg, t + 1, g[l], &m[l], &v[l]) : g[l];
        u[l] = step + e[l];
    }
    ora_quantize(qw, d, u, gidx, cfg->seed, (uint32_t)worker, t, words, scales, dec);
    if (cfg->error_feedback)
        for (int64_t l = 0; l < d; ++l) e[l] = u[l] - dec[l];
}

/*
 * The server, round t: decode the n worker messages, average them (sum in worker order, then one
 * division by n), form w = avg + e_s (W-mode) or w = alpha m/sqrt(v) + e_s after an Adam update of
 * the server moments on avg (S-mode), broadcast Q_s(w) and keep e_s = w - Q_s(w).
 * acc, w and dec are caller scratch of length d.
 */
void ora_server_step(const ora_config *cfg, const ora_quant *qw, const ora_quant *qs,
                     const int64_t *gidx, uint32_t t, const uint32_t *const *wwords,
                     const float *const *wscales, float *es, float *ms, float *vs, float *acc,
                     float *w, float *dec, uint32_t *swords, float *sscales)
{
    const int64_t d = cfg->d;
    for (int64_t l = 0; l < d; ++l) acc[l] = 0.0f;
    for (int32_t i = 0; i < cfg->n; ++i) {
        ora_decode(qw, d, wwords[i], wscales[i], dec);
        for (int64_t l = 0; l < d; ++l) acc[l] = acc[l] + dec[l];
    }
    for (int64_t l = 0; l < d; ++l) {
        const float avg = acc[l] / (float)cfg->n;
        const float step = (cfg->mode == ORA_ADAM_AT_SERVER) ? adam_step(cfg, t + 1, avg, &ms[l], &vs[l]) : avg;
        w[l] = step + es[l];
    }
    ora_quantize(qs, d, w, gidx, cfg->seed, (uint32_t)cfg->n, t, swords, sscales, dec);
    if (cfg->error_feedback)
        for (int64_t l = 0; l < d; ++l) es[l] = w[l] - dec[l];
}

/* x <- x - Q_s(w): Algorithm 1's and Algorithm 2's parameter update from the broadcast message. */
void ora_apply(const ora_quant *qs, int64_t d, const uint32_t *swords, const float *sscales, float *x,
               float *dec)
{
    ora_decode(qs, d, swords, sscales, dec);
    for (int64_t l = 0; l < d; ++l) x[l] = x[l] - dec[l];
}
