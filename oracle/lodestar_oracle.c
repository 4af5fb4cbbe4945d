/*
 * Lodestar routing hot path -- plain CPU oracle (test infrastructure only).
 *
 * This file is the checker for the CUDA path, not part of it.  Only the test
 * suite, the smoke check and the CPU-baseline leg of the benchmark load it.
 * It shares no code, header or table with the CUDA library.
 *
 * Everything here is written for obviousness, not speed: scalar loops, fp64
 * accumulation, qsort + bsearch for set membership, no blocking or fusion.
 *
 * Paper: "Lodestar" (online-learned LLM inference router).
 *   Sec. 2 (LLM inference serving): prefix reuse is strictly sequential -- a
 *          cached block helps only if all preceding blocks are cached.
 *   Sec. 2 (Gateway infrastructure): the gateway keeps a prefix index (radix
 *          tree or hash tables) and computes each instance's prefix-match ratio.
 *   Sec. 4.1 (Request-instance reward model): one shared f_theta scores each
 *          instance from [x_i || r]; route to argmax reward = argmin TTFT.
 *   Sec. 4.1 (Model architecture): MLP, ReLU, scalar output.
 *   Sec. 4.1 (Features): input length, expected KV-hit ratio, running / queued
 *          requests, inflight prefill / decode tokens, KV utilisation, GPU model.
 *   Algorithm 4: per-feature z-score normalisation, batched forward, argmax.
 *   Sec. 4.3.2 (Online learning): periodic retraining on logged
 *          (features, TTFT) records; FIFO buffer of recent samples.
 *   Sec. 4.3.1 (Fallback) and Algorithm 4: cold-start and out-of-range
 *          guards; Sec. 4.1 (Consistent hashing based filtering): the
 *          K-filter of Algorithm 4.
 *   Algorithms 1 and 2 (the comparison heuristics), which Algorithm 3
 *          pre-computes as the gateway's fallback choice.
 *   Sec. 4.3.2 (Training-data selection): FIFO + replay pool, admission of
 *          evicted samples by the diversity of their gradient embeddings.
 *
 * Readings where the paper is silent (each also listed in the design notes):
 *   - block hash: SplitMix64 finaliser based content hash, prefix state chained
 *     by a linear recurrence mod 2^64 (definition below);
 *   - hit length: stop at the first missing block, no cap at L-1;
 *   - kappa = 16h/L with kappa = 0 when L = 0; std < 1e-12 replaced by 1;
 *   - loss: mean squared error on TTFT in seconds; SGD or Adam (PyTorch
 *     defaults beta1 = 0.9, beta2 = 0.999, eps = 1e-8);
 *   - bf16 mode: weights, layer-1 input and hidden activations rounded to
 *     bf16 (round to nearest even); biases and accumulation stay wide;
 *   - argmin ties -> lowest index, -0 == +0, NaN after every number;
 *   - guards: n = records ever appended; bounds = NaN-skipping min / max over
 *     the records the ring holds; prefix group = key of the first full block;
 *     ConsistentHash_K = top-K rendezvous hashing; gpu_kv mean in fp64 (sum
 *     in index order); kappa_i |r| = 16 h_i; epsilon = 0, no random tiebreak;
 *   - heuristics: request count = queued + running columns, mean and
 *     population standard deviation in fp64, sort ties to the lowest index;
 *   - replay admission: one round per call, candidates ranked by distance to
 *     the nearest kept embedding, kept samples by distance to their nearest
 *     other kept sample, pairing while it raises diversity (or_replay_select).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_BLOCK 16
#define OR_G 0x9E3779B97F4A7C15ull /* floor(2^64 / golden ratio) */

enum { OR_F64 = 0, OR_F32 = 1, OR_BF16 = 2 };
enum { OR_SGD = 0, OR_ADAM = 1 };

/* ------------------------------------------------------------------------ */
/* block hash                                                               */
/* ------------------------------------------------------------------------ */

/* SplitMix64 output finaliser (Steele, Lea & Flood, OOPSLA 2014; Stafford's
 * "variant 13" mixer): xor-shift 30, multiply, xor-shift 27, multiply,
 * xor-shift 31. */
uint64_t or_mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

/* Content hash of one 16-token block: the 16 int32 tokens form 8 little-endian
 * 64-bit words w_j (token 2j in the low half), each word is mixed with its own
 * offset (j+1)*G, the 8 results are xor-ed and mixed once more. */
uint64_t or_block_content(const int32_t *t) {
    uint64_t acc = 0;
    for (int j = 0; j < 8; ++j) {
        uint64_t lo = (uint64_t)(uint32_t)t[2 * j];
        uint64_t hi = (uint64_t)(uint32_t)t[2 * j + 1];
        uint64_t w = lo | (hi << 32);
        acc ^= or_mix64(w + (uint64_t)(j + 1) * OR_G);
    }
    return or_mix64(acc);
}

/* Keys of the full blocks of each sequence.  Prefix state s_{-1} = G,
 * s_b = s_{b-1} * G + c_b (mod 2^64), key_b = mix64(s_b), with 0 mapped to 1
 * (0 marks an empty table slot).  key_b therefore depends on all tokens of
 * blocks 0..b, in order.  A trailing partial block gets no key.
 * keys for sequence s go to keys[key_off[s] .. key_off[s] + floor(L_s/16)). */
int or_hash_blocks(int64_t n_seq, const int32_t *tok, const int64_t *tok_off,
                   uint64_t *keys, const int64_t *key_off) {
    for (int64_t s = 0; s < n_seq; ++s) {
        int64_t L = tok_off[s + 1] - tok_off[s];
        if (L < 0) return -1;
        int64_t nb = L / OR_BLOCK;
        const int32_t *t = tok + tok_off[s];
        uint64_t state = OR_G;
        for (int64_t b = 0; b < nb; ++b) {
            state = state * OR_G + or_block_content(t + b * OR_BLOCK);
            uint64_t k = or_mix64(state);
            keys[key_off[s] + b] = k ? k : 1ull;
        }
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* prefix hit length                                                        */
/* ------------------------------------------------------------------------ */

static int cmp_u64(const void *a, const void *b) {
    uint64_t x = *(const uint64_t *)a, y = *(const uint64_t *)b;
    return (x > y) - (x < y);
}

static int contains(const uint64_t *sorted, int64_t n, uint64_t k) {
    return bsearch(&k, sorted, (size_t)n, sizeof(uint64_t), cmp_u64) != NULL;
}

/* h[r, i] = largest k <= n_r such that keys of blocks 0..k-1 of request r are
 * all in instance i's key set (scan stops at the first missing block).
 * Instance key sets are CSR lists (duplicates allowed). */
int or_prefix_hits(int64_t n_req, const uint64_t *req_keys, const int64_t *req_key_off,
                   int32_t n_inst, const uint64_t *inst_keys, const int64_t *inst_key_off,
                   int32_t *hits) {
    for (int32_t i = 0; i < n_inst; ++i) {
        int64_t n = inst_key_off[i + 1] - inst_key_off[i];
        uint64_t *set = (uint64_t *)malloc((size_t)(n > 0 ? n : 1) * sizeof(uint64_t));
        if (!set) return -1;
        memcpy(set, inst_keys + inst_key_off[i], (size_t)n * sizeof(uint64_t));
        qsort(set, (size_t)n, sizeof(uint64_t), cmp_u64);
        for (int64_t r = 0; r < n_req; ++r) {
            int64_t nb = req_key_off[r + 1] - req_key_off[r];
            int64_t b = 0;
            while (b < nb && contains(set, n, req_keys[req_key_off[r] + b])) ++b;
            hits[r * n_inst + i] = (int32_t)b;
        }
        free(set);
    }
    return 0;
}

/* The same h[r, i] against instance key sets given sorted ascending (built
 * once, as the router's snapshot tables are, outside the routing call).
 * Returns -2 if a set is not sorted. */
int or_prefix_hits_sorted(int64_t n_req, const uint64_t *req_keys, const int64_t *req_key_off,
                          int32_t n_inst, const uint64_t *sorted_keys, const int64_t *sorted_off,
                          int32_t *hits) {
    for (int32_t i = 0; i < n_inst; ++i) {
        const uint64_t *set = sorted_keys + sorted_off[i];
        int64_t n = sorted_off[i + 1] - sorted_off[i];
        for (int64_t q = 1; q < n; ++q)
            if (set[q - 1] > set[q]) return -2;
        for (int64_t r = 0; r < n_req; ++r) {
            int64_t nb = req_key_off[r + 1] - req_key_off[r];
            int64_t b = 0;
            while (b < nb && n > 0 && contains(set, n, req_keys[req_key_off[r] + b])) ++b;
            hits[r * n_inst + i] = (int32_t)b;
        }
    }
    return 0;
}

/* Same result, organised for few requests against huge instance sets: the
 * request keys are sorted once and every instance key is looked up among
 * them, marking (request block, instance) pairs that are cached. */
typedef struct { uint64_t key; int64_t pos; } or_kp;
static int cmp_kp(const void *a, const void *b) {
    uint64_t x = ((const or_kp *)a)->key, y = ((const or_kp *)b)->key;
    return (x > y) - (x < y);
}

int or_prefix_hits_by_marking(int64_t n_req, const uint64_t *req_keys, const int64_t *req_key_off,
                              int32_t n_inst, const uint64_t *inst_keys, const int64_t *inst_key_off,
                              int32_t *hits) {
    int64_t nk = req_key_off[n_req];
    or_kp *kp = (or_kp *)malloc((size_t)(nk > 0 ? nk : 1) * sizeof(or_kp));
    unsigned char *mark = (unsigned char *)malloc((size_t)(nk > 0 ? nk : 1));
    if (!kp || !mark) { free(kp); free(mark); return -1; }
    for (int64_t p = 0; p < nk; ++p) { kp[p].key = req_keys[p]; kp[p].pos = p; }
    qsort(kp, (size_t)nk, sizeof(or_kp), cmp_kp);
    for (int32_t i = 0; i < n_inst; ++i) {
        memset(mark, 0, (size_t)(nk > 0 ? nk : 1));
        for (int64_t q = inst_key_off[i]; q < inst_key_off[i + 1]; ++q) {
            /* binary search for the first entry with key >= inst key */
            uint64_t k = inst_keys[q];
            int64_t lo = 0, hi = nk;
            while (lo < hi) {
                int64_t mid = lo + (hi - lo) / 2;
                if (kp[mid].key < k) lo = mid + 1; else hi = mid;
            }
            for (int64_t p = lo; p < nk && kp[p].key == k; ++p) mark[kp[p].pos] = 1;
        }
        for (int64_t r = 0; r < n_req; ++r) {
            int64_t nb = req_key_off[r + 1] - req_key_off[r];
            int64_t b = 0;
            while (b < nb && mark[req_key_off[r] + b]) ++b;
            hits[r * n_inst + i] = (int32_t)b;
        }
    }
    free(kp);
    free(mark);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* features (Sec. 4.1 "Features"; Algorithm 4 Normalize)                    */
/* ------------------------------------------------------------------------ */

/* Raw feature row of pair (r, i): [pair(6) || instance state || request extras].
 * Pair block, all in fp32:
 *   f0 = L, f1 = h, f2 = 16h (hit tokens), f3 = kappa = 16h / L (hit ratio),
 *   f4 = L - 16h (tokens to prefill), f5 = ceil(L/16) - h (blocks to allocate). */
void or_raw_features_row(int64_t L, int32_t h, const float *inst, int d_inst,
                         const float *req, int d_req, float *x) {
    float hit_tok = (float)((int64_t)OR_BLOCK * h);
    x[0] = (float)L;
    x[1] = (float)h;
    x[2] = hit_tok;
    x[3] = L > 0 ? hit_tok / (float)L : 0.0f;
    x[4] = (float)(L - (int64_t)OR_BLOCK * h);
    x[5] = (float)((L + OR_BLOCK - 1) / OR_BLOCK - h);
    for (int k = 0; k < d_inst; ++k) x[6 + k] = inst[k];
    for (int k = 0; k < d_req; ++k) x[6 + d_inst + k] = req[k];
}

/* Per-feature z-score in fp32: (x - mean) / std, std < 1e-12 replaced by 1. */
void or_zscore(int d, const float *x, const float *mean, const float *std, float *out) {
    for (int k = 0; k < d; ++k) {
        float s = std[k] < 1e-12f ? 1.0f : std[k];
        float c = x[k] - mean[k];
        out[k] = c / s;
    }
}

/* Normalised features of all (r, i) pairs, row r*n_inst + i. */
int or_features(int64_t n_req, int32_t n_inst, const int64_t *L, const int32_t *hits,
                const float *inst, int d_inst, const float *req, int d_req,
                const float *mean, const float *std, float *out) {
    int d = 6 + d_inst + d_req;
    float *x = (float *)malloc((size_t)d * sizeof(float));
    if (!x) return -1;
    for (int64_t r = 0; r < n_req; ++r)
        for (int32_t i = 0; i < n_inst; ++i) {
            or_raw_features_row(L[r], hits[r * n_inst + i], inst + (int64_t)i * d_inst, d_inst,
                                req + r * d_req, d_req, x);
            or_zscore(d, x, mean, std, out + (r * n_inst + i) * d);
        }
    free(x);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* predictor (Sec. 4.1 "Model architecture")                                */
/* ------------------------------------------------------------------------ */

/* bf16 round-to-nearest-even of an fp32 value (NaN kept as a quiet NaN). */
float or_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) {
        u = (u | 0x00400000u) & 0xFFFF0000u;
    } else {
        u += 0x7FFFu + ((u >> 16) & 1u);
        u &= 0xFFFF0000u;
    }
    float r;
    memcpy(&r, &u, 4);
    return r;
}

/* value as stored at a rounding point of the given mode */
static double rnd(int mode, double v) {
    if (mode == OR_F64) return v;
    return (double)(float)v;
}
static double rnd_op(int mode, double v) { /* operand of a product */
    if (mode == OR_BF16) return (double)or_bf16((float)v);
    return rnd(mode, v);
}

/* parameter offsets: W_l [w[l+1], w[l]] row-major then b_l [w[l+1]] */
static int64_t param_offset(int n_layers, const int *w, int l, int bias) {
    int64_t off = 0;
    (void)n_layers;
    for (int k = 0; k < l; ++k) off += (int64_t)w[k + 1] * w[k] + w[k + 1];
    return bias ? off + (int64_t)w[l + 1] * w[l] : off;
}

int64_t or_param_count(int n_layers, const int *w) {
    return param_offset(n_layers, w, n_layers, 0);
}

/* Dropout between hidden layers (Sec. 4.1 Model architecture: dropout 0.1
 * between hidden layers; training only).  The keep decision of unit o of
 * hidden activation h (1-based layer output) for minibatch row j at optimiser
 * step t comes from a counter-based generator built on mix64:
 *   h1 = mix64(seed ^ ((t << 16) | h)),  u = mix64(h1 ^ ((j << 20) | o)),
 *   keep  <=>  (u >> 11) >= ceil(p 2^53)      (a uniform on [0, 1) >= p),
 * and kept units are scaled by s = fp32(1 / (1 - p)).  Hidden activations
 * that feed another hidden layer are dropped; the last one is not. */
typedef struct {
    uint64_t seed, thr;  /* thr = ceil(p 2^53); 0 = no dropout */
    float scale;         /* fp32 1 / (1 - p) (fp32 and bf16 modes) */
    double p;            /* the rate (fp64 mode scales by 1 / (1 - p) exactly) */
    int64_t t, j;
} or_drop;

static int drop_keep(const or_drop *dr, int h, int o) {
    uint64_t h1 = or_mix64(dr->seed ^ (((uint64_t)dr->t << 16) | (uint64_t)h));
    uint64_t u = or_mix64(h1 ^ (((uint64_t)dr->j << 20) | (uint64_t)o));
    return (u >> 11) >= dr->thr;
}

uint64_t or_drop_threshold(float p) { return (uint64_t)ceil((double)p * 9007199254740992.0); }
float or_drop_scale(float p) { return (float)(1.0 / (1.0 - (double)p)); }

/* keep decision for the pins: 1 kept, 0 dropped */
int or_drop_keep(uint64_t seed, float p, int64_t t, int h, int64_t j, int o) {
    or_drop dr = {seed, or_drop_threshold(p), or_drop_scale(p), (double)p, t, j};
    return drop_keep(&dr, h, o);
}

/* Forward pass of one row.  z_l = W_l a_{l-1} + b_l summed in fp64; a_l = relu(z_l)
 * for hidden layers; the last layer is linear.  Rounding per mode:
 *   F64 : none;  F32 : each z_l rounded to fp32;
 *   BF16: additionally W_l, a_0 = x and every hidden a_l rounded to bf16.
 * If z_save / a_save are given, z_l and a_l of every layer are stored at
 * offsets act_off[l] (the input a_0 at a_save + 0). */
static double forward_row_drop(int mode, int n_layers, const int *w, const double *params,
                               const double *x, double *z_save, double *a_save, const int64_t *act_off,
                               double *buf_a, double *buf_b, const or_drop *dr) {
    double *a = buf_a, *z = buf_b;
    for (int k = 0; k < w[0]; ++k) a[k] = rnd_op(mode, x[k]);
    if (a_save) for (int k = 0; k < w[0]; ++k) a_save[k] = a[k];
    for (int l = 0; l < n_layers; ++l) {
        const double *W = params + param_offset(n_layers, w, l, 0);
        const double *b = params + param_offset(n_layers, w, l, 1);
        for (int o = 0; o < w[l + 1]; ++o) {
            double s = 0.0;
            for (int k = 0; k < w[l]; ++k) s += rnd_op(mode, W[(int64_t)o * w[l] + k]) * a[k];
            z[o] = rnd(mode, s + rnd(mode, b[o]));
        }
        if (z_save) for (int o = 0; o < w[l + 1]; ++o) z_save[act_off[l + 1] + o] = z[o];
        if (l + 1 < n_layers) {
            int dropped = dr && dr->thr > 0 && l + 2 < n_layers;
            for (int o = 0; o < w[l + 1]; ++o) {
                double r = z[o] > 0.0 ? z[o] : 0.0;
                if (dropped) {  /* scale in the mode's working precision, then round the operand */
                    if (!drop_keep(dr, l + 1, o)) r = 0.0;
                    else r = mode == OR_F64 ? r * (1.0 / (1.0 - dr->p)) : (double)((float)r * dr->scale);
                }
                z[o] = rnd_op(mode, r);
            }
            if (a_save) for (int o = 0; o < w[l + 1]; ++o) a_save[act_off[l + 1] + o] = z[o];
        }
        double *t = a; a = z; z = t;
    }
    return a[0];
}

static double forward_row(int mode, int n_layers, const int *w, const double *params,
                          const double *x, double *z_save, double *a_save, const int64_t *act_off,
                          double *buf_a, double *buf_b) {
    return forward_row_drop(mode, n_layers, w, params, x, z_save, a_save, act_off, buf_a, buf_b, NULL);
}

static int max_width(int n_layers, const int *w) {
    int m = 1;
    for (int l = 0; l <= n_layers; ++l) m = w[l] > m ? w[l] : m;
    return m;
}

int or_mlp_forward(int mode, int n_layers, const int *w, const double *params,
                   int64_t rows, const double *x, double *y) {
    int m = max_width(n_layers, w);
    double *ba = (double *)malloc((size_t)m * sizeof(double));
    double *bb = (double *)malloc((size_t)m * sizeof(double));
    if (!ba || !bb) { free(ba); free(bb); return -1; }
    for (int64_t r = 0; r < rows; ++r)
        y[r] = forward_row(mode, n_layers, w, params, x + r * w[0], NULL, NULL, NULL, ba, bb);
    free(ba);
    free(bb);
    return 0;
}

/* Rounding analysis of the forward pass, per row, for comparing an
 * implementation that accumulates every dot product in fp32 (any order)
 * with this oracle's fp64 sums.  Not part of the method: it says how far such
 * an implementation may lie from y while computing the same definition.
 *
 *   ebound[r]: how far y_fp32acc may lie from y when every bf16 rounding
 *     point takes the same value on both sides.  The rounding error of a sum
 *     of K terms accumulated in fp32 behaves as a sum of independent errors
 *     of at most half an ulp of each partial sum; its standard deviation is
 *     below 2^-24 sqrt(K) sqrt(S2) / 2, S2 = sum_k (w_k a_k)^2 + b^2, and the
 *     radius taken is eight of those, 4 2^-24 sqrt(K + 1) sqrt(S2), plus two
 *     fp32 roundings of z (a statistical radius, not a worst-case bound: the
 *     worst case K 2^-24 sum |w_k a_k| is a hundred times larger and is never
 *     approached).  In F32 mode the radii carry through the layers, the
 *     independent errors of a layer's inputs adding in quadrature
 *     (sqrt sum_k (w_k e_k)^2; ReLU is 1-Lipschitz); in BF16 mode a
 *     hidden activation rounded to bf16 is the same bits on both sides unless
 *     its value lies within its radius of a bf16 rounding midpoint, so only
 *     the output layer's own radius remains.
 *   flip[r] (BF16): the sum over the rounding points that lie within their
 *     radius of a midpoint (an input feature within 1 fp32 ulp, the z-score's
 *     allowance; a hidden activation within its radius) of |y' - y|, y' the
 *     output with that one point rounded to the other bf16 neighbour.
 * The rows are the same as or_mlp_forward's; y is written too. */
static double bf16_other(double v, float rounded, double *dist) {
    /* the bf16 neighbour of fp32 value v that RNE did not choose, and the
     * distance of v from the midpoint between the two */
    float f = (float)v;
    uint32_t u;
    memcpy(&u, &f, 4);
    uint32_t lo_u = u & 0xFFFF0000u;
    float lo, hi;
    memcpy(&lo, &lo_u, 4);
    uint32_t hi_u = lo_u + 0x10000u;
    memcpy(&hi, &hi_u, 4);
    double mid = 0.5 * ((double)lo + (double)hi);
    *dist = fabs(v - mid);
    return rounded == lo ? (double)hi : (double)lo;
}

static double forward_from(int n_layers, const int *w, const double *params, int l0, const double *a_in,
                           double *buf_a, double *buf_b) {
    /* BF16 forward of layers l0.. from the layer-l0 input a_in (already bf16 values) */
    double *a = buf_a, *z = buf_b;
    for (int k = 0; k < w[l0]; ++k) a[k] = a_in[k];
    for (int l = l0; l < n_layers; ++l) {
        const double *W = params + param_offset(n_layers, w, l, 0);
        const double *b = params + param_offset(n_layers, w, l, 1);
        for (int o = 0; o < w[l + 1]; ++o) {
            double s = 0.0;
            for (int k = 0; k < w[l]; ++k) s += rnd_op(OR_BF16, W[(int64_t)o * w[l] + k]) * a[k];
            z[o] = rnd(OR_BF16, s + rnd(OR_BF16, b[o]));
        }
        if (l + 1 < n_layers)
            for (int o = 0; o < w[l + 1]; ++o) z[o] = rnd_op(OR_BF16, z[o] > 0.0 ? z[o] : 0.0);
        double *t = a; a = z; z = t;
    }
    return a[0];
}

int or_mlp_forward_bounds(int mode, int n_layers, const int *w, const double *params, int64_t rows,
                          const double *x, double *y, double *ebound, double *flip) {
    int m = max_width(n_layers, w);
    int64_t tot = 0;
    for (int l = 0; l <= n_layers; ++l) tot += w[l];
    double *act = (double *)malloc((size_t)tot * sizeof(double));     /* a_l per layer (as stored) */
    double *err = (double *)malloc((size_t)tot * sizeof(double));     /* F32: bound on a_l */
    double *alt = (double *)malloc((size_t)m * sizeof(double));
    double *ba = (double *)malloc((size_t)m * sizeof(double));
    double *bb = (double *)malloc((size_t)m * sizeof(double));
    int64_t *off = (int64_t *)malloc((size_t)(n_layers + 2) * sizeof(int64_t));
    if (!act || !err || !alt || !ba || !bb || !off) {
        free(act); free(err); free(alt); free(ba); free(bb); free(off);
        return -1;
    }
    off[0] = 0;
    for (int l = 0; l <= n_layers; ++l) off[l + 1] = off[l] + w[l];
    const double u = ldexp(1.0, -24);
    for (int64_t r = 0; r < rows; ++r) {
        const double *xr = x + r * w[0];
        double fl = 0.0, eb = 0.0;
        for (int k = 0; k < w[0]; ++k) {
            act[k] = rnd_op(mode, xr[k]);
            err[k] = 0.0;
        }
        int flips_n = 0;
        /* flip candidates of the input: within 1 fp32 ulp of a bf16 midpoint */
        double yv = 0.0;
        for (int l = 0; l < n_layers; ++l) {
            const double *W = params + param_offset(n_layers, w, l, 0);
            const double *b = params + param_offset(n_layers, w, l, 1);
            const double *a = act + off[l];
            const double *ea = err + off[l];
            double *an = act + off[l + 1];
            double *en = err + off[l + 1];
            const double gK = 4.0 * sqrt((double)w[l] + 1.0) * u;
            for (int o = 0; o < w[l + 1]; ++o) {
                double s = 0.0, s2 = 0.0, prop = 0.0;
                for (int k = 0; k < w[l]; ++k) {
                    double wk = rnd_op(mode, W[(int64_t)o * w[l] + k]);
                    s += wk * a[k];
                    s2 += (wk * a[k]) * (wk * a[k]);
                    prop += (wk * ea[k]) * (wk * ea[k]);
                }
                double bo = rnd(mode, b[o]);
                double z = rnd(mode, s + bo);
                double ez = gK * sqrt(s2 + bo * bo) + 2.0 * u * fabs(z) + (mode == OR_F32 ? sqrt(prop) : 0.0);
                if (l + 1 == n_layers) {
                    an[o] = z;
                    en[o] = ez + 2.0 * u * fabs(z);
                } else {
                    double rl = z > 0.0 ? z : 0.0;
                    an[o] = rnd_op(mode, rl);
                    en[o] = mode == OR_F32 ? ez : 0.0;
                }
            }
        }
        yv = act[off[n_layers]];
        eb = err[off[n_layers]];
        if (mode == OR_BF16) {
            /* rounding points near a midpoint: inputs (1 fp32 ulp), hidden (their bound) */
            for (int l = 0; l < n_layers; ++l) {
                for (int o = 0; o < w[l]; ++o) {
                    double pre, rad;
                    if (l == 0) {
                        pre = xr[o];
                        rad = ldexp(fabs(pre), -23);
                    } else {
                        /* recompute the pre-rounding value and its bound */
                        const double *W = params + param_offset(n_layers, w, l - 1, 0);
                        const double *b = params + param_offset(n_layers, w, l - 1, 1);
                        const double *a = act + off[l - 1];
                        double s = 0.0, s2 = 0.0;
                        for (int k = 0; k < w[l - 1]; ++k) {
                            double wk = rnd_op(OR_BF16, W[(int64_t)o * w[l - 1] + k]);
                            s += wk * a[k];
                            s2 += (wk * a[k]) * (wk * a[k]);
                        }
                        double bo = rnd(OR_BF16, b[o]);
                        double z = rnd(OR_BF16, s + bo);
                        pre = z > 0.0 ? z : 0.0;
                        rad = 4.0 * sqrt((double)w[l - 1] + 1.0) * u * sqrt(s2 + bo * bo) + 2.0 * u * fabs(z);
                        if (pre == 0.0) continue;  /* relu clamps: both sides give 0 or a value within rad */
                    }
                    double dist;
                    double other = bf16_other(pre, (float)act[off[l] + o], &dist);
                    if (dist > rad) continue;
                    for (int k = 0; k < w[l]; ++k) alt[k] = act[off[l] + k];
                    alt[o] = other;
                    double y2 = forward_from(n_layers, w, params, l, alt, ba, bb);
                    fl += fabs(y2 - yv);
                    ++flips_n;
                }
            }
        }
        (void)flips_n;
        y[r] = yv;
        ebound[r] = eb;
        if (flip) flip[r] = fl;
    }
    free(act); free(err); free(alt); free(ba); free(bb); free(off);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* greedy selection (Sec. 4.1; Algorithm 4 argmax of reward = -TTFT)        */
/* ------------------------------------------------------------------------ */

/* (a, i) precedes (b, j) in the lexicographic order (score, index), where NaN
 * comes after every number and -0 equals +0. */
static int precedes(float a, int32_t i, float b, int32_t j) {
    int an = isnan(a), bn = isnan(b);
    if (an != bn) return bn;          /* the number precedes the NaN */
    if (!an && a != b) return a < b;  /* -0 == +0 compares equal here */
    return i < j;
}

/* (a, i) before (b, j) in the order of or_argmin, for fp64 values. */
static int precedes_d(double a, int32_t i, double b, int32_t j) {
    if (isnan(a)) return isnan(b) && i < j;
    if (isnan(b)) return 1;
    return a < b || (a == b && i < j);
}

int or_argmin(int64_t n_req, int32_t n_inst, const float *scores, int32_t *choice, float *best) {
    for (int64_t r = 0; r < n_req; ++r) {
        int32_t c = 0;
        for (int32_t i = 1; i < n_inst; ++i)
            if (precedes(scores[r * n_inst + i], i, scores[r * n_inst + c], c)) c = i;
        choice[r] = n_inst > 0 ? c : -1;
        best[r] = n_inst > 0 ? scores[r * n_inst + c] : NAN;
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* sample ring (Sec. 4.3.2: recent records, oldest evicted on overflow)     */
/* ------------------------------------------------------------------------ */

/* Record j of the batch goes to slot (count + j) mod capacity. */
int or_ring_append(int64_t capacity, int d, float *ring_x, float *ring_y, int64_t count,
                   int64_t n, const float *x, const float *y) {
    for (int64_t j = 0; j < n; ++j) {
        int64_t slot = (count + j) % capacity;
        memcpy(ring_x + slot * d, x + j * d, (size_t)d * sizeof(float));
        ring_y[slot] = y[j];
    }
    return 0;
}

/* ------------------------------------------------------------------------ */
/* online training step (Sec. 4.3.2; loss and optimiser are readings)       */
/* ------------------------------------------------------------------------ */

/* One minibatch step.  Rows idx[j] of the ring are z-scored (fp32), run forward
 * (activations kept), the loss L = mean_j (yhat_j - y_j)^2 is formed and
 * back-propagated:
 *   dZ_L = 2 (yhat - y) / B
 *   for l = L..1:  G = dZ_l (rounded to bf16 in BF16 mode)
 *                  dW_l = G^T A_{l-1},  db_l = column sums of dZ_l (unrounded)
 *                  dA_{l-1} = G W_l (W_l rounded to bf16 in BF16 mode)
 *                  dZ_{l-1} = dA_{l-1} * [z_{l-1} > 0]
 * (every quantity rounded to fp32 when formed, except in F64 mode), then
 *   SGD : theta -= lr g
 *   Adam: m = b1 m + (1-b1) g; v = b2 v + (1-b2) g^2;
 *         theta -= lr (m / (1-b1^t)) / (sqrt(v / (1-b2^t)) + eps)
 * with t the 1-based step number.  params / m / v are updated in place; the
 * gradient is written to grad_out if given, the loss to *loss_out. */
int or_train_step(int mode, int n_layers, const int *w, double *params, double *adam_m,
                  double *adam_v, int64_t t, int opt, double lr, int batch,
                  const float *ring_x, const float *ring_y, const int32_t *idx,
                  const float *mean, const float *std, double *loss_out, double *grad_out,
                  float drop_p, uint64_t drop_seed) {
    const double b1 = 0.9, b2 = 0.999, eps = 1e-8;
    int d = w[0];
    int64_t P = or_param_count(n_layers, w);
    int64_t act_off[17];
    act_off[0] = 0;
    for (int l = 0; l < n_layers; ++l) act_off[l + 1] = act_off[l] + w[l];
    int64_t act_row = act_off[n_layers] + 1;  /* a_0..a_{L-1} plus the output */
    int m = max_width(n_layers, w);
    double *Z = (double *)calloc((size_t)batch * act_row, sizeof(double));
    double *A = (double *)calloc((size_t)batch * act_row, sizeof(double));
    double *g = (double *)calloc((size_t)P, sizeof(double));
    double *dz = (double *)calloc((size_t)batch * m, sizeof(double));
    double *dz_prev = (double *)calloc((size_t)batch * m, sizeof(double));
    double *ba = (double *)malloc((size_t)m * sizeof(double));
    double *bb = (double *)malloc((size_t)m * sizeof(double));
    double *xr = (double *)malloc((size_t)d * sizeof(double));
    float *xf = (float *)malloc((size_t)d * sizeof(float));
    double *yhat = (double *)malloc((size_t)(batch > 0 ? batch : 1) * sizeof(double));
    if (!Z || !A || !g || !dz || !dz_prev || !ba || !bb || !xr || !xf || !yhat) return -1;
    or_drop dr = {drop_seed, drop_p > 0.0f ? or_drop_threshold(drop_p) : 0, or_drop_scale(drop_p),
                  (double)drop_p, t, 0};

    /* forward */
    double loss = 0.0;
    for (int j = 0; j < batch; ++j) {
        or_zscore(d, ring_x + (int64_t)idx[j] * d, mean, std, xf);
        for (int k = 0; k < d; ++k) xr[k] = (double)xf[k];
        dr.j = j;
        yhat[j] = forward_row_drop(mode, n_layers, w, params, xr, Z + (int64_t)j * act_row,
                                   A + (int64_t)j * act_row, act_off, ba, bb, &dr);
        double e = yhat[j] - (double)ring_y[idx[j]];
        loss += e * e;
    }
    loss /= (double)batch;
    if (loss_out) *loss_out = loss;

    /* backward (the output layer has width 1) */
    for (int j = 0; j < batch; ++j)
        dz[(int64_t)j * m] = rnd(mode, 2.0 * (yhat[j] - (double)ring_y[idx[j]]) / (double)batch);
    for (int l = n_layers - 1; l >= 0; --l) {
        int fi = w[l], fo = w[l + 1];
        double *gW = g + param_offset(n_layers, w, l, 0);
        double *gb = g + param_offset(n_layers, w, l, 1);
        const double *W = params + param_offset(n_layers, w, l, 0);
        for (int o = 0; o < fo; ++o) {
            double sb = 0.0;
            for (int j = 0; j < batch; ++j) sb += dz[(int64_t)j * m + o];
            gb[o] = rnd(mode, sb);
            for (int k = 0; k < fi; ++k) {
                double s = 0.0;
                for (int j = 0; j < batch; ++j)
                    s += rnd_op(mode, dz[(int64_t)j * m + o]) * A[(int64_t)j * act_row + act_off[l] + k];
                gW[(int64_t)o * fi + k] = rnd(mode, s);
            }
        }
        if (l > 0) {
            /* input a_l is hidden activation h = l; it was dropped when it feeds
             * another hidden layer (l < n_layers - 1) */
            int dropped = dr.thr > 0 && l < n_layers - 1;
            for (int j = 0; j < batch; ++j) {
                dr.j = j;
                for (int k = 0; k < fi; ++k) {
                    double s = 0.0;
                    for (int o = 0; o < fo; ++o)
                        s += rnd_op(mode, dz[(int64_t)j * m + o]) * rnd_op(mode, W[(int64_t)o * fi + k]);
                    double zprev = Z[(int64_t)j * act_row + act_off[l] + k];
                    double v = zprev > 0.0 ? rnd(mode, s) : 0.0;
                    if (dropped && v != 0.0)
                        v = !drop_keep(&dr, l, k) ? 0.0
                            : (mode == OR_F64 ? v * (1.0 / (1.0 - dr.p)) : (double)((float)v * dr.scale));
                    dz_prev[(int64_t)j * m + k] = v;
                }
            }
            double *tmp = dz; dz = dz_prev; dz_prev = tmp;
        }
    }
    if (grad_out) memcpy(grad_out, g, (size_t)P * sizeof(double));

    /* update */
    if (opt == OR_SGD) {
        for (int64_t p = 0; p < P; ++p) params[p] = rnd(mode, params[p] - lr * g[p]);
    } else {
        double bc1 = 1.0 - pow(b1, (double)t), bc2 = 1.0 - pow(b2, (double)t);
        for (int64_t p = 0; p < P; ++p) {
            adam_m[p] = rnd(mode, b1 * adam_m[p] + (1.0 - b1) * g[p]);
            adam_v[p] = rnd(mode, b2 * adam_v[p] + (1.0 - b2) * g[p] * g[p]);
            double mh = adam_m[p] / bc1, vh = adam_v[p] / bc2;
            params[p] = rnd(mode, params[p] - lr * mh / (sqrt(vh) + eps));
        }
    }
    free(Z); free(A); free(g); free(dz); free(dz_prev);
    free(ba); free(bb); free(xr); free(xf); free(yhat);
    return 0;
}

/* Loss only (forward over the minibatch), for finite-difference checks. */
int or_loss(int mode, int n_layers, const int *w, const double *params, int batch,
            const float *ring_x, const float *ring_y, const int32_t *idx,
            const float *mean, const float *std, double *loss_out) {
    int d = w[0], m = max_width(n_layers, w);
    double *ba = (double *)malloc((size_t)m * sizeof(double));
    double *bb = (double *)malloc((size_t)m * sizeof(double));
    double *xr = (double *)malloc((size_t)d * sizeof(double));
    float *xf = (float *)malloc((size_t)d * sizeof(float));
    if (!ba || !bb || !xr || !xf) return -1;
    double loss = 0.0;
    for (int j = 0; j < batch; ++j) {
        or_zscore(d, ring_x + (int64_t)idx[j] * d, mean, std, xf);
        for (int k = 0; k < d; ++k) xr[k] = (double)xf[k];
        double e = forward_row(mode, n_layers, w, params, xr, NULL, NULL, NULL, ba, bb)
                   - (double)ring_y[idx[j]];
        loss += e * e;
    }
    *loss_out = loss / (double)batch;
    free(ba); free(bb); free(xr); free(xf);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Algorithm 4 guards (Sec. 4.3.1 fallback; Sec. 4.1 consistent hashing)    */
/* ------------------------------------------------------------------------ */

/* Feature bounds [l_j, u_j] of the training buffer (Algorithm 4 input; the
 * fallback paragraph of Sec. 4.3.1: the ranges observed in the buffer).  The
 * buffer is the sample ring: its first min(count, capacity) slots hold the
 * records it keeps.  l_j / u_j = smallest / largest value of column j over
 * those rows, NaN values skipped; a column with no number keeps the empty
 * range l = +inf, u = -inf. */
int or_ring_bounds(int64_t capacity, int d, const float *ring_x, int64_t count,
                   float *lo, float *hi) {
    int64_t rows = count < capacity ? count : capacity;
    for (int j = 0; j < d; ++j) {
        lo[j] = INFINITY;
        hi[j] = -INFINITY;
    }
    for (int64_t r = 0; r < rows; ++r)
        for (int j = 0; j < d; ++j) {
            float v = ring_x[r * d + j];
            if (isnan(v)) continue;
            if (v < lo[j]) lo[j] = v;
            if (v > hi[j]) hi[j] = v;
        }
    return 0;
}

/* Rendezvous weight of instance i for prefix-group key g. */
static uint64_t hrw_weight(uint64_t g, int32_t i) {
    return or_mix64(g ^ or_mix64((uint64_t)(i + 1) * OR_G));
}

/* (w_a, a) ranks before (w_b, b): larger weight first, then lower index. */
static int hrw_before(uint64_t wa, int32_t a, uint64_t wb, int32_t b) {
    if (wa != wb) return wa > wb;
    return a < b;
}

/* ConsistentHash_K (Algorithm 4; Sec. 4.1 "Consistent hashing based
 * filtering"): the K instances with the largest rendezvous weights for key g
 * (highest-random-weight hashing), in rank order.  Writes min(K, n_inst)
 * indices to cand and returns that count.  Selection sort: pass k takes the
 * best instance not yet taken. */
int32_t or_hrw_candidates(uint64_t g, int32_t n_inst, int32_t K, int32_t *cand) {
    int32_t m = K < n_inst ? K : n_inst;
    for (int32_t k = 0; k < m; ++k) {
        int32_t b = -1;
        for (int32_t i = 0; i < n_inst; ++i) {
            int taken = 0;
            for (int32_t q = 0; q < k; ++q) taken |= cand[q] == i;
            if (taken) continue;
            if (b < 0 || hrw_before(hrw_weight(g, i), i, hrw_weight(g, b), b)) b = i;
        }
        cand[k] = b;
    }
    return m < 0 ? 0 : m;
}

/* Guarded selection of Algorithm 4, given the predicted TTFT of every pair.
 *   status 1 (cold start): n < n_min                       -> choice -1, best NaN
 *   status 2 (OOD)       : ood_on and some raw feature of some pair of the
 *                          request lies outside [lo, hi] (NaN counts as
 *                          outside)                         -> choice -1, best NaN
 *   otherwise status 0 and choice = argmin over instances (= argmax of the
 *   reward -TTFT; order of or_argmin), then the K-filter: when K >= 1, the
 *   prompt has a full block (its group key gkey[r] is the key of block 0),
 *     mean_i inst[i, kv_col] > tau_sat   (the mean in fp64: the sum in index
 *                                         order, divided by N) and
 *     max_i 16 h_i > tau_ben             (kappa_i |r| = 16 h_i hit tokens),
 *   status gains bit 4 and a choice outside the candidates is replaced by the
 *   argmin over the candidates.  best = scores of the final choice.
 * Cold start is tested before OOD (Algorithm 4 order).  Exploration and the
 * random tiebreak are not taken (epsilon = 0; equal scores go to the lowest
 * index). */
int or_guards(int64_t n_req, int32_t n_inst, const int64_t *L, const uint64_t *gkey,
              const int32_t *hits, const float *inst, int d_inst, const float *req, int d_req,
              const float *scores, const float *lo, const float *hi, int64_t n, int64_t n_min,
              int ood_on, int32_t K, int32_t kv_col, float tau_sat, float tau_ben,
              int32_t *choice, float *best, int32_t *status) {
    int d = 6 + d_inst + d_req;
    float *x = (float *)malloc((size_t)d * sizeof(float));
    int32_t *cand = (int32_t *)malloc((size_t)(K > 0 ? K : 1) * sizeof(int32_t));
    if (!x || !cand) { free(x); free(cand); return -1; }
    double kv_sum = 0.0;
    if (K >= 1 && kv_col >= 0 && kv_col < d_inst)
        for (int32_t i = 0; i < n_inst; ++i) kv_sum += (double)inst[(int64_t)i * d_inst + kv_col];
    const double kv_mean = kv_sum / (double)n_inst;
    for (int64_t r = 0; r < n_req; ++r) {
        const float *sr = scores + r * n_inst;
        const int32_t *hr = hits + r * n_inst;
        if (n < n_min) {
            choice[r] = -1; best[r] = NAN; status[r] = 1;
            continue;
        }
        if (ood_on) {
            int out = 0;
            for (int32_t i = 0; i < n_inst && !out; ++i) {
                or_raw_features_row(L[r], hr[i], inst + (int64_t)i * d_inst, d_inst,
                                    req + r * d_req, d_req, x);
                for (int j = 0; j < d; ++j)
                    if (!(x[j] >= lo[j] && x[j] <= hi[j])) { out = 1; break; }
            }
            if (out) {
                choice[r] = -1; best[r] = NAN; status[r] = 2;
                continue;
            }
        }
        int32_t c = 0;
        for (int32_t i = 1; i < n_inst; ++i)
            if (precedes(sr[i], i, sr[c], c)) c = i;
        int32_t st = 0;
        if (K >= 1 && L[r] >= OR_BLOCK && kv_col >= 0 && kv_col < d_inst) {
            int32_t hmax = 0;
            for (int32_t i = 0; i < n_inst; ++i) if (hr[i] > hmax) hmax = hr[i];
            if (kv_mean > (double)tau_sat && 16.0 * (double)hmax > (double)tau_ben) {
                int32_t m = or_hrw_candidates(gkey[r], n_inst, K, cand);
                int in = 0;
                for (int32_t q = 0; q < m; ++q) in |= cand[q] == c;
                if (!in) {
                    c = cand[0];
                    for (int32_t q = 1; q < m; ++q)
                        if (precedes(sr[cand[q]], cand[q], sr[c], c)) c = cand[q];
                }
                st = 4;
            }
        }
        choice[r] = c; best[r] = sr[c]; status[r] = st;
    }
    free(x); free(cand);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* fallback heuristics (Algorithms 1 and 2; Algorithm 3 pre-computes one)   */
/* ------------------------------------------------------------------------ */

/* The heuristic choice of every request.  Inputs per instance: the request
 * count c_i = inst[i, c_col0] (+ inst[i, c_col1] when c_col1 >= 0), in fp64,
 * and per pair the prefix match ratio m_i = kappa = 16 h / L (fp32 as the
 * feature is, 0 when L = 0).
 *   mode 1, Algorithm 1 (prefix-cache and load aware):
 *     if c_max - c_min > theta_imbal (fp64): argmin_i c_i;
 *     else mu = mean c, sigma = population standard deviation (fp64: sums in
 *     index order, two passes, sqrt correctly rounded), and among the
 *     instances with c_i <= mu + k sigma (fp64) the first in the order
 *     (m desc, c asc, index asc); none: argmin_i c_i.
 *   mode 2, Algorithm 2 (prefix aware, threshold tau): i* = argmax m_i
 *     (ties to the lowest index); i* if m_{i*} > tau, else argmin_i c_i.
 * argmin_i c_i takes the lowest index among equal counts, NaN after every
 * number; c_min / c_max skip NaN counts. */
int or_heuristic(int64_t n_req, int32_t n_inst, const int64_t *L, const int32_t *hits,
                 const float *inst, int d_inst, int mode, int c_col0, int c_col1,
                 float theta_imbal, float k_over, float tau, int32_t *out) {
    double *c = (double *)malloc((size_t)n_inst * sizeof(double));
    float *m = (float *)malloc((size_t)n_inst * sizeof(float));
    if (!c || !m) { free(c); free(m); return -1; }
    for (int32_t i = 0; i < n_inst; ++i) {
        c[i] = (double)inst[(int64_t)i * d_inst + c_col0];
        if (c_col1 >= 0) c[i] = c[i] + (double)inst[(int64_t)i * d_inst + c_col1];
    }
    int32_t least = 0;
    double cmin = INFINITY, cmax = -INFINITY;      /* NaN counts skipped here */
    for (int32_t i = 0; i < n_inst; ++i) {
        if (precedes_d(c[i], i, c[least], least)) least = i;  /* NaN after numbers */
        if (c[i] < cmin) cmin = c[i];
        if (c[i] > cmax) cmax = c[i];
    }
    double mu = 0.0, var = 0.0;
    for (int32_t i = 0; i < n_inst; ++i) mu += c[i];
    mu = mu / (double)n_inst;
    for (int32_t i = 0; i < n_inst; ++i) {
        double dv = c[i] - mu;
        var += dv * dv;
    }
    var = var / (double)n_inst;
    double thr = mu + (double)k_over * sqrt(var);
    int imbalanced = cmax - cmin > (double)theta_imbal;
    for (int64_t r = 0; r < n_req; ++r) {
        const int32_t *hr = hits + r * n_inst;
        for (int32_t i = 0; i < n_inst; ++i) {
            float ht = (float)((int64_t)OR_BLOCK * hr[i]);
            m[i] = L[r] > 0 ? ht / (float)L[r] : 0.0f;
        }
        int32_t pick = least;
        if (mode == 1 && !imbalanced) {
            int32_t b = -1;
            for (int32_t i = 0; i < n_inst; ++i) {
                if (!(c[i] <= thr)) continue;
                if (b < 0 || m[i] > m[b] || (m[i] == m[b] && c[i] < c[b])) b = i;
            }
            if (b >= 0) pick = b;
        } else if (mode == 2) {
            int32_t b = 0;
            for (int32_t i = 1; i < n_inst; ++i) if (m[i] > m[b]) b = i;
            if (m[b] > tau) pick = b;
        }
        out[r] = pick;
    }
    free(c); free(m);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* two-pool training data (Sec. 4.3.2 Training-data selection)              */
/* ------------------------------------------------------------------------ */

/* Gradient embedding of logged records: each raw row is z-scored (fp32) and
 * run forward (rounding per mode); with a the last hidden activation (the
 * output layer's input, width H = w[n_layers - 1]) and yhat the prediction,
 * g = (yhat - y) a, the per-record gradient of the squared error with respect
 * to the output layer's weights up to the factor 2 ("last-hidden-layer
 * activations, weighted by prediction residual").  g is [M, H]. */
int or_replay_embed(int mode, int n_layers, const int *w, const double *params, int64_t M,
                    const float *x, const float *y, const float *mean, const float *std, double *g) {
    int d = w[0], m = max_width(n_layers, w), H = w[n_layers - 1];
    int64_t act_off[17];
    act_off[0] = 0;
    for (int l = 0; l < n_layers; ++l) act_off[l + 1] = act_off[l] + w[l];
    double *ba = (double *)malloc((size_t)m * sizeof(double));
    double *bb = (double *)malloc((size_t)m * sizeof(double));
    double *xr = (double *)malloc((size_t)d * sizeof(double));
    double *acts = (double *)malloc((size_t)act_off[n_layers] * sizeof(double));
    float *xf = (float *)malloc((size_t)d * sizeof(float));
    if (!ba || !bb || !xr || !acts || !xf) {
        free(ba); free(bb); free(xr); free(acts); free(xf);
        return -1;
    }
    for (int64_t s = 0; s < M; ++s) {
        or_zscore(d, x + s * d, mean, std, xf);
        for (int k = 0; k < d; ++k) xr[k] = (double)xf[k];
        double yhat = forward_row(mode, n_layers, w, params, xr, NULL, acts, act_off, ba, bb);
        double res = yhat - (double)y[s];
        for (int k = 0; k < H; ++k) g[s * H + k] = res * acts[act_off[n_layers - 1] + k];
    }
    free(ba); free(bb); free(xr); free(acts); free(xf);
    return 0;
}

/* Squared Euclidean distances between embeddings, written out:
 *   dcand[e] = min_j ||gc_e - gk_j||^2 over the nk kept embeddings (+inf if none);
 *   nkept[j] = min_{k != j} ||gk_j - gk_k||^2 (+inf if there is no other). */
int or_replay_distances(int64_t mc, const double *gc, int64_t nk, const double *gk, int H,
                        double *dcand, double *nkept) {
    for (int64_t e = 0; e < mc; ++e) {
        double best = INFINITY;
        for (int64_t j = 0; j < nk; ++j) {
            double s = 0.0;
            for (int k = 0; k < H; ++k) {
                double t = gc[e * H + k] - gk[j * H + k];
                s += t * t;
            }
            if (s < best) best = s;
        }
        dcand[e] = best;
    }
    for (int64_t j = 0; j < nk; ++j) {
        double best = INFINITY;
        for (int64_t q = 0; q < nk; ++q) {
            if (q == j) continue;
            double s = 0.0;
            for (int k = 0; k < H; ++k) {
                double t = gk[j * H + k] - gk[q * H + k];
                s += t * t;
            }
            if (s < best) best = s;
        }
        nkept[j] = best;
    }
    return 0;
}

/* key for ranking: NaN counts as -inf (no diversity) */
static double div_key(double v) { return isnan(v) ? -INFINITY : v; }

/* One admission round of the replay pool (reading of the two-pool design:
 * evicted samples are admitted when they are the most diverse with respect
 * to those kept).  Candidates are ranked by (dcand desc, index asc), kept
 * samples by (nkept asc, slot asc); free = cap - nk.  The candidate of rank
 * t < free fills slot nk + t; the candidate of rank free + q replaces the
 * kept sample of rank q when its dcand exceeds that sample's nkept (both
 * sequences are monotone, so the replacements are a prefix).
 * src[s] for the new pool's slots s < *new_count: c >= 0 = candidate c,
 * -1 - j = kept sample j stays. */
int or_replay_select(int64_t mc, const double *dcand, int64_t nk, const double *nkept, int64_t cap,
                     int64_t *src, int64_t *new_count) {
    int64_t *oc = (int64_t *)malloc((size_t)(mc > 0 ? mc : 1) * sizeof(int64_t));
    int64_t *ok = (int64_t *)malloc((size_t)(nk > 0 ? nk : 1) * sizeof(int64_t));
    if (!oc || !ok) { free(oc); free(ok); return -1; }
    /* rank by counting: rank_e = #{e' ranked before e} */
    for (int64_t e = 0; e < mc; ++e) {
        int64_t r = 0;
        for (int64_t f = 0; f < mc; ++f) {
            double a = div_key(dcand[f]), b = div_key(dcand[e]);
            if (a > b || (a == b && f < e)) ++r;
        }
        oc[r] = e;
    }
    for (int64_t j = 0; j < nk; ++j) {
        int64_t r = 0;
        for (int64_t q = 0; q < nk; ++q) {
            double a = div_key(nkept[q]), b = div_key(nkept[j]);
            if (a < b || (a == b && q < j)) ++r;
        }
        ok[r] = j;
    }
    for (int64_t s = 0; s < nk; ++s) src[s] = -1 - s;
    int64_t free_slots = cap - nk, t = 0;
    for (; t < mc && t < free_slots; ++t) src[nk + t] = oc[t];
    int64_t count = nk + t;
    for (int64_t q = 0; t + q < mc && q < nk; ++q) {
        int64_t c = oc[t + q], j = ok[q];
        if (!(div_key(dcand[c]) > div_key(nkept[j]))) break;
        src[j] = c;
    }
    *new_count = count;
    free(oc); free(ok);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* sequential-commit routing (Sec. 4.2 cluster snapshot manager and prefix  */
/* KV-cache tracker; Sec. 4.3.1 P1: requests are routed one at a time)      */
/* ------------------------------------------------------------------------ */

/* Requests r = 0, 1, ... in order.  Request r is routed as or_argmin routes
 * it -- hit lengths against each instance's current key set, features from
 * the current instance rows, the predictor (rounding per mode), the lowest
 * (score, index) -- and the decision is committed before request r + 1:
 * inst[c, q_col] += 1 (fp32; q_col < 0: no queue update) and every full-block
 * key of prompt r joins instance c's key set.  c is the oracle's own choice,
 * or forced[r] when forced is given (to replay another implementation's
 * decisions and check each step).  inst is updated in place.  Outputs per
 * request: hits [n_req, n_inst], scores [n_req, n_inst] (fp32 of the fp64
 * forward), choice [n_req] (the oracle's own argmin). */
typedef struct { uint64_t *k; int64_t n, cap; } or_keyset;

static int keyset_has(const or_keyset *s, uint64_t key) {
    return s->n > 0 && contains(s->k, s->n, key);
}

int or_route_sequential(int mode, int n_layers, const int *w, const double *params, int64_t n_req,
                        const int64_t *L, const uint64_t *req_keys, const int64_t *req_key_off,
                        int32_t n_inst, const uint64_t *inst_keys, const int64_t *inst_key_off,
                        float *inst, int d_inst, const float *req, int d_req, const float *mean,
                        const float *std, int32_t q_col, const int32_t *forced,
                        int32_t *hits, float *scores, int32_t *choice) {
    int d = 6 + d_inst + d_req, mw = max_width(n_layers, w);
    or_keyset *base = (or_keyset *)calloc((size_t)n_inst, sizeof(or_keyset));
    or_keyset *add = (or_keyset *)calloc((size_t)n_inst, sizeof(or_keyset));
    float *xf = (float *)malloc((size_t)d * sizeof(float));
    float *xz = (float *)malloc((size_t)d * sizeof(float));
    double *xd = (double *)malloc((size_t)d * sizeof(double));
    double *ba = (double *)malloc((size_t)mw * sizeof(double));
    double *bb = (double *)malloc((size_t)mw * sizeof(double));
    int rc = 0;
    if (!base || !add || !xf || !xz || !xd || !ba || !bb) { rc = -1; goto done; }
    for (int32_t i = 0; i < n_inst; ++i) {
        int64_t n = inst_key_off[i + 1] - inst_key_off[i];
        base[i].k = (uint64_t *)malloc((size_t)(n > 0 ? n : 1) * sizeof(uint64_t));
        if (!base[i].k) { rc = -1; goto done; }
        memcpy(base[i].k, inst_keys + inst_key_off[i], (size_t)n * sizeof(uint64_t));
        qsort(base[i].k, (size_t)n, sizeof(uint64_t), cmp_u64);
        base[i].n = n;
    }
    for (int64_t r = 0; r < n_req; ++r) {
        const uint64_t *rk = req_keys + req_key_off[r];
        int64_t nb = req_key_off[r + 1] - req_key_off[r];
        int32_t c = 0;
        for (int32_t i = 0; i < n_inst; ++i) {
            int64_t b = 0;
            while (b < nb && (keyset_has(&base[i], rk[b]) || keyset_has(&add[i], rk[b]))) ++b;
            hits[r * n_inst + i] = (int32_t)b;
            or_raw_features_row(L[r], (int32_t)b, inst + (int64_t)i * d_inst, d_inst, req + r * d_req, d_req, xf);
            or_zscore(d, xf, mean, std, xz);
            for (int k = 0; k < d; ++k) xd[k] = (double)xz[k];
            float y = (float)forward_row(mode, n_layers, w, params, xd, NULL, NULL, NULL, ba, bb);
            scores[r * n_inst + i] = y;
            if (i > 0 && precedes(y, i, scores[r * n_inst + c], c)) c = i;
        }
        choice[r] = c;
        int32_t cc = forced ? forced[r] : c;
        if (cc < 0 || cc >= n_inst) continue;
        if (q_col >= 0) inst[(int64_t)cc * d_inst + q_col] = inst[(int64_t)cc * d_inst + q_col] + 1.0f;
        or_keyset *s = &add[cc];
        if (s->n + nb > s->cap) {
            int64_t ncap = (s->n + nb) * 2 + 16;
            uint64_t *nk = (uint64_t *)realloc(s->k, (size_t)ncap * sizeof(uint64_t));
            if (!nk) { rc = -1; goto done; }
            s->k = nk;
            s->cap = ncap;
        }
        memcpy(s->k + s->n, rk, (size_t)nb * sizeof(uint64_t));
        s->n += nb;
        qsort(s->k, (size_t)s->n, sizeof(uint64_t), cmp_u64);
    }
done:
    if (base) for (int32_t i = 0; i < n_inst; ++i) free(base[i].k);
    if (add) for (int32_t i = 0; i < n_inst; ++i) free(add[i].k);
    free(base); free(add); free(xf); free(xz); free(xd); free(ba); free(bb);
    return rc;
}
