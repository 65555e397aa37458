/*
 * ts_oracle.c -- plain fp64 CPU oracle for the dReLU activation-sparse FFN.
 *
 * TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and the
 * CPU-baseline leg of bench.py may load or call this file. The CUDA library
 * shares no code, header, table or helper with it, and neither side includes
 * or imports the other.
 *
 * What it computes (Turbo Sparse, arXiv 2406.05955):
 *   Gated-MLP block, Eq. 1 (Sec. 2):
 *       Gate(x) = F(x W_gate),  Up(x) = x W_up,
 *       Combined(x) = Gate(x) * Up(x),  out = Combined(x) W_down
 *   dReLU, Eq. 2 (Sec. 3.2), no biases (footnote to Eq. 2):
 *       Combined(x) = max(0, x W_gate) * max(0, x W_up)
 *   Activation sparsity (Sec. 6.2): a neuron counts as active when its
 *   activation is non-zero, i.e. here when g_j > 0 and u_j > 0.
 *   Predictor-driven computation (Sec. 7): only the neurons a predictor lists
 *   are computed; unlisted neurons contribute nothing.
 *   MoE (Sec. 4, Sec. 6.2): a router picks the top-k experts per token and
 *   the token's output is the softmax-weighted sum of those experts' FFNs.
 *
 * Storage is neuron-major, [m][d] row-major for all three matrices: row j of
 * W_gate and W_up is column j of the paper's d x m matrices (neuron j's input
 * weights); row j of W_down is row j of the paper's m x d W_down. Hence
 *     g_j = sum_i W_gate[j][i] x_i,   u_j = sum_i W_up[j][i] x_i,
 *     y_i = sum_j max(0,g_j) max(0,u_j) W_down[j][i].
 *
 * Every sum runs in double, in ascending index order, one output per thread,
 * with fused multiply-add disabled at build time (-ffp-contract=off), so the
 * result is bit-identical on every host and for every thread count.
 * Inputs are the stored values themselves: fp32, or bf16 bit patterns (the
 * upper 16 bits of an IEEE binary32), decoded exactly to double. Weights may
 * also be stored as INT4 groups (the weight-only 4-bit storage of the paper's
 * Mixtral-47B-INT4 rows, Tables 7-9): per neuron row of d weights, d/2 bytes
 * of 4-bit codes followed by d/32 IEEE binary16 scales, one per group of 32
 * consecutive elements; the weight is scale * (code - 8), decoded exactly to
 * double. A group's 16 code bytes are four little-endian 32-bit words;
 * element e = 8s + 2t + h (s, t in 0..3, h in 0..1) of the group is the
 * nibble s + 4h of word t.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { ORACLE_F32 = 0, ORACLE_BF16 = 1, ORACLE_INT4 = 2 };

/* Exact IEEE binary16 -> double (by the bit definition). */
static double half_to_double(uint16_t h) {
    const int sgn = h >> 15, e = (h >> 10) & 31, f = h & 1023;
    double v;
    if (e == 0)
        v = ldexp((double)f, -24); /* subnormal: f * 2^-24 */
    else if (e == 31)
        v = f ? NAN : INFINITY;
    else
        v = ldexp((double)(f + 1024), e - 25); /* (1 + f/1024) * 2^(e-15) */
    return sgn ? -v : v;
}

/* Bytes of one INT4 row of d weights. */
static size_t int4_row_bytes(int d) { return (size_t)d / 2 + (size_t)(d / 32) * 2; }

/* Weight (j, i) of a [m][d] matrix stored as wdtype. */
static double welem(const void* base, int wdtype, int d, int j, int i) {
    if (wdtype != ORACLE_INT4) {
        const size_t idx = (size_t)j * (size_t)d + (size_t)i;
        if (wdtype == ORACLE_F32) return (double)((const float*)base)[idx];
        uint32_t bits = (uint32_t)((const uint16_t*)base)[idx] << 16;
        float f;
        memcpy(&f, &bits, sizeof f);
        return (double)f;
    }
    const uint8_t* row = (const uint8_t*)base + (size_t)j * int4_row_bytes(d);
    const int e = i % 32, s = e / 8, t = (e % 8) / 2, hh = e % 2;
    const int nib = s + 4 * hh; /* nibble of word t */
    const uint8_t byte = row[(size_t)(i / 32) * 16 + 4 * t + nib / 2];
    const int code = (byte >> (4 * (nib % 2))) & 15;
    const uint8_t* sp = row + d / 2 + (size_t)(i / 32) * 2;
    const uint16_t h = (uint16_t)(sp[0] | (sp[1] << 8)); /* little-endian */
    return half_to_double(h) * (double)(code - 8);
}

/* Exact decode of one stored element to double. */
static double elem(const void* base, int dtype, size_t idx) {
    if (dtype == ORACLE_F32) return (double)((const float*)base)[idx];
    uint32_t bits = (uint32_t)((const uint16_t*)base)[idx] << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

static double relu(double v) { return v > 0.0 ? v : 0.0; }

static void set_threads(int n_threads) {
#ifdef _OPENMP
    if (n_threads > 0) omp_set_num_threads(n_threads);
#else
    (void)n_threads;
#endif
}

/* Number of threads the next parallel region will use (1 without OpenMP). */
int ts_oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/*
 * Dense definition of the dReLU Gated-MLP (Eq. 1 with Eq. 2) for B tokens.
 *
 *   x        [B][d]  activations (dtype: fp32 or bf16)
 *   w_gate   [m][d]  w_up [m][d]  w_down [m][d]  (wdtype: fp32, bf16, or
 *            INT4 rows of d/2 code bytes + d/32 binary16 scales)
 *   rows     NULL: every neuron 0..m-1 takes part.
 *            else: the n_rows listed neurons only (Sec. 7 predictor mode);
 *            the list must be strictly ascending and inside [0, m).
 *   g, u     [B][m]  out: pre-activations of the neurons that take part,
 *            0 for the others
 *   gate_mask[B][m]  out: 1 iff the neuron takes part and g > 0
 *   both_mask[B][m]  out: 1 iff the neuron takes part, g > 0 and u > 0
 *   y        [B][d]  out: sum over every neuron that takes part (ascending
 *            j, zero activations included) of Combined_j * W_down[j][:]
 *
 * Returns 0, or -1 if an argument is invalid (nothing is written then).
 */
int ts_oracle_ffn_w(int d, int m, int B, int dtype, const void* x, int wdtype, const void* w_gate,
                    const void* w_up, const void* w_down, const int32_t* rows, int n_rows,
                    double* g, double* u, uint8_t* gate_mask, uint8_t* both_mask, double* y,
                    int n_threads) {
    if (d <= 0 || m <= 0 || B < 0 || (dtype != ORACLE_F32 && dtype != ORACLE_BF16)) return -1;
    if (wdtype != ORACLE_F32 && wdtype != ORACLE_BF16 && wdtype != ORACLE_INT4) return -1;
    if (wdtype == ORACLE_INT4 && d % 32 != 0) return -1;
    if (rows != NULL) {
        if (n_rows < 0 || n_rows > m) return -1;
        for (int p = 0; p < n_rows; ++p) {
            if (rows[p] < 0 || rows[p] >= m) return -1;
            if (p > 0 && rows[p] <= rows[p - 1]) return -1;
        }
    }
    set_threads(n_threads);
    /* part[j] = 1 iff neuron j takes part in the sum */
    uint8_t* part = (uint8_t*)calloc((size_t)m, 1);
    double* c = (double*)malloc(sizeof(double) * (size_t)m);
    if (!part || !c) {
        free(part);
        free(c);
        return -1;
    }
    if (rows == NULL) {
        memset(part, 1, (size_t)m);
    } else {
        for (int p = 0; p < n_rows; ++p) part[rows[p]] = 1;
    }

    for (int b = 0; b < B; ++b) {
        const size_t xo = (size_t)b * (size_t)d;
        double* gb = g + (size_t)b * (size_t)m;
        double* ub = u + (size_t)b * (size_t)m;
        uint8_t* gm = gate_mask + (size_t)b * (size_t)m;
        uint8_t* bm = both_mask + (size_t)b * (size_t)m;

        /* Gate(x) and Up(x): one dot product per neuron, i ascending. */
#pragma omp parallel for schedule(static)
        for (int j = 0; j < m; ++j) {
            double gj = 0.0, uj = 0.0;
            if (part[j]) {
                for (int i = 0; i < d; ++i) {
                    double xi = elem(x, dtype, xo + (size_t)i);
                    gj += welem(w_gate, wdtype, d, j, i) * xi;
                    uj += welem(w_up, wdtype, d, j, i) * xi;
                }
            }
            gb[j] = gj;
            ub[j] = uj;
            gm[j] = (uint8_t)(part[j] && gj > 0.0);
            bm[j] = (uint8_t)(part[j] && gj > 0.0 && uj > 0.0);
            /* Eq. 2: Combined = max(0, g) * max(0, u) */
            c[j] = part[j] ? relu(gj) * relu(uj) : 0.0;
        }

        /* out = Combined W_down = sum over j ascending of Combined_j * W_down[j][:];
           every output element starts at 0 and adds its terms in j order. */
        double* yb = y + (size_t)b * (size_t)d;
        for (int i = 0; i < d; ++i) yb[i] = 0.0;
#pragma omp parallel
        for (int j = 0; j < m; ++j) {
            if (!part[j]) continue;
#pragma omp for schedule(static)
            for (int i = 0; i < d; ++i)
                yb[i] += c[j] * welem(w_down, wdtype, d, j, i);
        }
    }
    free(part);
    free(c);
    return 0;
}

/* As ts_oracle_ffn_w with weights stored like the activations. */
int ts_oracle_ffn(int d, int m, int B, int dtype, const void* x, const void* w_gate,
                  const void* w_up, const void* w_down, const int32_t* rows, int n_rows,
                  double* g, double* u, uint8_t* gate_mask, uint8_t* both_mask, double* y,
                  int n_threads) {
    return ts_oracle_ffn_w(d, m, B, dtype, x, dtype, w_gate, w_up, w_down, rows, n_rows, g, u,
                           gate_mask, both_mask, y, n_threads);
}

/*
 * Top-k magnitude mask (Eq. 3 and Eq. 4, Sec. 5): per token, Mask keeps the
 * `keep` neurons with the largest |Combined| (Combined = max(0, g) max(0, u),
 * Eq. 2), a lower neuron index winning a tie, and the output is
 * (Combined * Mask) W_down.
 *
 *   x, w_gate, w_up, w_down, dtypes: as ts_oracle_ffn_w (no row list)
 *   keep          neurons kept per token, 0 <= keep <= m
 *   g, u [B][m]   out: the pre-activations (as ts_oracle_ffn_w)
 *   sel  [B][m]   out: 1 iff the neuron is among the kept ones
 *   y    [B][d]   out: sum over the kept neurons (ascending j) of
 *                 Combined_j * W_down[j][:]
 *
 * The selection sorts all m neurons by (|Combined| descending, index
 * ascending) and keeps the first `keep`. Returns 0, or -1 on invalid arguments.
 */
static const double* g_sort_key;
static int by_magnitude_then_index(const void* pa, const void* pb) {
    const int a = *(const int*)pa, b = *(const int*)pb;
    const double ka = fabs(g_sort_key[a]), kb = fabs(g_sort_key[b]);
    if (ka > kb) return -1;
    if (ka < kb) return 1;
    return a < b ? -1 : (a > b ? 1 : 0);
}

static const double* g_sort_key_signed;
static int by_value_then_index(const void* pa, const void* pb) {
    const int a = *(const int*)pa, b = *(const int*)pb;
    const double ka = g_sort_key_signed[a], kb = g_sort_key_signed[b];
    if (ka > kb) return -1;
    if (ka < kb) return 1;
    return a < b ? -1 : (a > b ? 1 : 0);
}

int ts_oracle_ffn_topk(int d, int m, int B, int dtype, const void* x, int wdtype, const void* w_gate,
                       const void* w_up, const void* w_down, int keep, double* g, double* u, uint8_t* sel,
                       double* y, int n_threads) {
    if (keep < 0 || keep > m || B < 0) return -1;
    uint8_t* gm = (uint8_t*)malloc((size_t)B * (size_t)m + 1);
    uint8_t* bm = (uint8_t*)malloc((size_t)B * (size_t)m + 1);
    double* c = (double*)malloc(sizeof(double) * (size_t)m);
    int* order = (int*)malloc(sizeof(int) * (size_t)m);
    if (!gm || !bm || !c || !order) {
        free(gm);
        free(bm);
        free(c);
        free(order);
        return -1;
    }
    /* g and u of every neuron (the plain FFN's y is overwritten below) */
    int rc = ts_oracle_ffn_w(d, m, B, dtype, x, wdtype, w_gate, w_up, w_down, NULL, 0, g, u, gm, bm, y,
                             n_threads);
    for (int b = 0; rc == 0 && b < B; ++b) {
        const double* gb = g + (size_t)b * (size_t)m;
        const double* ub = u + (size_t)b * (size_t)m;
        uint8_t* sb = sel + (size_t)b * (size_t)m;
        for (int j = 0; j < m; ++j) {
            c[j] = relu(gb[j]) * relu(ub[j]); /* Eq. 2 */
            order[j] = j;
            sb[j] = 0;
        }
        g_sort_key = c;
        qsort(order, (size_t)m, sizeof(int), by_magnitude_then_index);
        for (int q = 0; q < keep; ++q) sb[order[q]] = 1; /* Eq. 3 */
        /* Eq. 4: (Combined * Mask) W_down, j ascending */
        double* yb = y + (size_t)b * (size_t)d;
        for (int i = 0; i < d; ++i) yb[i] = 0.0;
        for (int j = 0; j < m; ++j) {
            if (!sb[j]) continue;
#pragma omp parallel for schedule(static)
            for (int i = 0; i < d; ++i) yb[i] += c[j] * welem(w_down, wdtype, d, j, i);
        }
    }
    free(gm);
    free(bm);
    free(c);
    free(order);
    return rc;
}

/*
 * Activation predictor (Sec. 7 names a predictor per FFN block without its
 * architecture; reading: a two-layer ReLU MLP of rank r that outputs, for a
 * batch, the list of the K neurons it rates most likely to be active):
 *   h_t   = max(0, W1 x_t)                 W1 [r][d], h_t [r]
 *   s_t,j = sum_i W2[j][i] h_t,i           W2 [m][r]
 *   key_j = max over the batch's tokens of s_t,j
 * The K neurons with the largest key (a lower index winning a tie) are the
 * list, in ascending neuron order.
 *
 *   x [B][d] (dtype), w1 [r][d], w2 [m][r] (wdtype = dtype); K: 0 <= K <= m
 *   scores [B][m] out: s;  list [K] out: ascending neuron ids
 * Returns 0, or -1 on invalid arguments.
 */
int ts_oracle_predict(int d, int r, int m, int B, int dtype, const void* x, const void* w1, const void* w2,
                      int K, double* scores, int32_t* list) {
    if (d <= 0 || r <= 0 || m <= 0 || B <= 0 || K < 0 || K > m) return -1;
    if (dtype != ORACLE_F32 && dtype != ORACLE_BF16) return -1;
    double* h = (double*)malloc(sizeof(double) * (size_t)r);
    double* key = (double*)malloc(sizeof(double) * (size_t)m);
    int* order = (int*)malloc(sizeof(int) * (size_t)m);
    uint8_t* pick = (uint8_t*)calloc((size_t)m, 1);
    if (!h || !key || !order || !pick) {
        free(h);
        free(key);
        free(order);
        free(pick);
        return -1;
    }
    for (int b = 0; b < B; ++b) {
        for (int i = 0; i < r; ++i) {
            double v = 0.0;
            for (int k = 0; k < d; ++k)
                v += elem(w1, dtype, (size_t)i * (size_t)d + (size_t)k) * elem(x, dtype, (size_t)b * (size_t)d + (size_t)k);
            h[i] = relu(v);
        }
        double* sb = scores + (size_t)b * (size_t)m;
#pragma omp parallel for schedule(static)
        for (int j = 0; j < m; ++j) {
            double v = 0.0;
            for (int i = 0; i < r; ++i) v += elem(w2, dtype, (size_t)j * (size_t)r + (size_t)i) * h[i];
            sb[j] = v;
        }
    }
    for (int j = 0; j < m; ++j) {
        double kj = scores[j];
        for (int b = 1; b < B; ++b) {
            const double v = scores[(size_t)b * (size_t)m + (size_t)j];
            if (v > kj) kj = v;
        }
        key[j] = kj;
        order[j] = j;
    }
    g_sort_key_signed = key;
    qsort(order, (size_t)m, sizeof(int), by_value_then_index);
    for (int q = 0; q < K; ++q) pick[order[q]] = 1;
    int n = 0;
    for (int j = 0; j < m; ++j)
        if (pick[j]) list[n++] = j;
    free(h);
    free(key);
    free(order);
    free(pick);
    return 0;
}

/*
 * Router of a top-k MoE layer (Sec. 4; Mixtral routes each token to 2 of 8
 * experts, Sec. 6.2): logits r_e = sum_i W_r[e][i] x_i; the k experts with
 * the largest logits are chosen, a lower expert index winning a tie; their
 * weights are the softmax over the k chosen logits.
 *
 *   x [B][d], w_r [E][d] (dtype);  logits [B][E], sel [B][k] (experts in
 *   selection order: largest logit first), w [B][k].
 * Returns 0, or -1 on invalid arguments.
 */
int ts_oracle_router(int d, int E, int B, int dtype, const void* x, const void* w_r, int k,
                     double* logits, int32_t* sel, double* w) {
    if (d <= 0 || E <= 0 || B < 0 || k <= 0 || k > E) return -1;
    if (dtype != ORACLE_F32 && dtype != ORACLE_BF16) return -1;
    for (int b = 0; b < B; ++b) {
        double* lb = logits + (size_t)b * (size_t)E;
        for (int e = 0; e < E; ++e) {
            double acc = 0.0;
            for (int i = 0; i < d; ++i)
                acc += elem(w_r, dtype, (size_t)e * (size_t)d + (size_t)i) *
                       elem(x, dtype, (size_t)b * (size_t)d + (size_t)i);
            lb[e] = acc;
        }
        /* repeated arg-max over the experts not yet taken; strict '>' keeps
           the lower index on a tie */
        int32_t* sb = sel + (size_t)b * (size_t)k;
        for (int t = 0; t < k; ++t) {
            int best = -1;
            for (int e = 0; e < E; ++e) {
                int taken = 0;
                for (int q = 0; q < t; ++q) taken |= (sb[q] == e);
                if (taken) continue;
                if (best < 0 || lb[e] > lb[best]) best = e;
            }
            sb[t] = best;
        }
        /* softmax over the chosen logits (the first one is the largest) */
        double* wb = w + (size_t)b * (size_t)k;
        double z = 0.0;
        for (int t = 0; t < k; ++t) z += exp(lb[sb[t]] - lb[sb[0]]);
        for (int t = 0; t < k; ++t) wb[t] = exp(lb[sb[t]] - lb[sb[0]]) / z;
    }
    return 0;
}

/* Round-to-nearest-even of a binary32 to bfloat16 (the upper 16 bits),
   by the definition: add half of the dropped range, plus one if the kept
   part is odd, then truncate. NaN stays a quiet NaN. */
static uint16_t bf16_rne(float f) {
    uint32_t bits;
    memcpy(&bits, &f, sizeof bits);
    if ((bits & 0x7fffffffu) > 0x7f800000u) return (uint16_t)((bits >> 16) | 0x0040u);
    uint32_t keep_odd = (bits >> 16) & 1u;
    bits += 0x7fffu + keep_odd;
    return (uint16_t)(bits >> 16);
}

/*
 * Glue between the layers of the synthetic FFN stack (no counterpart in the
 * paper, which leaves the rest of the transformer block out of the FFN
 * problem): x = round(h / sqrt(mean(h^2) + eps)) with x[d-1] = 1 (the bias
 * channel). The quotient is taken in double, rounded to binary32, and for
 * out_dtype bf16 rounded again to bfloat16 from that binary32 value -- the
 * precision the CUDA path makes the same decision in.
 *   h [B][d] fp32;  x_out [B][d] float or bf16 bits.
 */
int ts_oracle_rmsnorm(int d, int B, const float* h, double eps, int out_dtype, void* x_out) {
    if (d <= 0 || B < 0 || (out_dtype != ORACLE_F32 && out_dtype != ORACLE_BF16)) return -1;
    for (int b = 0; b < B; ++b) {
        const float* hb = h + (size_t)b * (size_t)d;
        double ss = 0.0;
        for (int i = 0; i < d; ++i) ss += (double)hb[i] * (double)hb[i];
        double rms = sqrt(ss / (double)d + eps);
        for (int i = 0; i < d; ++i) {
            float v = (i == d - 1) ? 1.0f : (float)((double)hb[i] / rms);
            if (out_dtype == ORACLE_F32)
                ((float*)x_out)[(size_t)b * (size_t)d + (size_t)i] = v;
            else
                ((uint16_t*)x_out)[(size_t)b * (size_t)d + (size_t)i] = bf16_rne(v);
        }
    }
    return 0;
}
