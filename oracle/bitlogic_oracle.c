/*
 * CPU oracle for the LUT-network hot path of BitLogic (arXiv 2602.07400).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test-suite, the smoke check of the
 * entry module and the CPU-baseline leg of the benchmark may load this
 * library.  The product path (the CUDA library under the package) shares no
 * code with it and never calls it.
 *
 * Every function is the plain definition written out as nested loops, in
 * double precision, with no blocking, fusion or reordering.  The loops over
 * independent outputs carry OpenMP pragmas; each output is still computed by
 * exactly one thread, in the order written, so the result does not depend on
 * the thread count.
 *
 * Layouts (shared with the CUDA path by convention only):
 *   raw inputs       x[s*d + j]            uint8, sample-major
 *   soft activations X[row*B + s]          feature-major, batch contiguous
 *   connectivity     conn[j*k + i]         slot i of node j
 *   table logits     theta[j*2^k + a]      fp32 (the model's parameters)
 *   hard tables      table[j] bit a        entry a of node j
 *   packed bits      xp[row*W + s/32] bit (s%32), W = ceil(N/32)
 *
 * Index convention (the paper leaves the LUT input bit order open, App. C.1
 * "Bit-packed inference"): connectivity slot i is bit i of the table index a.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* Linear thermometer thresholds: b equispaced levels at i/(b+1) of the value
 * range (§3 "Encoders and heads"; App. A "Scope of the prior-method
 * reproduction" places them at i/(b+1)).  On uint8 pixels the real threshold
 * is 256*i/(b+1); a strict comparison p > 256*i/(b+1) equals p > floor(...).
 * The paper states no integer thresholds; the tests pin this reading to the
 * threshold sets the workloads state ({64, 128, 192} for b = 3, multiples of
 * 32 for b = 7, of 16 for b = 15). */
void oracle_linear_thresholds(int32_t b, int32_t* thr) {
    for (int32_t i = 1; i <= b; ++i) thr[i - 1] = (int32_t)((256 * i) / (b + 1));
}

/* Thermometer encoder E: R^d -> {0,1}^{db} (§3 "Encoders and heads"):
 * wire j*b + i is 1 when feature j exceeds threshold i (strict, as in the
 * "(pixel > 0)" comparison of App. B "MNIST-specific encoder collapse"). */
void oracle_encode_thermometer(const uint8_t* x, int64_t B, int32_t d,
                               const uint8_t* thr, int32_t b, double* bits) {
    for (int32_t j = 0; j < d; ++j)
        for (int32_t i = 0; i < b; ++i)
            for (int64_t s = 0; s < B; ++s)
                bits[((int64_t)j * b + i) * B + s] = (x[s * d + j] > thr[i]) ? 1.0 : 0.0;
}

static int cmp_u8(const void* a, const void* b) {
    return (int)*(const uint8_t*)a - (int)*(const uint8_t*)b;
}

/* Distributive (quantile) thermometer fit (§3 "Encoders and heads"; App. A
 * "Initialization": fit once from the empirical pixel quantiles of the
 * training split; App. B "MNIST-specific encoder collapse": quantiles of the
 * globally flattened pixel distribution).  Reading: threshold i (1..b) is
 * the quantile at level i/(b+1) with linear interpolation between order
 * statistics, h = (n-1) i/(b+1), q = v[floor h] + (h - floor h)(v[floor h + 1]
 * - v[floor h]) over the sorted pixels v; on integer pixels the encoder's
 * strict compare pixel > q equals pixel > floor(q), so the stored threshold
 * is floor(q), here in exact integer arithmetic.  n >= 1. */
void oracle_quantile_thresholds(const uint8_t* x, int64_t n, int32_t b, uint8_t* thr) {
    uint8_t* v = (uint8_t*)malloc((size_t)n);
    memcpy(v, x, (size_t)n);
    qsort(v, (size_t)n, 1, cmp_u8);
    for (int32_t i = 1; i <= b; ++i) {
        const int64_t num = (n - 1) * (int64_t)i;      /* h = num / (b + 1) */
        const int64_t lo = num / (b + 1), rem = num % (b + 1);
        const int64_t step = lo + 1 < n ? (int64_t)v[lo + 1] - (int64_t)v[lo] : 0;
        thr[i - 1] = (uint8_t)((int64_t)v[lo] + (rem * step) / (b + 1));
    }
    free(v);
}

static double sigmoid(double z) { return 1.0 / (1.0 + exp(-z)); }

/* Corner weight of table entry a for node inputs xs[0..k-1]:
 * w_a = prod_i x_i^{a_i} (1 - x_i)^{1 - a_i} (the Kronecker-indicator basis of
 * LightLUT, §2 "Gradient-based LUT methods"; 2^k parameters per node). */
static double corner_weight(const double* xs, int32_t k, int64_t a) {
    double wa = 1.0;
    for (int32_t i = 0; i < k; ++i) wa *= ((a >> i) & 1) ? xs[i] : (1.0 - xs[i]);
    return wa;
}

/* Value of table entry theta for the two LightLUT node forms of the node
 * sweep (§2 "Gradient-based LUT methods", §4 "Node parameterization"):
 * node 0 (soft) uses t = sigmoid(theta); node 1 (straight-through hard) uses
 * the hard sample t = [theta > 0] -- the value the entry discretizes to --
 * while the gradient still reaches theta through the sigmoid (see the
 * backward).  theta = 0 samples 0, as in the table discretization below. */
static double table_value(float theta, int32_t node) {
    if (node == 1) return theta > 0.0f ? 1.0 : 0.0;
    return sigmoid((double)theta);
}

/* LUT layer forward (one logic layer L_M(f_theta^(n)) of Eq. (1), §3):
 * y_j(s) = sum_a t(theta_j[a]) * w_a(x_{M_j(0)}(s), ..., x_{M_j(k-1)}(s)),
 * t the node form's table value (table_value). */
void oracle_lut_forward(const double* X, int32_t w_in, int64_t B,
                        const int32_t* conn, const float* theta, int32_t w, int32_t k,
                        int32_t node, double* Y) {
    const int64_t K = (int64_t)1 << k;
    (void)w_in;
#pragma omp parallel for schedule(dynamic, 16)
    for (int32_t j = 0; j < w; ++j) {
        double xs[8], t[64];
        for (int64_t a = 0; a < K; ++a) t[a] = table_value(theta[(int64_t)j * K + a], node);
        for (int64_t s = 0; s < B; ++s) {
            for (int32_t i = 0; i < k; ++i) xs[i] = X[(int64_t)conn[(int64_t)j * k + i] * B + s];
            double y = 0.0;
            for (int64_t a = 0; a < K; ++a) y += t[a] * corner_weight(xs, k, a);
            Y[(int64_t)j * B + s] = y;
        }
    }
}

/* Group-sum head with temperature and cross-entropy (§3 "Encoders and
 * heads": popcount GroupSum; §4 "Training": cross-entropy on the raw head
 * logits, mean over the batch).  Class c owns the contiguous nodes
 * [c*g, (c+1)*g), g = w/C, and logit[s][c] = (sum of its outputs)/tau.
 * Gradients: dlogit = (softmax - onehot)/B, dY[j][s] = dlogit[s][c(j)]/tau.
 * logits and dY may be NULL. */
void oracle_head_loss(const double* Y, int32_t w, int64_t B, int32_t C, double tau,
                      const int32_t* labels, double* logits, double* loss, double* dY) {
    const int32_t g = w / C;
    double* lg = (double*)malloc(sizeof(double) * (size_t)B * C);
    double* per = (double*)malloc(sizeof(double) * (size_t)B);
#pragma omp parallel for schedule(static)
    for (int64_t s = 0; s < B; ++s) {
        for (int32_t c = 0; c < C; ++c) {
            double sum = 0.0;
            for (int32_t j = c * g; j < (c + 1) * g; ++j) sum += Y[(int64_t)j * B + s];
            lg[s * C + c] = sum / tau;
        }
        double m = lg[s * C];
        for (int32_t c = 1; c < C; ++c) if (lg[s * C + c] > m) m = lg[s * C + c];
        double z = 0.0;
        for (int32_t c = 0; c < C; ++c) z += exp(lg[s * C + c] - m);
        const double lse = m + log(z);
        per[s] = lse - lg[s * C + labels[s]];
        if (dY) {
            for (int32_t c = 0; c < C; ++c) {
                const double p = exp(lg[s * C + c] - lse);
                const double dl = (p - (c == labels[s] ? 1.0 : 0.0)) / (double)B;
                for (int32_t j = c * g; j < (c + 1) * g; ++j) dY[(int64_t)j * B + s] = dl / tau;
            }
        }
    }
    double tot = 0.0;
    for (int64_t s = 0; s < B; ++s) tot += per[s];
    if (loss) *loss = tot / (double)B;
    if (logits) memcpy(logits, lg, sizeof(double) * (size_t)B * C);
    free(lg);
    free(per);
}

/* LUT layer backward, by the chain rule on the forward definition, with
 * sg_a = sigmoid(theta_j[a]) and t_a the node form's table value:
 *   dtheta_j[a] = sg_a (1 - sg_a) * sum_s dY[j][s] * w_a(x(s))
 *   dy_j/dx_i   = sum_a t_a * (a_i ? +1 : -1) * prod_{m != i} (a_m ? x_m : 1 - x_m)
 *   dX[M_j(i)][s] += dY[j][s] * dy_j/dx_i        (scatter-add in node order)
 * For the soft node t_a = sg_a and this is the exact gradient.  For the
 * straight-through node the forward used t_a = [theta > 0]; the estimator
 * passes dL/dt_a = sum_s dY w_a to theta as if t_a were sigmoid(theta), and
 * the input gradient is the exact one of the hard-table forward.
 * dX (optional) is overwritten.  For each element of dX the additions happen
 * in increasing (j, i) order. */
void oracle_lut_backward(const double* X, int32_t w_in, int64_t B,
                         const int32_t* conn, const float* theta, int32_t w, int32_t k,
                         int32_t node, const double* dY, double* dtheta, double* dX) {
    const int64_t K = (int64_t)1 << k;
#pragma omp parallel for schedule(dynamic, 16)
    for (int32_t j = 0; j < w; ++j) {
        double xs[8];
        for (int64_t a = 0; a < K; ++a) {
            const double t = sigmoid((double)theta[(int64_t)j * K + a]);
            double acc = 0.0;
            for (int64_t s = 0; s < B; ++s) {
                for (int32_t i = 0; i < k; ++i) xs[i] = X[(int64_t)conn[(int64_t)j * k + i] * B + s];
                acc += dY[(int64_t)j * B + s] * corner_weight(xs, k, a);
            }
            dtheta[(int64_t)j * K + a] = t * (1.0 - t) * acc;
        }
    }
    if (!dX) return;
    memset(dX, 0, sizeof(double) * (size_t)w_in * (size_t)B);
    double* tt = (double*)malloc(sizeof(double) * (size_t)w * (size_t)K);
    for (int64_t q = 0; q < (int64_t)w * K; ++q) tt[q] = table_value(theta[q], node);
    /* samples are independent: one thread owns each sample column and walks
     * the nodes in order, so the per-element addition order is (j, i) */
#pragma omp parallel for schedule(static)
    for (int64_t s = 0; s < B; ++s) {
        double xs[8];
        for (int32_t j = 0; j < w; ++j) {
            for (int32_t i = 0; i < k; ++i) xs[i] = X[(int64_t)conn[(int64_t)j * k + i] * B + s];
            const double g = dY[(int64_t)j * B + s];
            for (int32_t i = 0; i < k; ++i) {
                double der = 0.0;
                for (int64_t a = 0; a < K; ++a) {
                    double p = ((a >> i) & 1) ? 1.0 : -1.0;
                    for (int32_t m = 0; m < k; ++m)
                        if (m != i) p *= ((a >> m) & 1) ? xs[m] : (1.0 - xs[m]);
                    der += tt[(int64_t)j * K + a] * p;
                }
                dX[(int64_t)conn[(int64_t)j * k + i] * B + s] += g * der;
            }
        }
    }
    free(tt);
}

/* Learnable routing (§3, the paragraph on connectivity: a per-slot
 * candidate pool, a selection that is differentiable in training
 * and snapped to a sparse mapping at discretization; App. A
 * "Initialization": pools drawn uniformly, routing logits zero so the
 * expected selection is uniform).  Slot e (e = j*k + i, n_slots = w*k) has
 * candidates cand[e*Kc + m] and logits r[e*Kc + m], m < Kc; its input is the
 * expected selection
 *   p_e = softmax(r_e),  Xr[e][s] = sum_m p_e[m] X[cand[e][m]][s].
 * prob (optional) receives p. */
void oracle_route_forward(const double* X, int32_t w_in, int64_t B, const int32_t* cand,
                          const float* r, int64_t n_slots, int32_t Kc, double* Xr, double* prob) {
    (void)w_in;
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t e = 0; e < n_slots; ++e) {
        double p[64], mx = -INFINITY, z = 0.0;
        for (int32_t m = 0; m < Kc; ++m) if ((double)r[e * Kc + m] > mx) mx = (double)r[e * Kc + m];
        for (int32_t m = 0; m < Kc; ++m) z += exp((double)r[e * Kc + m] - mx);
        for (int32_t m = 0; m < Kc; ++m) p[m] = exp((double)r[e * Kc + m] - mx) / z;
        if (prob) for (int32_t m = 0; m < Kc; ++m) prob[e * Kc + m] = p[m];
        for (int64_t s = 0; s < B; ++s) {
            double v = 0.0;
            for (int32_t m = 0; m < Kc; ++m) v += p[m] * X[(int64_t)cand[e * Kc + m] * B + s];
            Xr[e * B + s] = v;
        }
    }
}

/* Routing backward by the chain rule, G[e][s] = dL/dXr[e][s]:
 *   dr[e][m]  = sum_s G[e][s] sum_m' (dp[m']/dr[m]) X[cand[e][m']][s],
 *               dp[m']/dr[m] = p[m'] ([m' == m] - p[m])
 *   dX[c][s] += p[m] G[e][s] for every (e, m) with cand[e][m] == c,
 *               added in increasing (e, m) order (dX optional, overwritten). */
void oracle_route_backward(const double* X, int32_t w_in, int64_t B, const int32_t* cand,
                           const float* r, int64_t n_slots, int32_t Kc, const double* G,
                           double* dr, double* dX) {
    double* prob = (double*)malloc(sizeof(double) * (size_t)n_slots * (size_t)Kc);
    double* Xr = (double*)malloc(sizeof(double) * (size_t)n_slots * (size_t)B);
    oracle_route_forward(X, w_in, B, cand, r, n_slots, Kc, Xr, prob);
    free(Xr);
#pragma omp parallel for schedule(dynamic, 64)
    for (int64_t e = 0; e < n_slots; ++e) {
        const double* p = prob + e * Kc;
        for (int32_t m = 0; m < Kc; ++m) {
            double acc = 0.0;
            for (int64_t s = 0; s < B; ++s) {
                double dxr = 0.0;   /* dXr[e][s] / dr[m] */
                for (int32_t q = 0; q < Kc; ++q)
                    dxr += p[q] * ((q == m ? 1.0 : 0.0) - p[m]) * X[(int64_t)cand[e * Kc + q] * B + s];
                acc += G[e * B + s] * dxr;
            }
            dr[e * Kc + m] = acc;
        }
    }
    if (dX) {
        memset(dX, 0, sizeof(double) * (size_t)w_in * (size_t)B);
#pragma omp parallel for schedule(static)
        for (int64_t s = 0; s < B; ++s)
            for (int64_t e = 0; e < n_slots; ++e)
                for (int32_t m = 0; m < Kc; ++m)
                    dX[(int64_t)cand[e * Kc + m] * B + s] += prob[e * Kc + m] * G[e * B + s];
    }
    free(prob);
}

/* Discretization of learnable routing: each slot keeps its most likely
 * candidate (the first one on ties). */
void oracle_route_snap(const int32_t* cand, const float* r, int64_t n_slots, int32_t Kc, int32_t* conn) {
    for (int64_t e = 0; e < n_slots; ++e) {
        int32_t best = 0;
        for (int32_t m = 1; m < Kc; ++m) if (r[e * Kc + m] > r[e * Kc + best]) best = m;
        conn[e] = cand[e * Kc + best];
    }
}

/* Table discretization (§3 "Nodes are parameterizations": every surrogate
 * discretizes to a 2^n-entry truth table; App. C.1 extracts it once per
 * layer): entry a is 1 exactly when theta_j[a] > 0, i.e. sigmoid > 1/2. */
void oracle_binarize_tables(const float* theta, int32_t w, int32_t k, uint64_t* table) {
    const int64_t K = (int64_t)1 << k;
    for (int32_t j = 0; j < w; ++j) {
        uint64_t t = 0;
        for (int64_t a = 0; a < K; ++a)
            if (theta[(int64_t)j * K + a] > 0.0f) t |= (uint64_t)1 << a;
        table[j] = t;
    }
}

/* Thermometer encoding followed by packing 32 samples per uint32 along the
 * batch (App. C.1 "Bit-packed inference" packs 64 per 64-bit word; this
 * layout uses 32 per 32-bit word): sample s is bit s%32 of word s/32. */
void oracle_pack_bits(const uint8_t* x, int64_t N, int32_t d,
                      const uint8_t* thr, int32_t b, uint32_t* xp) {
    const int64_t W = (N + 31) / 32;
    /* word q holds samples 32q .. 32q + 31: the words are independent outputs */
#pragma omp parallel for schedule(static)
    for (int64_t q = 0; q < W; ++q)
        for (int32_t j = 0; j < d; ++j)
            for (int32_t i = 0; i < b; ++i) {
                uint32_t word = 0;
                for (int t = 0; t < 32 && 32 * q + t < N; ++t)   /* sample s = 32 q + t */
                    if (x[(32 * q + t) * d + j] > thr[i]) word |= (uint32_t)1 << t;
                xp[((int64_t)j * b + i) * W + q] = word;
            }
}

/* Hard LUT layer on packed bits (App. C.1): for each sample, the node's
 * index a = sum_i bit(input M_j(i), s) << i selects table bit a.  Written
 * per sample as a plain lookup on unpacked bits; the k input words that hold
 * a sample's bits are read once for the 32 samples of the word. */
void oracle_hard_forward(const uint32_t* xp, int32_t w_in, int64_t N,
                         const int32_t* conn, const uint64_t* table, int32_t w, int32_t k,
                         uint32_t* yp) {
    const int64_t W = (N + 31) / 32;
    (void)w_in;
#pragma omp parallel for schedule(static)
    for (int32_t j = 0; j < w; ++j) {
        const uint64_t T = table[j];
        for (int64_t q = 0; q < W; ++q) {
            uint32_t in[6];
            for (int32_t i = 0; i < k; ++i) in[i] = xp[(int64_t)conn[(int64_t)j * k + i] * W + q];
            uint32_t out = 0;
            for (int t = 0; t < 32 && 32 * q + t < N; ++t) {   /* sample s = 32 q + t */
                uint32_t a = 0;
                for (int32_t i = 0; i < k; ++i) a |= ((in[i] >> t) & 1u) << i;
                out |= (uint32_t)((T >> a) & 1u) << t;
            }
            yp[(int64_t)j * W + q] = out;
        }
    }
}

/* Popcount GroupSum head in hard mode (§3 "Encoders and heads"): the score
 * of class c is the number of ones among its contiguous group of g = w/C
 * nodes; the prediction is the first class with the largest score.  The
 * samples of one packed word are counted together (each word of a node is
 * read once for its 32 samples; integer counts do not depend on the order
 * of the additions). */
void oracle_popcount_head(const uint32_t* yp, int32_t w, int64_t N, int32_t C,
                          int32_t* counts, int32_t* pred) {
    const int64_t W = (N + 31) / 32;
    const int32_t g = w / C;
#pragma omp parallel for schedule(static)
    for (int64_t q = 0; q < W; ++q) {
        int32_t cnt[32];
        int32_t best[32], bestc[32];
        for (int32_t c = 0; c < C; ++c) {
            for (int t = 0; t < 32; ++t) cnt[t] = 0;
            for (int32_t j = c * g; j < (c + 1) * g; ++j) {
                const uint32_t word = yp[(int64_t)j * W + q];
                for (int t = 0; t < 32; ++t) cnt[t] += (int32_t)((word >> t) & 1u);
            }
            for (int64_t s = 32 * q; s < N && s < 32 * q + 32; ++s) {
                const int t = (int)(s % 32);
                if (counts) counts[s * C + c] = cnt[t];
                if (c == 0 || cnt[t] > best[t]) { best[t] = cnt[t]; bestc[t] = c; }
            }
        }
        for (int64_t s = 32 * q; s < N && s < 32 * q + 32; ++s)
            if (pred) pred[s] = bestc[s % 32];
    }
}

/* One AdamW step (§4 "Training": AdamW with beta1 0.9, beta2 0.999,
 * eps 1e-8, constant learning rate 0.01, weight decay 0), with decoupled
 * weight decay, for step number t >= 1 and every parameter i:
 *   m_i     = beta1 m_i + (1 - beta1) g_i
 *   v_i     = beta2 v_i + (1 - beta2) g_i^2
 *   theta_i = theta_i - lr ( (m_i / (1 - beta1^t)) / (sqrt(v_i / (1 - beta2^t)) + eps)
 *                             + wd theta_i )                                       */
void oracle_adamw_step(double* theta, double* m, double* v, const double* g, int64_t n,
                       int64_t t, double lr, double beta1, double beta2, double eps,
                       double wd) {
    const double bc1 = 1.0 - pow(beta1, (double)t);
    const double bc2 = 1.0 - pow(beta2, (double)t);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        m[i] = beta1 * m[i] + (1.0 - beta1) * g[i];
        v[i] = beta2 * v[i] + (1.0 - beta2) * g[i] * g[i];
        const double mhat = m[i] / bc1;
        const double vhat = v[i] / bc2;
        theta[i] = theta[i] - lr * (mhat / (sqrt(vhat) + eps) + wd * theta[i]);
    }
}
