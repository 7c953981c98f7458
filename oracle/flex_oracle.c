/*
 * flex_oracle.c -- plain, slow, fp64 CPU oracle for Flexformer's random-Fourier-feature
 * linear attention (stationary and nonstationary variants), forward and backward.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the bench's CPU
 * baseline may load this library.  It shares no code, header or constant with the CUDA
 * path; it is written directly from the paper's equations:
 *
 *   Sec. 2.2, Eq. (kernel) / Eq. (linear att):
 *       O_i = phi(Q_i)^T sum_j phi(K_j) V_j^T  /  phi(Q_i)^T sum_j phi(K_j)
 *   Sec. 3.1, Eq. (phi_n):    stationary random Fourier features
 *       phi(x) = sigma/sqrt(n) [cos w_1.x .. cos w_n.x, sin w_1.x .. sin w_n.x]
 *   Sec. 3.2, Flexformer_s:   the frequencies w_i are the learnable matrix W1 (n = M rows)
 *   Sec. 3.2, Eq. (phi_non):  nonstationary (Yaglom) features with frequency pairs (W1, W2)
 *       w'_1i = (w_1i + w_2i)/2,  w'_2i = (w_1i - w_2i)/2
 *       phi(x) = c [cos w'_1i.x cos w'_2i.x ..., sin w'_1i.x cos w'_2i.x ...]
 *
 * Readings taken where the paper is silent or garbled (each is listed in the design notes):
 *   - scale: sigma = 1 and c = M^{-1/2} for both variants.  The printed nonstationary
 *     constant sigma/(2 sqrt n) drops the factor 4 that the sum-to-product step produces;
 *     M^{-1/2} is the value that makes the last two lines of Eq. (phi_non) agree.
 *     Any global scale cancels in O and in every gradient.
 *   - causal attention sums over j <= i (the diagonal is included).
 *   - the denominator is used as it is: no epsilon, no clamp.
 *   - the learned parameters of Flexformer_n are (W1, W2); dW1 and dW2 are returned.
 *   - the norm prefactor of Sec. 3.2, phi~(x) = exp(|x|^2 / exp(tau)) phi(x), is optional
 *     (tau per head; NULL = none).  The query's factor multiplies every term of row i of
 *     both sums in Eq. (linear att) and cancels; what remains is a weight
 *     w_j = exp(|k_j|^2 exp(-tau)) on key j, so S = sum_j w_j phi(k_j) v_j^T and
 *     z = sum_j w_j phi(k_j).  den is phi(q_i)^T z (without the query factor), and dtau
 *     is returned with the other gradients.
 *
 * The backward pass is the analytic gradient of L = sum_i dO_i . O_i, derived by hand
 * from Eq. (linear att) (the paper gives none; it only states that the frequencies are
 * trained end to end):
 *   g_i = dO_i / den_i,  c_i = -(dO_i . O_i) / den_i
 *   dphi(q_i) = S_i g_i + c_i z_i           (S_i, z_i: running sums over j <= i)
 *   dphi(k_j) = R_j v_j + r_j               (R_j = sum_{i>=j} phi(q_i) g_i^T, r_j = sum c_i phi(q_i))
 *   dv_j      = R_j^T phi(k_j)
 * and through the feature map by the chain rule.  With the key weight w_j the same
 * formulas hold for phi~(k_j) = w_j phi(k_j); then dphi(k_j) = w_j dphi~(k_j) and, with
 * dw_j = phi(k_j) . dphi~(k_j):  dk_j += dw_j w_j 2 exp(-tau) k_j,
 * dtau += -dw_j w_j |k_j|^2 exp(-tau).  For non-causal attention every
 * running sum is replaced by the total.
 *
 * Layouts: q, k, v, out, dout, dq, dk, dv are [B][H][N][d]; W1, W2, dW1, dW2 are [H][M][d];
 * den is [B][H][N]; phi is [B][H][N][2M].  All doubles, row-major, contiguous.
 */
#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------------------ */
/* Feature map (Eq. phi_n, Eq. phi_non), one vector.                                       */
/* ------------------------------------------------------------------------------------ */

static double dot(int d, const double* a, const double* b)
{
    double s = 0.0;
    for (int t = 0; t < d; ++t) s += a[t] * b[t];
    return s;
}

/* phi (length 2M) of x (length d).  W2 == NULL selects the stationary map. */
static void feature(int d, int M, const double* x, const double* W1, const double* W2,
                    double* phi)
{
    const double c = 1.0 / sqrt((double)M);
    for (int i = 0; i < M; ++i) {
        const double* w1 = W1 + (size_t)i * d;
        if (W2 == NULL) {
            double a = dot(d, w1, x);
            phi[i] = c * cos(a);
            phi[M + i] = c * sin(a);
        } else {
            const double* w2 = W2 + (size_t)i * d;
            double u = 0.0, w = 0.0;           /* u = w'_1i . x,  w = w'_2i . x */
            for (int t = 0; t < d; ++t) {
                u += 0.5 * (w1[t] + w2[t]) * x[t];
                w += 0.5 * (w1[t] - w2[t]) * x[t];
            }
            phi[i] = c * cos(u) * cos(w);
            phi[M + i] = c * sin(u) * cos(w);
        }
    }
}

/* The same nonstationary map written as the Monte Carlo sum of Eq. (phi_non) before the
 * sum-to-product step: (cos w_1i.x + cos w_2i.x, sin w_1i.x + sin w_2i.x) / (2 sqrt M).
 * Used only to check the product form above against the paper's own derivation. */
static void feature_sumform(int d, int M, const double* x, const double* W1, const double* W2,
                            double* phi)
{
    const double c = 0.5 / sqrt((double)M);
    for (int i = 0; i < M; ++i) {
        double a = dot(d, W1 + (size_t)i * d, x);
        double b = dot(d, W2 + (size_t)i * d, x);
        phi[i] = c * (cos(a) + cos(b));
        phi[M + i] = c * (sin(a) + sin(b));
    }
}

/* Gradient of the feature map.  Given x and dphi (length 2M), adds the contribution to
 * dx (length d) and to dA, dB ([M][d] each).  Stationary: dA = dW1, dB unused.
 * Nonstationary: dA = dU, dB = dV for U = (W1+W2)/2 and V = (W1-W2)/2; the caller turns
 * them into dW1 = (dU+dV)/2, dW2 = (dU-dV)/2. */
static void feature_backward(int d, int M, const double* x, const double* W1,
                             const double* W2, const double* dphi, double* dx, double* dA,
                             double* dB)
{
    const double c = 1.0 / sqrt((double)M);
    for (int i = 0; i < M; ++i) {
        const double* w1 = W1 + (size_t)i * d;
        const double dc = dphi[i], ds = dphi[M + i];
        if (W2 == NULL) {
            double a = dot(d, w1, x);
            double da = c * (-sin(a) * dc + cos(a) * ds);
            for (int t = 0; t < d; ++t) {
                dx[t] += da * w1[t];
                dA[(size_t)i * d + t] += da * x[t];
            }
        } else {
            const double* w2 = W2 + (size_t)i * d;
            double u = 0.0, w = 0.0;
            for (int t = 0; t < d; ++t) {
                u += 0.5 * (w1[t] + w2[t]) * x[t];
                w += 0.5 * (w1[t] - w2[t]) * x[t];
            }
            /* phi_c = c cos u cos w, phi_s = c sin u cos w */
            double du = c * cos(w) * (-sin(u) * dc + cos(u) * ds);
            double dw = -c * sin(w) * (cos(u) * dc + sin(u) * ds);
            for (int t = 0; t < d; ++t) {
                dx[t] += du * 0.5 * (w1[t] + w2[t]) + dw * 0.5 * (w1[t] - w2[t]);
                dA[(size_t)i * d + t] += du * x[t];
                dB[(size_t)i * d + t] += dw * x[t];
            }
        }
    }
}

/* ------------------------------------------------------------------------------------ */
/* Linear attention of one (b, h) sequence (Eq. linear att).                               */
/* ------------------------------------------------------------------------------------ */

typedef struct {
    int N, d, M, causal;
    const double *q, *k, *v, *W1, *W2, *dout;
    double *out, *den, *dq, *dk, *dv, *dA, *dB;
    double itau;   /* exp(-tau) of the head, 0 without the prefactor (then w_j = 1) */
    double *dtau;  /* this sequence's dtau (backward with the prefactor), else NULL */
} seq_job;

/* Key weight of the norm prefactor (Sec. 3.2): w = exp(|k|^2 exp(-tau)). */
static double key_weight(int d, const double* k, double itau)
{
    return exp(dot(d, k, k) * itau);
}

/* out[i] = phi(q_i)^T S / phi(q_i)^T z with S = sum phi(k_j) v_j^T, z = sum phi(k_j);
 * j runs over j <= i when causal, over all j otherwise. */
static void forward_seq(const seq_job* J)
{
    const int N = J->N, d = J->d, M = J->M, D = 2 * M;
    double* S = calloc((size_t)D * d, sizeof(double));
    double* z = calloc((size_t)D, sizeof(double));
    double* pk = malloc(sizeof(double) * D);
    double* pq = malloc(sizeof(double) * D);
    double* num = malloc(sizeof(double) * d);

    if (!J->causal) {
        for (int j = 0; j < N; ++j) {
            feature(d, M, J->k + (size_t)j * d, J->W1, J->W2, pk);
            const double wj = key_weight(d, J->k + (size_t)j * d, J->itau);
            for (int f = 0; f < D; ++f) pk[f] *= wj;
            for (int f = 0; f < D; ++f) {
                z[f] += pk[f];
                for (int e = 0; e < d; ++e) S[(size_t)f * d + e] += pk[f] * J->v[(size_t)j * d + e];
            }
        }
    }
    for (int i = 0; i < N; ++i) {
        if (J->causal) {
            feature(d, M, J->k + (size_t)i * d, J->W1, J->W2, pk);
            const double wi = key_weight(d, J->k + (size_t)i * d, J->itau);
            for (int f = 0; f < D; ++f) pk[f] *= wi;
            for (int f = 0; f < D; ++f) {
                z[f] += pk[f];
                for (int e = 0; e < d; ++e) S[(size_t)f * d + e] += pk[f] * J->v[(size_t)i * d + e];
            }
        }
        feature(d, M, J->q + (size_t)i * d, J->W1, J->W2, pq);
        double dn = 0.0;
        for (int e = 0; e < d; ++e) num[e] = 0.0;
        for (int f = 0; f < D; ++f) {
            dn += pq[f] * z[f];
            for (int e = 0; e < d; ++e) num[e] += pq[f] * S[(size_t)f * d + e];
        }
        for (int e = 0; e < d; ++e) J->out[(size_t)i * d + e] = num[e] / dn;
        if (J->den) J->den[i] = dn;
    }
    free(S); free(z); free(pk); free(pq); free(num);
}

/* Gradient of L = sum_i dout_i . out_i with respect to q, k, v and the frequencies. */
static void backward_seq(const seq_job* J)
{
    const int N = J->N, d = J->d, M = J->M, D = 2 * M;
    double* out = malloc(sizeof(double) * (size_t)N * d);
    double* den = malloc(sizeof(double) * (size_t)N);
    seq_job F = *J;
    F.out = out;
    F.den = den;
    forward_seq(&F);

    double* PQ = malloc(sizeof(double) * (size_t)N * D);   /* phi(q_i) */
    double* PK = malloc(sizeof(double) * (size_t)N * D);   /* phi~(k_j) = w_j phi(k_j) */
    double* wk = malloc(sizeof(double) * (size_t)N);       /* w_j */
    double* g = malloc(sizeof(double) * (size_t)N * d);    /* dout_i / den_i */
    double* cc = malloc(sizeof(double) * (size_t)N);       /* -(dout_i . out_i) / den_i */
    for (int i = 0; i < N; ++i) {
        feature(d, M, J->q + (size_t)i * d, J->W1, J->W2, PQ + (size_t)i * D);
        feature(d, M, J->k + (size_t)i * d, J->W1, J->W2, PK + (size_t)i * D);
        wk[i] = key_weight(d, J->k + (size_t)i * d, J->itau);
        for (int f = 0; f < D; ++f) PK[(size_t)i * D + f] *= wk[i];
        const double* dO = J->dout + (size_t)i * d;
        double s = 0.0;
        for (int e = 0; e < d; ++e) {
            g[(size_t)i * d + e] = dO[e] / den[i];
            s += dO[e] * out[(size_t)i * d + e];
        }
        cc[i] = -s / den[i];
    }

    double* S = calloc((size_t)D * d, sizeof(double));
    double* z = calloc((size_t)D, sizeof(double));
    double* dphi = malloc(sizeof(double) * D);

    /* dq: forward-direction running sums S_i, z_i (totals when non-causal). */
    if (!J->causal) {
        for (int j = 0; j < N; ++j)
            for (int f = 0; f < D; ++f) {
                z[f] += PK[(size_t)j * D + f];
                for (int e = 0; e < d; ++e)
                    S[(size_t)f * d + e] += PK[(size_t)j * D + f] * J->v[(size_t)j * d + e];
            }
    }
    for (int i = 0; i < N; ++i) {
        if (J->causal)
            for (int f = 0; f < D; ++f) {
                z[f] += PK[(size_t)i * D + f];
                for (int e = 0; e < d; ++e)
                    S[(size_t)f * d + e] += PK[(size_t)i * D + f] * J->v[(size_t)i * d + e];
            }
        for (int f = 0; f < D; ++f) {
            double s = cc[i] * z[f];
            for (int e = 0; e < d; ++e) s += S[(size_t)f * d + e] * g[(size_t)i * d + e];
            dphi[f] = s;
        }
        feature_backward(d, M, J->q + (size_t)i * d, J->W1, J->W2, dphi, J->dq + (size_t)i * d,
                         J->dA, J->dB);
    }

    /* dk, dv: reverse-direction running sums R_j, r_j (totals when non-causal). */
    double* R = S;  /* reuse: R[f][e] */
    double* r = z;
    memset(R, 0, sizeof(double) * (size_t)D * d);
    memset(r, 0, sizeof(double) * D);
    if (!J->causal) {
        for (int i = 0; i < N; ++i)
            for (int f = 0; f < D; ++f) {
                r[f] += cc[i] * PQ[(size_t)i * D + f];
                for (int e = 0; e < d; ++e)
                    R[(size_t)f * d + e] += PQ[(size_t)i * D + f] * g[(size_t)i * d + e];
            }
    }
    for (int j = N - 1; j >= 0; --j) {
        if (J->causal)
            for (int f = 0; f < D; ++f) {
                r[f] += cc[j] * PQ[(size_t)j * D + f];
                for (int e = 0; e < d; ++e)
                    R[(size_t)f * d + e] += PQ[(size_t)j * D + f] * g[(size_t)j * d + e];
            }
        const double* vj = J->v + (size_t)j * d;
        const double* kj = J->k + (size_t)j * d;
        const double* pk = PK + (size_t)j * D;
        for (int f = 0; f < D; ++f) dphi[f] = r[f] + dot(d, R + (size_t)f * d, vj);
        for (int e = 0; e < d; ++e) {
            double s = 0.0;
            for (int f = 0; f < D; ++f) s += R[(size_t)f * d + e] * pk[f];
            J->dv[(size_t)j * d + e] = s;
        }
        /* dphi is the gradient with respect to phi~(k_j); dw_j = phi(k_j) . dphi. */
        const double dw = dot(D, pk, dphi) / wk[j];
        for (int f = 0; f < D; ++f) dphi[f] *= wk[j];
        feature_backward(d, M, kj, J->W1, J->W2, dphi, J->dk + (size_t)j * d, J->dA, J->dB);
        for (int e = 0; e < d; ++e) J->dk[(size_t)j * d + e] += dw * wk[j] * 2.0 * J->itau * kj[e];
        if (J->dtau) *J->dtau += -dw * wk[j] * dot(d, kj, kj) * J->itau;
    }
    free(out); free(den); free(PQ); free(PK); free(wk); free(g); free(cc);
    free(S); free(z); free(dphi);
}

/* ------------------------------------------------------------------------------------ */
/* Threading over independent (b, h) sequences.                                            */
/* ------------------------------------------------------------------------------------ */

typedef struct {
    seq_job* jobs;
    int njobs, stride, first, backward;
} worker_arg;

static void* worker(void* p)
{
    worker_arg* a = (worker_arg*)p;
    for (int u = a->first; u < a->njobs; u += a->stride) {
        if (a->backward) backward_seq(&a->jobs[u]);
        else forward_seq(&a->jobs[u]);
    }
    return NULL;
}

static void run_jobs(seq_job* jobs, int njobs, int nthreads, int backward)
{
    if (nthreads < 1) nthreads = 1;
    if (nthreads > njobs) nthreads = njobs;
    pthread_t* th = malloc(sizeof(pthread_t) * nthreads);
    worker_arg* args = malloc(sizeof(worker_arg) * nthreads);
    for (int t = 0; t < nthreads; ++t) {
        args[t] = (worker_arg){jobs, njobs, nthreads, t, backward};
        if (t > 0) pthread_create(&th[t], NULL, worker, &args[t]);
    }
    worker(&args[0]);
    for (int t = 1; t < nthreads; ++t) pthread_join(th[t], NULL);
    free(th); free(args);
}

static int bad_shape(int B, int H, int N, int d, int M)
{
    return B < 1 || H < 1 || N < 1 || d < 1 || M < 1;
}

/* ------------------------------------------------------------------------------------ */
/* Exported entry points.  Return 0 on success, -1 on a bad shape.                         */
/* ------------------------------------------------------------------------------------ */

int oracle_featmap(int B, int H, int N, int d, int M, const double* x, const double* W1,
                   const double* W2, double* phi)
{
    if (bad_shape(B, H, N, d, M)) return -1;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            const double* w1 = W1 + (size_t)h * M * d;
            const double* w2 = W2 ? W2 + (size_t)h * M * d : NULL;
            for (int n = 0; n < N; ++n) {
                size_t row = ((size_t)b * H + h) * N + n;
                feature(d, M, x + row * d, w1, w2, phi + row * 2 * M);
            }
        }
    return 0;
}

int oracle_featmap_sumform(int B, int H, int N, int d, int M, const double* x,
                           const double* W1, const double* W2, double* phi)
{
    if (bad_shape(B, H, N, d, M) || W2 == NULL) return -1;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h)
            for (int n = 0; n < N; ++n) {
                size_t row = ((size_t)b * H + h) * N + n;
                feature_sumform(d, M, x + row * d, W1 + (size_t)h * M * d,
                                W2 + (size_t)h * M * d, phi + row * 2 * M);
            }
    return 0;
}

int oracle_linattn_fwd(int B, int H, int N, int d, int M, const double* q, const double* k,
                       const double* v, const double* W1, const double* W2,
                       const double* tau, int causal, double* out, double* den, int nthreads)
{
    if (bad_shape(B, H, N, d, M)) return -1;
    seq_job* jobs = calloc((size_t)B * H, sizeof(seq_job));
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            size_t u = (size_t)b * H + h, off = u * N * d;
            jobs[u] = (seq_job){N, d, M, causal, q + off, k + off, v + off,
                                W1 + (size_t)h * M * d, W2 ? W2 + (size_t)h * M * d : NULL,
                                NULL, out + off, den ? den + u * N : NULL,
                                NULL, NULL, NULL, NULL, NULL, tau ? exp(-tau[h]) : 0.0, NULL};
        }
    run_jobs(jobs, B * H, nthreads, 0);
    free(jobs);
    return 0;
}

/* dW1 (and dW2, dtau) are sums over the batch and the sequence; they are overwritten. */
int oracle_linattn_bwd(int B, int H, int N, int d, int M, const double* q, const double* k,
                       const double* v, const double* W1, const double* W2,
                       const double* tau, int causal, const double* dout, double* dq,
                       double* dk, double* dv, double* dW1, double* dW2, double* dtau,
                       int nthreads)
{
    if (bad_shape(B, H, N, d, M)) return -1;
    if ((W2 == NULL) != (dW2 == NULL) || (tau == NULL) != (dtau == NULL)) return -1;
    const size_t per = (size_t)M * d;
    double* dA = calloc((size_t)B * H * per, sizeof(double));
    double* dB = calloc((size_t)B * H * per, sizeof(double));
    double* dt = calloc((size_t)B * H, sizeof(double));
    seq_job* jobs = calloc((size_t)B * H, sizeof(seq_job));
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            size_t u = (size_t)b * H + h, off = u * N * d;
            memset(dq + off, 0, sizeof(double) * (size_t)N * d);
            memset(dk + off, 0, sizeof(double) * (size_t)N * d);
            jobs[u] = (seq_job){N, d, M, causal, q + off, k + off, v + off,
                                W1 + (size_t)h * per, W2 ? W2 + (size_t)h * per : NULL,
                                dout + off, NULL, NULL, dq + off, dk + off, dv + off,
                                dA + u * per, dB + u * per, tau ? exp(-tau[h]) : 0.0,
                                tau ? dt + u : NULL};
        }
    run_jobs(jobs, B * H, nthreads, 1);
    /* Sum the per-sequence parameter gradients over the batch in a fixed order. */
    for (int h = 0; h < H; ++h)
        for (size_t t = 0; t < per; ++t) {
            double a = 0.0, bb = 0.0;
            for (int b = 0; b < B; ++b) {
                size_t u = (size_t)b * H + h;
                a += dA[u * per + t];
                bb += dB[u * per + t];
            }
            if (W2 == NULL) {
                dW1[h * per + t] = a;
            } else {
                dW1[h * per + t] = 0.5 * (a + bb);
                dW2[h * per + t] = 0.5 * (a - bb);
            }
        }
    if (dtau)
        for (int h = 0; h < H; ++h) {
            double a = 0.0;
            for (int b = 0; b < B; ++b) a += dt[(size_t)b * H + h];
            dtau[h] = a;
        }
    free(dA); free(dB); free(dt); free(jobs);
    return 0;
}

/* ------------------------------------------------------------------------------------ */
/* Attention-weight distillation loss (the loss of the softmax-recovery experiments, the   */
/* appendix's distillation setting): per query i, the teacher distribution                 */
/* P_ij = softmax_j(q_i . k_j / sqrt(d)) and the kernel's normalised weights               */
/* R_ij = A~_ij / D_i with A~_ij = phi~(q_i) . phi~(k_j), D_i = sum_l A~_il; the loss of   */
/* a sequence is L = -(1/N) sum_i sum_j P_ij log R_ij (j over all keys, or j <= i when     */
/* causal).  The query's prefactor and the global scale cancel in R, so A~_ij =            */
/* w_j phi(q_i) . phi(k_j) with the key weight of the norm prefactor (w = 1 without tau).  */
/* Reading: RFF estimates can be negative, and so can a row sum D_i; an entry whose        */
/* normalised weight R_ij = A~_ij / D_i is not positive has no logarithm and contributes    */
/* log(AWD_EPS) and no gradient.                                                            */
/* ------------------------------------------------------------------------------------ */
#define AWD_EPS 1e-6

static double awd_seq(int N, int d, int M, int causal, const double* q, const double* k,
                      const double* W1, const double* W2, double itau)
{
    const int D = 2 * M;
    double* PQ = malloc(sizeof(double) * (size_t)N * D);
    double* PK = malloc(sizeof(double) * (size_t)N * D);
    double* sc = malloc(sizeof(double) * (size_t)N);
    double* at = malloc(sizeof(double) * (size_t)N);
    for (int i = 0; i < N; ++i) {
        feature(d, M, q + (size_t)i * d, W1, W2, PQ + (size_t)i * D);
        feature(d, M, k + (size_t)i * d, W1, W2, PK + (size_t)i * D);
        const double wk = key_weight(d, k + (size_t)i * d, itau);
        for (int f = 0; f < D; ++f) PK[(size_t)i * D + f] *= wk;
    }
    double loss = 0.0;
    for (int i = 0; i < N; ++i) {
        const int J = causal ? i + 1 : N;
        double smax = -INFINITY, Dn = 0.0;
        for (int j = 0; j < J; ++j) {
            sc[j] = dot(d, q + (size_t)i * d, k + (size_t)j * d) / sqrt((double)d);
            at[j] = dot(D, PQ + (size_t)i * D, PK + (size_t)j * D);
            if (sc[j] > smax) smax = sc[j];
            Dn += at[j];
        }
        double Z = 0.0, ce = 0.0;
        for (int j = 0; j < J; ++j) Z += exp(sc[j] - smax);
        for (int j = 0; j < J; ++j) {
            const double Pij = exp(sc[j] - smax) / Z;
            const double r = at[j] / Dn;
            ce -= Pij * (r > 0.0 ? log(r) : log(AWD_EPS));
        }
        loss += ce;
    }
    free(PQ); free(PK); free(sc); free(at);
    return loss / N;
}

/* loss [B][H]: the distillation loss of every (b, h) sequence; tau [H] or NULL. */
int oracle_awd(int B, int H, int N, int d, int M, const double* q, const double* k,
               const double* W1, const double* W2, const double* tau, int causal,
               double* loss)
{
    if (bad_shape(B, H, N, d, M)) return -1;
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            const size_t u = (size_t)b * H + h, off = u * N * d;
            loss[u] = awd_seq(N, d, M, causal, q + off, k + off, W1 + (size_t)h * M * d,
                              W2 ? W2 + (size_t)h * M * d : NULL, tau ? exp(-tau[h]) : 0.0);
        }
    return 0;
}

/* Gradient of the distillation loss with respect to the kernel's parameters (the
 * distillation trains only the feature map: W1, W2 and tau; q and k are frozen).
 * For an entry with R_ij > 0, log R_ij = log|A~_ij| - log|D_i|; entries with R_ij <= 0
 * are constant.  With c_i = sum of P_ij over the entries with R_ij > 0 and the upstream
 * gradient dl of this sequence's loss:
 *   dL/dA~_ij = -(dl/N) ( [R_ij > 0] P_ij / A~_ij  -  c_i / D_i )     (j in the row)
 * (the second term from D_i = sum_j A~_ij), then
 *   dphi(q_i) = sum_j dA~_ij phi~(k_j),   dphi~(k_j) = sum_i dA~_ij phi(q_i),
 *   dphi(k_j) = w_j dphi~(k_j),   dtau += -(phi~(k_j) . dphi~(k_j)) |k_j|^2 exp(-tau)
 * (from dw_j/dtau = -w_j |k_j|^2 exp(-tau)), and the feature map's chain rule into dA, dB
 * ([M][d], as in the attention backward). */
static void awd_grad_seq(int N, int d, int M, int causal, const double* q, const double* k,
                         const double* W1, const double* W2, double itau, double dl,
                         double* dA, double* dB, double* dtau)
{
    const int D = 2 * M;
    double* PQ = malloc(sizeof(double) * (size_t)N * D);
    double* PK = malloc(sizeof(double) * (size_t)N * D);
    double* dPQ = calloc((size_t)N * D, sizeof(double));
    double* dPK = calloc((size_t)N * D, sizeof(double));
    double* wk = malloc(sizeof(double) * (size_t)N);
    double* sc = malloc(sizeof(double) * (size_t)N);
    double* at = malloc(sizeof(double) * (size_t)N);
    double* P = malloc(sizeof(double) * (size_t)N);
    double* dx = calloc((size_t)d, sizeof(double));  /* dq, dk: not needed, discarded */
    for (int i = 0; i < N; ++i) {
        feature(d, M, q + (size_t)i * d, W1, W2, PQ + (size_t)i * D);
        feature(d, M, k + (size_t)i * d, W1, W2, PK + (size_t)i * D);
        wk[i] = key_weight(d, k + (size_t)i * d, itau);
        for (int f = 0; f < D; ++f) PK[(size_t)i * D + f] *= wk[i];
    }
    for (int i = 0; i < N; ++i) {
        const int J = causal ? i + 1 : N;
        double smax = -INFINITY, Dn = 0.0, Z = 0.0, ci = 0.0;
        for (int j = 0; j < J; ++j) {
            sc[j] = dot(d, q + (size_t)i * d, k + (size_t)j * d) / sqrt((double)d);
            at[j] = dot(D, PQ + (size_t)i * D, PK + (size_t)j * D);
            if (sc[j] > smax) smax = sc[j];
            Dn += at[j];
        }
        for (int j = 0; j < J; ++j) Z += exp(sc[j] - smax);
        for (int j = 0; j < J; ++j) {
            P[j] = exp(sc[j] - smax) / Z;
            if (at[j] / Dn > 0.0) ci += P[j];
        }
        for (int j = 0; j < J; ++j) {
            const double first = at[j] / Dn > 0.0 ? P[j] / at[j] : 0.0;
            const double g = -(dl / N) * (first - ci / Dn);
            for (int f = 0; f < D; ++f) {
                dPQ[(size_t)i * D + f] += g * PK[(size_t)j * D + f];
                dPK[(size_t)j * D + f] += g * PQ[(size_t)i * D + f];
            }
        }
    }
    for (int i = 0; i < N; ++i) {
        feature_backward(d, M, q + (size_t)i * d, W1, W2, dPQ + (size_t)i * D, dx, dA, dB);
        const double* kj = k + (size_t)i * d;
        double s = dot(D, PK + (size_t)i * D, dPK + (size_t)i * D);
        if (dtau) *dtau += -s * dot(d, kj, kj) * itau;
        for (int f = 0; f < D; ++f) dPK[(size_t)i * D + f] *= wk[i];
        feature_backward(d, M, kj, W1, W2, dPK + (size_t)i * D, dx, dA, dB);
    }
    free(PQ); free(PK); free(dPQ); free(dPK); free(wk); free(sc); free(at); free(P); free(dx);
}

/* dW1, dW2 [H][M][d] (dW2 only with W2) and dtau [H] (only with tau): the gradient of
 * sum_{b,h} dloss[b][h] L[b][h] with L the distillation loss of oracle_awd. */
int oracle_awd_bwd(int B, int H, int N, int d, int M, const double* q, const double* k,
                   const double* W1, const double* W2, const double* tau, int causal,
                   const double* dloss, double* dW1, double* dW2, double* dtau)
{
    if (bad_shape(B, H, N, d, M)) return -1;
    const size_t per = (size_t)M * d;
    double* dA = malloc(sizeof(double) * per);
    double* dB = malloc(sizeof(double) * per);
    for (int h = 0; h < H; ++h) {
        memset(dA, 0, sizeof(double) * per);
        memset(dB, 0, sizeof(double) * per);
        double dt = 0.0;
        const double* w1 = W1 + (size_t)h * per;
        const double* w2 = W2 ? W2 + (size_t)h * per : NULL;
        for (int b = 0; b < B; ++b) {
            const size_t u = (size_t)b * H + h, off = u * N * d;
            awd_grad_seq(N, d, M, causal, q + off, k + off, w1, w2, tau ? exp(-tau[h]) : 0.0,
                         dloss[u], dA, dB, tau ? &dt : NULL);
        }
        for (size_t t = 0; t < per; ++t) {
            if (W2 == NULL) {
                dW1[h * per + t] = dA[t];
            } else {               /* U = (W1+W2)/2, V = (W1-W2)/2 */
                dW1[h * per + t] = 0.5 * (dA[t] + dB[t]);
                dW2[h * per + t] = 0.5 * (dA[t] - dB[t]);
            }
        }
        if (tau) dtau[h] = dt;
    }
    free(dA); free(dB);
    return 0;
}

/* One step of the causal recurrence behind Eq. (linear att) with j <= i: the running sums
 * S = sum_j phi(k_j) v_j^T and z = sum_j phi(k_j) absorb the new token (inclusive), then
 * out = phi(q)^T S / den with den = phi(q)^T z.  Per (b, h): q, k, v, out [d]; S [2M][d]
 * and z [2M] are updated in place; den [1].  With tau, the new key's phi carries its
 * weight w = exp(|k|^2 exp(-tau)) as in the forward. */
int oracle_linattn_decode(int B, int H, int d, int M, const double* q, const double* k,
                          const double* v, const double* W1, const double* W2,
                          const double* tau, double* S, double* z, double* out, double* den)
{
    if (bad_shape(B, H, 1, d, M)) return -1;
    const int F = 2 * M;
    double* pq = malloc((size_t)F * sizeof(double));
    double* pk = malloc((size_t)F * sizeof(double));
    for (int b = 0; b < B; ++b)
        for (int h = 0; h < H; ++h) {
            const size_t u = (size_t)b * H + h;
            const double* w1 = W1 + (size_t)h * M * d;
            const double* w2 = W2 ? W2 + (size_t)h * M * d : NULL;
            feature(d, M, q + u * d, w1, w2, pq);
            feature(d, M, k + u * d, w1, w2, pk);
            const double wk = key_weight(d, k + u * d, tau ? exp(-tau[h]) : 0.0);
            for (int f = 0; f < F; ++f) pk[f] *= wk;
            double* Su = S + u * F * d;
            double* zu = z + u * F;
            for (int f = 0; f < F; ++f) {
                for (int e = 0; e < d; ++e) Su[(size_t)f * d + e] += pk[f] * v[u * d + e];
                zu[f] += pk[f];
            }
            double dn = 0.0;
            for (int f = 0; f < F; ++f) dn += pq[f] * zu[f];
            for (int e = 0; e < d; ++e) {
                double num = 0.0;
                for (int f = 0; f < F; ++f) num += pq[f] * Su[(size_t)f * d + e];
                out[u * d + e] = num / dn;
            }
            den[u] = dn;
        }
    free(pq);
    free(pk);
    return 0;
}
