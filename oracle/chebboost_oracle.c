/*
 * Plain CPU oracle for ChebBooster's online extrapolation stage.
 *
 * TEST INFRASTRUCTURE ONLY. The tests, the smoke check and the bench's CPU
 * baseline leg load this file's shared object; the CUDA library never links,
 * includes or calls it, and it shares no code, header or table with that
 * library. Everything here is written straight from the paper, in fp64, with
 * no blocking, fusion or reordering beyond what the definitions state, so
 * that each function can be checked against the paper by eye.
 *
 * Functions and the passages they follow:
 *   orc_full_schedule   Sec. 3.3, Eq. for the full-computation set F, plus the
 *                       warm-up reading of Sec. 3.3: a step extrapolates only
 *                       once the history buffer H holds n entries.
 *   orc_normalize       Sec. 3.3: timesteps mapped affinely onto [-1, 1].
 *   orc_nodal           App. A: nodal polynomial omega(x) = prod_k (x - x_k).
 *   orc_rho             App. A, Eq. general_weights: rho_j = 1 / omega'(x_j),
 *                       omega'(x_j) = prod_{k != j} (x_j - x_k).
 *   orc_bary_coeff      Sec. 3.2, Eq. barycentric_coeff:
 *                       w_j = (rho_j / (x - x_j)) / sum_i rho_i / (x - x_i).
 *   orc_lagrange_basis  App. A: l_j(x) = prod_{k != j} (x - x_k) / (x_j - x_k).
 *   orc_taylor_weights  Sec. 3.2, Fig. 4's Taylor expansion: f(t) ~ sum_i theta^i/i!
 *                       times the i-th backward difference at the newest node
 *                       (derivatives estimated on equispaced nodes), written as
 *                       one weight per node.
 *   orc_extrapolate     Sec. 3.3 Eq. for f_t (Alg. 1, extrapolation branch):
 *                       f_t = sum_j w_j f_{s_j}, per element, in fp64, then one
 *                       rounding to the output type; optionally the block
 *                       residual of Sec. 3.1 (B(x) = x + S + C + M): the hidden
 *                       state plus every branch prediction, each optionally
 *                       times its per-element gate, rounded once.
 *   orc_convert         the cache write of Alg. 1 (the full step's pair goes
 *                       into H): a copy, or fp32 -> bf16 round-to-nearest-even.
 *   orc_bf16_encode /   bf16 <-> fp64 from the IEEE-754 bit layout (8 exponent
 *   orc_bf16_decode     bits, 7 stored fraction bits), round-to-nearest-even.
 *
 * Data types: 0 = bf16 (uint16 bit patterns), 1 = fp32, 2 = fp64 (oracle-only
 * output type used by the self-tests).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_BF16 0
#define ORC_FP32 1
#define ORC_FP64 2

/* ---------------------------------------------------------------- bf16 --- */

double orc_bf16_decode(uint16_t h) {
    /* A bf16 value is the upper half of the binary32 with the same bits. */
    uint32_t bits = (uint32_t)h << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

uint16_t orc_bf16_encode(double x) {
    if (isnan(x)) return 0x7FC0;
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (isinf(a)) return sign | 0x7F80;
    if (a == 0.0) return sign;
    int e;
    frexp(a, &e); /* a lies in [2^(e-1), 2^e) */
    /* A normal bf16 carries 8 significant bits, so in that binade the spacing
     * is 2^(e-1-7) = 2^(e-8). Below 2^-126 the spacing stays at 2^-133 (the
     * subnormal range). */
    int q = e - 8;
    if (q < -133) q = -133;
    double r = ldexp(a, -q); /* exact: scaling by a power of two */
    double fl = floor(r);
    double frac = r - fl; /* exact */
    if (frac > 0.5 || (frac == 0.5 && fmod(fl, 2.0) != 0.0)) fl += 1.0;
    double v = ldexp(fl, q);
    if (v > 0x1.FEp127) return sign | 0x7F80; /* past the largest finite bf16 */
    float f = (float)v;                         /* exact: v has <= 8 bits */
    uint32_t bits;
    memcpy(&bits, &f, sizeof bits);
    return sign | (uint16_t)(bits >> 16);
}

static double load_elem(const void* p, int dtype, int64_t i) {
    switch (dtype) {
    case ORC_BF16: return orc_bf16_decode(((const uint16_t*)p)[i]);
    case ORC_FP32: return (double)((const float*)p)[i];
    default: return ((const double*)p)[i];
    }
}

static void store_elem(void* p, int dtype, int64_t i, double v) {
    switch (dtype) {
    case ORC_BF16: ((uint16_t*)p)[i] = orc_bf16_encode(v); break;
    case ORC_FP32: ((float*)p)[i] = (float)v; break; /* C conversion: RNE */
    default: ((double*)p)[i] = v; break;
    }
}

/* ------------------------------------------------------------ schedule --- */

int orc_full_schedule(int T, int r, int s0, int s1, int K, unsigned char* is_full) {
    if (T <= 0 || r <= 0 || s0 < 0 || s1 < 0 || K < 0 || !is_full) return -1;
    int count = 0, hist = 0;
    for (int s = 0; s < T; ++s) {
        /* s is in F when it lies outside [s0, T-1-s1] or r divides s - s0. */
        int outside = (s < s0) || (s > T - 1 - s1);
        int full = outside || ((s - s0) % r == 0);
        /* A step whose history holds fewer than K entries cannot be
         * extrapolated; it is computed fully (and so pushed). */
        if (hist < K) full = 1;
        is_full[s] = (unsigned char)full;
        if (full) {
            ++count;
            if (hist < K) ++hist;
        }
    }
    return count;
}

void orc_normalize(const double* t, int n, double t_min, double t_max, double* tau) {
    for (int i = 0; i < n; ++i) tau[i] = 2.0 * (t[i] - t_min) / (t_max - t_min) - 1.0;
}

/* ------------------------------------------------------------- weights --- */

double orc_nodal(const double* x, int n, double xq) {
    double w = 1.0;
    for (int k = 0; k < n; ++k) w *= (xq - x[k]);
    return w;
}

int orc_rho(const double* x, int n, double* rho) {
    for (int j = 0; j < n; ++j) {
        double d = 1.0;
        for (int k = 0; k < n; ++k)
            if (k != j) d *= (x[j] - x[k]);
        if (d == 0.0) return -1; /* duplicate nodes */
        rho[j] = 1.0 / d;
    }
    return 0;
}

int orc_bary_coeff(const double* x, const double* rho, int n, double xq, double* w) {
    for (int j = 0; j < n; ++j) {
        if (xq == x[j]) { /* the target is a node: the interpolant is h(x_j) */
            for (int i = 0; i < n; ++i) w[i] = (i == j) ? 1.0 : 0.0;
            return 0;
        }
    }
    double den = 0.0;
    for (int i = 0; i < n; ++i) den += rho[i] / (xq - x[i]);
    for (int j = 0; j < n; ++j) w[j] = (rho[j] / (xq - x[j])) / den;
    return 0;
}

int orc_lagrange_basis(const double* x, int n, double xq, double* l) {
    for (int j = 0; j < n; ++j) {
        double p = 1.0;
        for (int k = 0; k < n; ++k) {
            if (k == j) continue;
            if (x[j] == x[k]) return -1;
            p *= (xq - x[k]) / (x[j] - x[k]);
        }
        l[j] = p;
    }
    return 0;
}

/* Weight of node j (0 = oldest) in the truncated Taylor series about the
 * newest node: each backward difference nabla^i f_n = sum_k (-1)^k C(i,k)
 * f_{n-k} is spread over the nodes it touches. Plain nested loops; C(i,k) and
 * i! from their products. */
int orc_taylor_weights(const double* x, int n, double xq, double* w) {
    if (n < 1) return -1;
    double h = n >= 2 ? x[n - 1] - x[n - 2] : 1.0;
    if (n >= 2 && h == 0.0) return -1;
    double theta = n >= 2 ? (xq - x[n - 1]) / h : 0.0;
    for (int j = 0; j < n; ++j) w[j] = 0.0;
    for (int i = 0; i < n; ++i) {
        double fact = 1.0, pw = 1.0;
        for (int q = 1; q <= i; ++q) {
            fact *= q;
            pw *= theta;
        }
        for (int k = 0; k <= i; ++k) {
            double c = 1.0; /* C(i, k) = i! / (k! (i-k)!) */
            for (int q = 1; q <= k; ++q) c = c * (i - k + q) / q;
            double sign = (k % 2 == 0) ? 1.0 : -1.0;
            w[n - 1 - k] += pw / fact * sign * c;
        }
    }
    return 0;
}

/* ---------------------------------------------------------- cache write --- */

void orc_convert(const void* src, int src_dtype, int64_t n, void* dst, int dst_dtype) {
    for (int64_t i = 0; i < n; ++i) {
        if (src_dtype == ORC_BF16 && dst_dtype == ORC_BF16)
            ((uint16_t*)dst)[i] = ((const uint16_t*)src)[i]; /* bit copy */
        else
            store_elem(dst, dst_dtype, i, load_elem(src, src_dtype, i));
    }
}

/* -------------------------------------------------------- extrapolation --- */

typedef struct {
    int K, nb;
    const void* const* F; /* nb*K pointers: F[b*K + j], j oldest .. newest */
    int f_dtype;
    const double* w; /* K weights, same order as j */
    const void* X;   /* residual hidden state or NULL */
    int x_dtype;
    void* const* outs; /* nb pointers, entries may be NULL */
    int out_dtype;
    void* resid_out; /* NULL when no residual is written */
    int resid_dtype;
    const double* const* G; /* nb per-element gate arrays (NULL array or entry: 1) */
    int64_t begin, end;
} orc_job;

static void* orc_extrapolate_range(void* arg) {
    const orc_job* J = (const orc_job*)arg;
    for (int64_t e = J->begin; e < J->end; ++e) {
        double total = J->X ? load_elem(J->X, J->x_dtype, e) : 0.0;
        for (int b = 0; b < J->nb; ++b) {
            double p = 0.0;
            for (int j = 0; j < J->K; ++j) p += J->w[j] * load_elem(J->F[b * J->K + j], J->f_dtype, e);
            if (J->outs && J->outs[b]) store_elem(J->outs[b], J->out_dtype, e, p);
            total += (J->G && J->G[b]) ? J->G[b][e] * p : p; /* gated residual, Sec. 3.1 */
        }
        if (J->resid_out) store_elem(J->resid_out, J->resid_dtype, e, total);
    }
    return NULL;
}

int orc_extrapolate_gated(int K, int nb, const void* const* F, int f_dtype, const double* w,
                          const void* X, int x_dtype, int64_t n, void* const* outs, int out_dtype,
                          void* resid_out, int resid_dtype, const double* const* G, int nthreads);

int orc_extrapolate(int K, int nb, const void* const* F, int f_dtype, const double* w,
                    const void* X, int x_dtype, int64_t n, void* const* outs, int out_dtype,
                    void* resid_out, int resid_dtype, int nthreads) {
    return orc_extrapolate_gated(K, nb, F, f_dtype, w, X, x_dtype, n, outs, out_dtype, resid_out,
                                 resid_dtype, NULL, nthreads);
}

int orc_extrapolate_gated(int K, int nb, const void* const* F, int f_dtype, const double* w,
                          const void* X, int x_dtype, int64_t n, void* const* outs, int out_dtype,
                          void* resid_out, int resid_dtype, const double* const* G, int nthreads) {
    if (K <= 0 || nb <= 0 || !F || !w || n < 0) return -1;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    orc_job jobs[256];
    pthread_t tid[256];
    int64_t chunk = (n + nthreads - 1) / nthreads;
    for (int t = 0; t < nthreads; ++t) {
        orc_job* J = &jobs[t];
        J->K = K; J->nb = nb; J->F = F; J->f_dtype = f_dtype; J->w = w;
        J->X = X; J->x_dtype = x_dtype; J->outs = outs; J->out_dtype = out_dtype;
        J->resid_out = resid_out; J->resid_dtype = resid_dtype; J->G = G;
        J->begin = t * chunk < n ? t * chunk : n;
        J->end = (t + 1) * chunk < n ? (t + 1) * chunk : n;
    }
    if (nthreads == 1) {
        orc_extrapolate_range(&jobs[0]);
        return 0;
    }
    for (int t = 0; t < nthreads; ++t)
        if (pthread_create(&tid[t], NULL, orc_extrapolate_range, &jobs[t]) != 0) {
            for (int u = 0; u < t; ++u) pthread_join(tid[u], NULL);
            return -2;
        }
    for (int t = 0; t < nthreads; ++t) pthread_join(tid[t], NULL);
    return 0;
}
