/*
 * oracle.c -- plain fp64 CPU oracle for the rotated-hypercube mixing layer.
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  Only the test suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load this library.
 * It shares no code, header, table or helper with the CUDA path, and the
 * CUDA path never calls it.
 *
 * What it computes (paper "Reaching Every Position Without Searching",
 * arXiv 2609.18145):
 *
 *   Positions i = 0..n-1 of each sample, n = 2^b, are vertices of a
 *   b-dimensional hypercube (Sec. 3.1).  Layer l wires position i to its
 *   partner p(i) = i XOR 2^s along cube dimension s = l mod b (Sec. 3.1).
 *   Under the causal rule only the earlier endpoint of each link is kept
 *   (Sec. 3.1): position i receives from p(i) exactly when p(i) < i, that
 *   is when bit s of i is set, and then p(i) = i - 2^s, so the link is the
 *   shift x_{i-k} of Eq. (1) with k = 2^s.  Without the causal rule every
 *   position receives from its partner.
 *
 *   Eq. (1): y_i = W_self x_i + W_off x_{i-k}: two d x d linear maps acting
 *   on column vectors.  W_off is called W_nbr here.  Matrices are stored
 *   row-major as W[o][k] (output index o, input index k), so
 *       z[b,i,o] = bias[o] + sum_k W_self[o][k] x[b,i,k]
 *                          + m_i * sum_k W_nbr[o][k] x[b,p(i),k]
 *   with m_i the receive mask above.  The paper states no bias, activation
 *   or residual; they are optional here:
 *       y = act(z) + (RESIDUAL ? x : 0),  act in {identity, ReLU}.
 *   ReLU'(0) is taken as 0.
 *
 *   Backward (derived from the forward by the chain rule, no step of the
 *   paper's):
 *       dz  = dy * act'(z)
 *       dx[b,i,k] = sum_o dz[b,i,o] W_self[o][k]
 *                 + m_{p(i)} * sum_o dz[b,p(i),o] W_nbr[o][k]
 *                 + (RESIDUAL ? dy[b,i,k] : 0)
 *       dW_self[o][k] = sum_{b,i} dz[b,i,o] x[b,i,k]
 *       dW_nbr[o][k]  = sum_{b,i} m_i dz[b,i,o] x[b,p(i),k]
 *       dbias[o]      = sum_{b,i} dz[b,i,o]
 *
 *   Stack (Sec. 3.3, "rot"): layer l of a stack starting at layer index
 *   layer0 uses dimension (layer0 + l) mod b, or a fixed dimension (the
 *   "fixed" control of Sec. 3.3), or an explicit list of layers (the order
 *   variants of Sec. 4, and the schedules of Sec. 3.3 / App. A).  In a list,
 *   an entry s >= 0 is the hypercube link along dimension s ("jump 2^s" of
 *   App. A), and an entry s < 0 is the shift of Eq. (1) itself with distance
 *   k = -s: position i receives x_{i-k} when i >= k, within its sample
 *   ("near" of App. A is k = 1, the "local" schedule of Sec. 3.3).  A shift
 *   always links the earlier position to the later one, so the causal rule
 *   does not change it.
 *
 * Precision: every sum is an fp64 loop in index order.  With round_bf16 set,
 * every stored activation (y, z, dx) is rounded to bfloat16 (round to
 * nearest, ties to even) after it is computed, mirroring a device path that
 * stores activations in bf16; sums stay in fp64.
 *
 * Layout: x, y, z, dy, dx are [B][n][d] row-major; weights [d][d] as above;
 * stacks of weights are [L][d][d]; bias [d] (stacks [L][d]).
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORACLE_CAUSAL   1u
#define ORACLE_RESIDUAL 2u
#define ORACLE_ACT_RELU 4u

int oracle_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

static int log2_exact(int n) {
    int b = 0;
    if (n < 2) return -1;
    while ((1 << b) < n) b++;
    return ((1 << b) == n) ? b : -1;
}

/* Cube dimension used by layer `layer` (Sec. 3.1: l mod b), or the fixed
 * dimension of the "fixed" control (Sec. 3.3) when dim_override >= 0. */
int oracle_dim(int layer, int dim_override, int n) {
    int b = log2_exact(n);
    if (b < 1) return -1;
    if (dim_override >= 0) return dim_override < b ? dim_override : -1;
    return layer % b;
}

/* Partner of position i along dimension s (Sec. 3.1). */
int oracle_partner(int i, int s) { return i ^ (1 << s); }

/* 1 if position i takes its partner's input at dimension s.  Causal rule
 * (Sec. 3.1): keep the link only towards the earlier endpoint, i.e. the
 * partner precedes i. */
int oracle_receives(int i, int s, unsigned flags) {
    if (!(flags & ORACLE_CAUSAL)) return 1;
    return oracle_partner(i, s) < i;
}

/* The link of a layer, s >= 0 (hypercube dimension) or s < 0 (shift by -s).
 * link_partner: the position whose input position i takes at this layer.
 * link_receives: whether position i takes it (n = positions per sample).
 * link_reader: the position that takes x_i as its partner input, or -1. */
static int link_partner(int i, int s) { return s >= 0 ? oracle_partner(i, s) : i + s; }

static int link_receives(int i, int s, int n, unsigned flags) {
    (void)n;
    if (s < 0) return i + s >= 0;
    return oracle_receives(i, s, flags);
}

static int link_reader(int i, int s, int n, unsigned flags) {
    if (s < 0) return (i - s < n) ? i - s : -1;
    int p = oracle_partner(i, s);
    return oracle_receives(p, s, flags) ? p : -1;
}

/* partner[i] = p(i) if position i receives at this layer, else -1. */
int oracle_partner_table(int layer, int dim_override, int n, unsigned flags, int* partner) {
    int s = oracle_dim(layer, dim_override, n);
    if (s < 0) return -1;
    for (int i = 0; i < n; i++)
        partner[i] = oracle_receives(i, s, flags) ? oracle_partner(i, s) : -1;
    return 0;
}

/* Round to the nearest bfloat16 value (8 significant bits, exponent range of
 * IEEE binary32), ties to even.  Written from the format's definition. */
double oracle_round_bf16(double v) {
    if (isnan(v) || isinf(v) || v == 0.0) return v;
    double a = fabs(v);
    int e;
    double r;
    if (a < ldexp(1.0, -126)) {
        /* subnormal range: fixed quantum 2^-133 */
        r = nearbyint(a * ldexp(1.0, 133)) * ldexp(1.0, -133);
    } else {
        double m = frexp(a, &e);          /* a = m * 2^e, 0.5 <= m < 1 */
        r = ldexp(nearbyint(ldexp(m, 8)), e - 8);
        /* largest finite bf16 is (2 - 2^-7) * 2^127 */
        if (r > ldexp(255.0, 120)) r = INFINITY;
    }
    return v < 0 ? -r : r;
}

/* oracle_round_bf16 applied to each of a[0 .. count) in place. */
void oracle_round_bf16_array(double* a, long long count) {
    for (long long i = 0; i < count; ++i) a[i] = oracle_round_bf16(a[i]);
}

static double act_fwd(double z, unsigned flags) {
    if (flags & ORACLE_ACT_RELU) return z > 0.0 ? z : 0.0;
    return z;
}

static double act_grad(double z, unsigned flags) {
    if (flags & ORACLE_ACT_RELU) return z > 0.0 ? 1.0 : 0.0;
    return 1.0;
}

/* One layer forward with link s (see link_partner).  z_out may be NULL. */
static void layer_fwd_dim(const double* x, const double* Ws, const double* Wn,
                          const double* bias, int s, int B, int n, int d,
                          unsigned flags, int round_bf16, double* y, double* z_out) {
    long long rows = (long long)B * n;
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
    for (long long r = 0; r < rows; r++) {
        int b = (int)(r / n), i = (int)(r % n);
        const double* xi = x + ((size_t)b * n + i) * d;
        int recv = link_receives(i, s, n, flags);
        const double* xp = recv ? x + ((size_t)b * n + link_partner(i, s)) * d : NULL;
        for (int o = 0; o < d; o++) {
            double z = bias ? bias[o] : 0.0;
            for (int k = 0; k < d; k++) z += Ws[(size_t)o * d + k] * xi[k];
            if (recv)
                for (int k = 0; k < d; k++) z += Wn[(size_t)o * d + k] * xp[k];
            double out = act_fwd(z, flags);
            if (flags & ORACLE_RESIDUAL) out += xi[o];
            if (round_bf16) {
                out = oracle_round_bf16(out);
                z = oracle_round_bf16(z);       /* the stored copy of z */
            }
            y[((size_t)b * n + i) * d + o] = out;
            if (z_out) z_out[((size_t)b * n + i) * d + o] = z;
        }
    }
}

/* One layer backward with link s.  z may be NULL when no activation is
 * used.  dW_self, dW_nbr, dbias may each be NULL. */
static void layer_bwd_dim(const double* x, const double* z, const double* dy,
                          const double* Ws, const double* Wn, int s, int B, int n, int d,
                          unsigned flags, int round_bf16, double* dx,
                          double* dWs, double* dWn, double* dbias) {
    size_t total = (size_t)B * n * d;
    double* dz = (double*)malloc(total * sizeof(double));
    for (size_t t = 0; t < total; t++)
        dz[t] = dy[t] * ((flags & ORACLE_ACT_RELU) ? act_grad(z[t], flags) : 1.0);

    long long rows = (long long)B * n;
    if (dx) {
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
        for (long long r = 0; r < rows; r++) {
            int b = (int)(r / n), i = (int)(r % n);
            int j = link_reader(i, s, n, flags);          /* who reads x_i, if anyone */
            const double* dzi = dz + ((size_t)b * n + i) * d;
            const double* dzj = j >= 0 ? dz + ((size_t)b * n + j) * d : NULL;
            for (int k = 0; k < d; k++) {
                double g = 0.0;
                for (int o = 0; o < d; o++) g += dzi[o] * Ws[(size_t)o * d + k];
                if (dzj)
                    for (int o = 0; o < d; o++) g += dzj[o] * Wn[(size_t)o * d + k];
                if (flags & ORACLE_RESIDUAL) g += dy[((size_t)b * n + i) * d + k];
                if (round_bf16) g = oracle_round_bf16(g);
                dx[((size_t)b * n + i) * d + k] = g;
            }
        }
    }
    if (dWs || dWn) {
#ifdef _OPENMP
#pragma omp parallel for schedule(static)
#endif
        for (int o = 0; o < d; o++) {
            for (int k = 0; k < d; k++) {
                double gs = 0.0, gn = 0.0;
                for (long long r = 0; r < rows; r++) {
                    int b = (int)(r / n), i = (int)(r % n);
                    double dzo = dz[((size_t)b * n + i) * d + o];
                    gs += dzo * x[((size_t)b * n + i) * d + k];
                    if (link_receives(i, s, n, flags))
                        gn += dzo * x[((size_t)b * n + link_partner(i, s)) * d + k];
                }
                if (dWs) dWs[(size_t)o * d + k] = gs;
                if (dWn) dWn[(size_t)o * d + k] = gn;
            }
        }
    }
    if (dbias) {
        for (int o = 0; o < d; o++) {
            double g = 0.0;
            for (long long r = 0; r < rows; r++) g += dz[(size_t)r * d + o];
            dbias[o] = g;
        }
    }
    free(dz);
}

int oracle_layer_fwd(const double* x, const double* Ws, const double* Wn, const double* bias,
                     int layer, int dim_override, int B, int n, int d, unsigned flags,
                     int round_bf16, double* y, double* z_out) {
    int s = oracle_dim(layer, dim_override, n);
    if (s < 0 || B < 0 || d < 1) return -1;
    layer_fwd_dim(x, Ws, Wn, bias, s, B, n, d, flags, round_bf16, y, z_out);
    return 0;
}

int oracle_layer_bwd(const double* x, const double* z, const double* dy,
                     const double* Ws, const double* Wn, int layer, int dim_override,
                     int B, int n, int d, unsigned flags, int round_bf16,
                     double* dx, double* dWs, double* dWn, double* dbias) {
    int s = oracle_dim(layer, dim_override, n);
    if (s < 0 || B < 0 || d < 1) return -1;
    if ((flags & ORACLE_ACT_RELU) && !z) return -1;
    layer_bwd_dim(x, z, dy, Ws, Wn, s, B, n, d, flags, round_bf16, dx, dWs, dWn, dbias);
    return 0;
}

/* Marker of an invalid layer (a shift is a negative link). */
#define NO_LINK (-(1 << 30))

/* Link of stack layer l: dims[l] if a schedule is given (a dimension in
 * [0, b) or a shift -k with 1 <= k < n), else the rotated (or fixed) rule
 * applied to layer index layer0 + l; NO_LINK if invalid. */
static int stack_dim(const int* dims, int layer0, int l, int dim_override, int n) {
    int b = log2_exact(n);
    if (b < 1) return NO_LINK;
    if (dims) {
        if (dims[l] >= 0) return dims[l] < b ? dims[l] : NO_LINK;
        return -dims[l] < n ? dims[l] : NO_LINK;
    }
    int s = oracle_dim(layer0 + l, dim_override, n);
    return s >= 0 ? s : NO_LINK;
}

/* Stack forward.  acts [L][B][n][d] receives each layer's input (acts[0] is
 * a copy of x); zs [L][B][n][d] each layer's pre-activation (may be NULL);
 * y the last layer's output.  bias may be NULL (no bias in any layer). */
int oracle_stack_fwd(const double* x, const double* Ws, const double* Wn, const double* bias,
                     const int* dims, int layer0, int L, int dim_override,
                     int B, int n, int d, unsigned flags, int round_bf16,
                     double* y, double* acts, double* zs) {
    size_t act = (size_t)B * n * d;
    if (L < 1) return -1;
    for (int l = 0; l < L; l++)
        if (stack_dim(dims, layer0, l, dim_override, n) == NO_LINK) return -1;
    memcpy(acts, x, act * sizeof(double));
    for (int l = 0; l < L; l++) {
        int s = stack_dim(dims, layer0, l, dim_override, n);
        double* out = (l + 1 < L) ? acts + (size_t)(l + 1) * act : y;
        layer_fwd_dim(acts + (size_t)l * act, Ws + (size_t)l * d * d, Wn + (size_t)l * d * d,
                      bias ? bias + (size_t)l * d : NULL, s, B, n, d, flags, round_bf16, out,
                      zs ? zs + (size_t)l * act : NULL);
    }
    return 0;
}

/* Stack backward from the saved layer inputs `acts` and pre-activations
 * `zs` of oracle_stack_fwd.  Writes dx (gradient of the stack input) and the
 * per-layer weight gradients dWs, dWn [L][d][d] and dbias [L][d] (may be
 * NULL). */
int oracle_stack_bwd(const double* acts, const double* zs, const double* dy,
                     const double* Ws, const double* Wn, const int* dims, int layer0, int L,
                     int dim_override, int B, int n, int d, unsigned flags, int round_bf16,
                     double* dx, double* dWs, double* dWn, double* dbias) {
    size_t act = (size_t)B * n * d;
    if (L < 1) return -1;
    if ((flags & ORACLE_ACT_RELU) && !zs) return -1;
    double* g = (double*)malloc(act * sizeof(double));
    double* g_next = (double*)malloc(act * sizeof(double));
    memcpy(g, dy, act * sizeof(double));
    for (int l = L - 1; l >= 0; l--) {
        int s = stack_dim(dims, layer0, l, dim_override, n);
        if (s == NO_LINK) { free(g); free(g_next); return -1; }
        layer_bwd_dim(acts + (size_t)l * act, zs ? zs + (size_t)l * act : NULL, g,
                      Ws + (size_t)l * d * d, Wn + (size_t)l * d * d, s, B, n, d, flags,
                      round_bf16, g_next, dWs + (size_t)l * d * d, dWn + (size_t)l * d * d,
                      dbias ? dbias + (size_t)l * d : NULL);
        double* t = g; g = g_next; g_next = t;
    }
    memcpy(dx, g, act * sizeof(double));
    free(g);
    free(g_next);
    return 0;
}
