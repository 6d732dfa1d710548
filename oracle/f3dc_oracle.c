/*
 * Fast3Dcache CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * Only the test suite, the smoke check and the CPU-baseline / reference legs
 * of the benchmark may load this library.  The product path (the CUDA
 * library and its Python binding) never calls it and shares no code with it.
 *
 * A plain, slow, obviously-correct restatement of what the paper defines:
 *   - shifted time schedule                     (Supp. Sec. D, eq. for t)
 *   - three-phase cache budget, PCSC            (Sec. 4.2 eqs. for log dS, dS_hat, c_t;
 *                                                Sec. 4.3; Algorithm 1 step 1)
 *   - error-accumulation elimination tau        (Sec. 4.3 Phase 2; Algorithm 1 SSC)
 *   - SSC score and lowest-c selection          (Sec. 4.1 V_i, Eq. ICE; Sec. 4.2 Eq. ssc,
 *                                                Eq. normalize; Algorithm 1 SSC)
 *   - flow transformer on the active subset     (Sec. 4.2 token compaction; Supp. Sec. F
 *                                                block structure: adaLN, self-attention,
 *                                                LayerNorm, cross-attention, MLP)
 *   - cache merge and rectified-flow Euler step (Algorithm 1 step 3; Sec. 3.1)
 *   - dynamic-voxel count                       (Sec. 4.1 Eq. 1)
 *   - data-driven PCSC slope (RANSAC, median)   (Supp. "Data-driven Parameter Selection")
 *   - classifier-free guidance in its interval  (Sec. 4.3 Phase 3 "CFG-free";
 *                                                Supp. Sec. D CFG interval t in [0.5, 1])
 *   - the whole sampler                         (Algorithm 1)
 *
 * Precision: the SSC score, the selection order, the Euler update and the
 * occupancy logits are fp32 in the stated operation order (each + and * rounds;
 * compile with -ffp-contract=off), because they decide integers or must be
 * reproduced bit for bit.  The transformer keeps fp32 tensors and accumulates
 * every dot product and reduction in fp64.
 *
 * Architecture details the paper leaves open are fixed as readings (pos-emb,
 * t-embedding, QK RMSNorm, eps, GELU form); each is named where it is used.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_LN_EPS 1e-6
#define ORC_ALIGN 64

/* ------------------------------------------------------------------------ */
/* bf16 storage helpers (format conversion only)                            */
/* ------------------------------------------------------------------------ */
static float bf2f(uint16_t u)
{
    uint32_t x = (uint32_t)u << 16;
    float f;
    memcpy(&f, &x, 4);
    return f;
}

static uint16_t f2bf(float f)
{
    uint32_t x;
    memcpy(&x, &f, 4);
    if (isnan(f)) return 0x7FC0;
    uint32_t rounding = ((x >> 16) & 1u) + 0x7FFFu; /* round to nearest even */
    return (uint16_t)((x + rounding) >> 16);
}

uint16_t orc_f32_to_bf16(float f) { return f2bf(f); }

/* ------------------------------------------------------------------------ */
/* Supp. Sec. D: shifted schedule t = eta t_l / (1 + (eta - 1) t_l),         */
/* t_l uniform from 1 (noise) to 0 (data).  t_out[k-1] = t_k, k = 1..T+1.    */
/* ------------------------------------------------------------------------ */
void orc_time_schedule(int T, double eta, float *t_out)
{
    for (int k = 1; k <= T + 1; ++k) {
        double tl = 1.0 - (double)(k - 1) / (double)T;
        double t = eta * tl / (1.0 + (eta - 1.0) * tl);
        t_out[k - 1] = (float)t;
    }
}

/* ceil(T * rho): the anchor step (Sec. 4.2) and the CFG-off step (Alg. 1). */
int orc_ceil_steps(int T, double rho) { return (int)ceil((double)T * rho); }

/* ------------------------------------------------------------------------ */
/* Algorithm 1, step 1 (cache budget c_t by phase), with PCSC (Sec. 4.2):   */
/*   dS_hat_k = sigma * exp(mu (k - k_a)),  c_k = N - dS_hat_k / gamma_up,  */
/* floored (c_t is an upper bound on cached tokens) and clamped to [0, N].  */
/* Phase 3: c = floor(N xi), except every f_corr-th step (k_r + 1 = 0 mod   */
/* f_corr, k_r = k - k_off) which is a full correction step; f_corr <= 0    */
/* disables the correction.  Returns the number of tokens to CACHE.         */
/* ------------------------------------------------------------------------ */
int orc_phase_quota(int N, int T, double rho_a, double rho_off, double mu, double xi,
                    int f_corr, int gamma_up, double sigma, int k, int *phase_out)
{
    int ka = orc_ceil_steps(T, rho_a);
    int koff = orc_ceil_steps(T, rho_off);
    int phase, c;
    if (k <= ka) {
        phase = 1;
        c = 0;
    } else if (k < koff) {
        phase = 2;
        double ds = sigma * exp(mu * (double)(k - ka));
        double cd = floor((double)N - ds / (double)gamma_up);
        if (!(cd > 0.0)) cd = 0.0; /* also maps NaN to 0 (no caching) */
        if (cd > (double)N) cd = (double)N;
        c = (int)cd;
    } else {
        phase = 3;
        int kr = k - koff;
        if (f_corr > 0 && (kr + 1) % f_corr == 0) {
            c = 0;
        } else {
            double cd = floor((double)N * xi);
            if (!(cd > 0.0)) cd = 0.0;
            if (cd > (double)N) cd = (double)N;
            c = (int)cd;
        }
    }
    if (phase_out) *phase_out = phase;
    return c;
}

/* ------------------------------------------------------------------------ */
/* Error-accumulation elimination (Sec. 4.3 Phase 2; Alg. 1 SSC):           */
/* mode 0 (period reading): at most tau-1 consecutive cached steps, then a  */
/*        forced full step, i.e. one full refresh every tau steps;          */
/* mode 1 (literal reading): force a full step once consec >= tau.         */
/* tau <= 0 disables the rule.  *consec counts the consecutive cached steps */
/* before this one and is updated.  Returns the effective cache quota.      */
/* ------------------------------------------------------------------------ */
int orc_tau_gate(int quota, int tau, int mode, int *consec)
{
    if (quota > 0 && tau > 0) {
        int limit = (mode == 0) ? tau - 1 : tau;
        if (*consec >= limit) quota = 0;
    }
    if (quota > 0) *consec += 1;
    else *consec = 0;
    return quota;
}

/* ------------------------------------------------------------------------ */
/* SSC cache-ability score (Sec. 4.1, 4.2):                                 */
/*   V_i = ||v_i(t-1)||_2,  A_i = ||v_i(t-1) - v_i(t-2)||_2,                 */
/*   norm(X_i) = (X_i - min_j X_j) / (max_j X_j - min_j X_j),               */
/*   C_i = w norm(A_i) + (1 - w) norm(V_i).                                 */
/* fp32, channel sums in order 0..C-1 (one rounding per + and *), correctly */
/* rounded sqrt and division.  min / max skip NaN; a NaN stays NaN; when    */
/* max <= min (degenerate range) every non-NaN norm is 0.                   */
/* ------------------------------------------------------------------------ */
static float orc_norm1(float x, float mn, float mx)
{
    if (isnan(x)) return x;
    if (!(mx > mn)) return 0.0f;
    float num = x - mn;
    float den = mx - mn;
    return num / den;
}

/*
 * Variant (SSC with three predictions): v3 = v_i(t-3) non-NULL replaces the
 * first difference by the second difference of the velocity,
 *   A_i = ||(v_i(t-1) - v_i(t-2)) - (v_i(t-2) - v_i(t-3))||_2,
 * the discrete rate of change of Sec. 4.1's acceleration; each channel's
 * term is (x - y) - (y - z), two subtractions then one, in fp32.
 */
void orc_ssc_score3(const uint16_t *v1, const uint16_t *v2, const uint16_t *v3, int N, int C, double omega,
                    float *score)
{
    float *V = (float *)malloc(sizeof(float) * (size_t)(N > 0 ? N : 1));
    float *A = (float *)malloc(sizeof(float) * (size_t)(N > 0 ? N : 1));
    float mnV = INFINITY, mxV = -INFINITY, mnA = INFINITY, mxA = -INFINITY;
    for (int i = 0; i < N; ++i) {
        float sv = 0.0f, sa = 0.0f;
        for (int c = 0; c < C; ++c) {
            float x = bf2f(v1[(size_t)i * C + c]);
            float y = bf2f(v2[(size_t)i * C + c]);
            float d = x - y;
            if (v3) {
                float z = bf2f(v3[(size_t)i * C + c]);
                float e = y - z;
                d = d - e;
            }
            float xx = x * x;
            float dd = d * d;
            sv = sv + xx;
            sa = sa + dd;
        }
        V[i] = sqrtf(sv);
        A[i] = sqrtf(sa);
        if (V[i] < mnV) mnV = V[i];
        if (V[i] > mxV) mxV = V[i];
        if (A[i] < mnA) mnA = A[i];
        if (A[i] > mxA) mxA = A[i];
    }
    float wa = (float)omega;
    float wv = 1.0f - wa;
    for (int i = 0; i < N; ++i) {
        float na = orc_norm1(A[i], mnA, mxA);
        float nv = orc_norm1(V[i], mnV, mxV);
        float ta = wa * na;
        float tv = wv * nv;
        score[i] = ta + tv;
    }
    free(V);
    free(A);
}

void orc_ssc_score(const uint16_t *v1, const uint16_t *v2, int N, int C, double omega, float *score)
{
    orc_ssc_score3(v1, v2, NULL, N, C, omega, score);
}

/* ------------------------------------------------------------------------ */
/* Alg. 1 SSC: I_cache = the c tokens with the lowest C_i; I_active = the   */
/* rest, listed in ascending index.  Total order: lower score first, equal  */
/* scores by lower index, NaN scores after every number (never cached).     */
/* ------------------------------------------------------------------------ */
static const float *g_sort_scores; /* qsort context (single-threaded use) */

static int orc_precedes(float sa, int a, float sb, int b)
{
    int na = isnan(sa), nb = isnan(sb);
    if (na != nb) return nb;
    if (!na && sa != sb) return sa < sb;
    return a < b;
}

static int orc_cmp(const void *pa, const void *pb)
{
    int a = *(const int *)pa, b = *(const int *)pb;
    if (a == b) return 0;
    return orc_precedes(g_sort_scores[a], a, g_sort_scores[b], b) ? -1 : 1;
}

int orc_select(const float *score, int N, int c, uint8_t *cached, int32_t *active_idx)
{
    if (c < 0) c = 0;
    if (c > N) c = N;
    int *order = (int *)malloc(sizeof(int) * (size_t)(N > 0 ? N : 1));
    for (int i = 0; i < N; ++i) order[i] = i;
    g_sort_scores = score;
    qsort(order, (size_t)N, sizeof(int), orc_cmp);
    for (int r = 0; r < N; ++r) cached[order[r]] = (uint8_t)(r < c);
    int na = 0;
    for (int i = 0; i < N; ++i)
        if (!cached[i]) active_idx[na++] = i;
    free(order);
    return na;
}

/* ------------------------------------------------------------------------ */
/* Sec. 4.1 Eq. 1: decoded occupancy and dynamic voxels.                    */
/* Stand-in decoder (reading; the TRELLIS decoder is not given): sub-voxel  */
/* j of token i has logit sum_c S_ic W_dec[c, j] (fp32, c in order, one     */
/* rounding per op) and is occupied iff logit > 0.                          */
/* ------------------------------------------------------------------------ */
void orc_occupancy(const float *S, int N, int C, const uint16_t *dec_w, int G, uint8_t *occ)
{
    for (int i = 0; i < N; ++i) {
        for (int j = 0; j < G; ++j) {
            float l = 0.0f;
            for (int c = 0; c < C; ++c) {
                float p = S[(size_t)i * C + c] * bf2f(dec_w[(size_t)c * G + j]);
                l = l + p;
            }
            occ[(size_t)i * G + j] = (uint8_t)(l > 0.0f);
        }
    }
}

long long orc_dynamic_voxels(const uint8_t *occ_a, const uint8_t *occ_b, long long n)
{
    long long s = 0;
    for (long long q = 0; q < n; ++q) s += (occ_a[q] ^ occ_b[q]) & 1;
    return s;
}

/* ------------------------------------------------------------------------ */
/* Alg. 1 step 3: v_t <- v_cache; v_t[I_active] <- v_active;                */
/* S <- S - (t - t_prev) v_t  (dt = t - t_prev, one fp32 mul then one sub). */
/* The velocity history is bf16; fresh velocities are rounded to nearest    */
/* even before they are stored and used, so a cached token carries its      */
/* stored velocity bit for bit.                                             */
/* ------------------------------------------------------------------------ */
void orc_merge_euler(int N, int C, const int32_t *active_idx, int a, const float *v_active,
                     const uint16_t *v_cache, float dt, float *S, uint16_t *v_t)
{
    for (long long q = 0; q < (long long)N * C; ++q) v_t[q] = v_cache[q];
    for (int r = 0; r < a; ++r) {
        int i = active_idx[r];
        for (int c = 0; c < C; ++c) v_t[(size_t)i * C + c] = f2bf(v_active[(size_t)r * C + c]);
    }
    for (long long q = 0; q < (long long)N * C; ++q) {
        float step = dt * bf2f(v_t[q]);
        S[q] = S[q] - step;
    }
}

/* ------------------------------------------------------------------------ */
/* Classifier-free guidance.  The sampler guides the steps whose start time */
/* lies in the CFG interval [t_lo, 1] (Supp. Sec. D: TRELLIS's flow         */
/* sampler applies CFG for t in [0.5, 1]; Phase 3 is the CFG-free stage).   */
/* The guided velocity moves from the unconditional prediction towards the  */
/* conditional one by the strength s: v = v_u + s (v_c - v_u), in fp32:     */
/* one subtraction, one multiplication by (float)s, one addition.           */
/* ------------------------------------------------------------------------ */
int orc_cfg_on(int T, double eta, double t_lo, int k)
{
    float *t = (float *)malloc(sizeof(float) * (size_t)(T + 1));
    orc_time_schedule(T, eta, t);
    const int on = (double)t[k - 1] >= t_lo;
    free(t);
    return on;
}

void orc_cfg_combine(long long n, const float *v_c, const float *v_u, double s, float *v)
{
    const float sf = (float)s;
    for (long long q = 0; q < n; ++q) {
        const float d = v_c[q] - v_u[q];
        const float g = sf * d;
        v[q] = v_u[q] + g;
    }
}

/* ======================================================================== */
/* Flow transformer (Supp. Sec. F block structure) on an active subset.     */
/* ======================================================================== */
typedef struct {
    int grid, C, W, L, H, mlp, Nc, Dc, G;
    /* globals */
    float *in_w, *in_b, *t_w1, *t_b1, *t_w2, *t_b2, *fmod_w, *fmod_b, *out_w, *out_b;
    uint16_t *dec_w;
    /* per block */
    float **mod_w, **mod_b, **qkv_w, **qkv_b, **qn_g, **kn_g, **o_w, **o_b, **ln2_g, **ln2_b;
    float **cq_w, **cq_b, **ckv_w, **ckv_b, **co_w, **co_b, **fc1_w, **fc1_b, **fc2_w, **fc2_b;
    /* convolutional stand-in decoder */
    uint16_t *dc1_w, *dc1_b, *dc2_w, *dc2_b, *dc3_w, *dc3_b;
} orc_model;

static float *take(const uint16_t *blob, size_t *pos, size_t n)
{
    float *t = (float *)malloc(sizeof(float) * n);
    for (size_t q = 0; q < n; ++q) t[q] = bf2f(blob[*pos + q]);
    *pos += (n + ORC_ALIGN - 1) / ORC_ALIGN * ORC_ALIGN;
    return t;
}

static uint16_t *take_bits(const uint16_t *blob, size_t *pos, size_t n)
{
    uint16_t *t = (uint16_t *)malloc(sizeof(uint16_t) * n);
    memcpy(t, blob + *pos, sizeof(uint16_t) * n);
    *pos += (n + ORC_ALIGN - 1) / ORC_ALIGN * ORC_ALIGN;
    return t;
}

/* Weight blob layout version 2: bf16, nn.Linear [out, in] row-major, in the
 * order below, each tensor starting at a multiple of 64 elements. */
void *orc_model_create(int grid, int C, int W, int L, int H, int mlp, int Nc, int Dc, int G,
                       const uint16_t *blob)
{
    orc_model *m = (orc_model *)calloc(1, sizeof(orc_model));
    m->grid = grid; m->C = C; m->W = W; m->L = L; m->H = H; m->mlp = mlp;
    m->Nc = Nc; m->Dc = Dc; m->G = G;
    size_t p = 0;
    size_t Wm = (size_t)mlp * W;
    m->in_w = take(blob, &p, (size_t)W * C);
    m->in_b = take(blob, &p, W);
    m->t_w1 = take(blob, &p, (size_t)W * 256);
    m->t_b1 = take(blob, &p, W);
    m->t_w2 = take(blob, &p, (size_t)W * W);
    m->t_b2 = take(blob, &p, W);
#define ALLOC_BLK(f) m->f = (float **)calloc((size_t)L, sizeof(float *))
    ALLOC_BLK(mod_w); ALLOC_BLK(mod_b); ALLOC_BLK(qkv_w); ALLOC_BLK(qkv_b); ALLOC_BLK(qn_g);
    ALLOC_BLK(kn_g); ALLOC_BLK(o_w); ALLOC_BLK(o_b); ALLOC_BLK(ln2_g); ALLOC_BLK(ln2_b);
    ALLOC_BLK(cq_w); ALLOC_BLK(cq_b); ALLOC_BLK(ckv_w); ALLOC_BLK(ckv_b); ALLOC_BLK(co_w);
    ALLOC_BLK(co_b); ALLOC_BLK(fc1_w); ALLOC_BLK(fc1_b); ALLOC_BLK(fc2_w); ALLOC_BLK(fc2_b);
#undef ALLOC_BLK
    for (int l = 0; l < L; ++l) {
        m->mod_w[l] = take(blob, &p, (size_t)6 * W * W);
        m->mod_b[l] = take(blob, &p, (size_t)6 * W);
        m->qkv_w[l] = take(blob, &p, (size_t)3 * W * W);
        m->qkv_b[l] = take(blob, &p, (size_t)3 * W);
        m->qn_g[l] = take(blob, &p, W);
        m->kn_g[l] = take(blob, &p, W);
        m->o_w[l] = take(blob, &p, (size_t)W * W);
        m->o_b[l] = take(blob, &p, W);
        m->ln2_g[l] = take(blob, &p, W);
        m->ln2_b[l] = take(blob, &p, W);
        m->cq_w[l] = take(blob, &p, (size_t)W * W);
        m->cq_b[l] = take(blob, &p, W);
        m->ckv_w[l] = take(blob, &p, (size_t)2 * W * Dc);
        m->ckv_b[l] = take(blob, &p, (size_t)2 * W);
        m->co_w[l] = take(blob, &p, (size_t)W * W);
        m->co_b[l] = take(blob, &p, W);
        m->fc1_w[l] = take(blob, &p, Wm * W);
        m->fc1_b[l] = take(blob, &p, Wm);
        m->fc2_w[l] = take(blob, &p, (size_t)W * Wm);
        m->fc2_b[l] = take(blob, &p, W);
    }
    m->fmod_w = take(blob, &p, (size_t)2 * W * W);
    m->fmod_b = take(blob, &p, (size_t)2 * W);
    m->out_w = take(blob, &p, (size_t)C * W);
    m->out_b = take(blob, &p, C);
    m->dec_w = take_bits(blob, &p, (size_t)C * G);
    m->dc1_w = take_bits(blob, &p, (size_t)16 * C * 27);
    m->dc1_b = take_bits(blob, &p, 16);
    m->dc2_w = take_bits(blob, &p, (size_t)8 * 16 * 27);
    m->dc2_b = take_bits(blob, &p, 8);
    m->dc3_w = take_bits(blob, &p, (size_t)8 * 27);
    m->dc3_b = take_bits(blob, &p, 1);
    return m;
}

void orc_model_free(void *vm)
{
    orc_model *m = (orc_model *)vm;
    if (!m) return;
    free(m->in_w); free(m->in_b); free(m->t_w1); free(m->t_b1); free(m->t_w2); free(m->t_b2);
    free(m->fmod_w); free(m->fmod_b); free(m->out_w); free(m->out_b); free(m->dec_w);
    free(m->dc1_w); free(m->dc1_b); free(m->dc2_w); free(m->dc2_b); free(m->dc3_w); free(m->dc3_b);
    float **blk[] = {m->mod_w, m->mod_b, m->qkv_w, m->qkv_b, m->qn_g, m->kn_g, m->o_w, m->o_b,
                     m->ln2_g, m->ln2_b, m->cq_w, m->cq_b, m->ckv_w, m->ckv_b, m->co_w, m->co_b,
                     m->fc1_w, m->fc1_b, m->fc2_w, m->fc2_b};
    for (size_t q = 0; q < sizeof(blk) / sizeof(blk[0]); ++q) {
        for (int l = 0; l < m->L; ++l) free(blk[q][l]);
        free(blk[q]);
    }
    free(m);
}

/* ---- generic dense ops (fp32 tensors, fp64 accumulation) ---- */

/* y[r, n] = b[n] + sum_k x[r, k] w[n, k]   (nn.Linear, w is [n_out, n_in]) */
void orc_linear(const float *x, int rows, int n_in, const float *w, const float *b, int n_out, float *y)
{
#pragma omp parallel for schedule(static)
    for (int r = 0; r < rows; ++r) {
        const float *xr = x + (size_t)r * n_in;
        for (int n = 0; n < n_out; ++n) {
            const float *wn = w + (size_t)n * n_in;
            double acc = b ? (double)b[n] : 0.0;
            for (int k = 0; k < n_in; ++k) acc += (double)xr[k] * (double)wn[k];
            y[(size_t)r * n_out + n] = (float)acc;
        }
    }
}

/* LayerNorm without affine: (x - mean) / sqrt(var + eps), biased variance. */
void orc_layernorm(const float *x, int rows, int n, float *y)
{
#pragma omp parallel for schedule(static)
    for (int r = 0; r < rows; ++r) {
        const float *xr = x + (size_t)r * n;
        double mean = 0.0;
        for (int k = 0; k < n; ++k) mean += xr[k];
        mean /= n;
        double var = 0.0;
        for (int k = 0; k < n; ++k) var += ((double)xr[k] - mean) * ((double)xr[k] - mean);
        var /= n;
        double rs = 1.0 / sqrt(var + ORC_LN_EPS);
        for (int k = 0; k < n; ++k) y[(size_t)r * n + k] = (float)(((double)xr[k] - mean) * rs);
    }
}

/* GELU, tanh form (reading: the form DiT-style MLPs use). */
static double orc_gelu_tanh(double x)
{
    const double k0 = 0.7978845608028654; /* sqrt(2/pi) */
    return 0.5 * x * (1.0 + tanh(k0 * (x + 0.044715 * x * x * x)));
}

float orc_gelu(float x) { return (float)orc_gelu_tanh(x); }

static double orc_silu(double x) { return x / (1.0 + exp(-x)); }

/* Per-head RMSNorm on rows of width H*dh (reading: qk RMS norm in the self-
 * attention of the sparse-structure flow transformer):                     */
/* y = x / sqrt(mean_d(x^2) + eps) * g.                                     */
static void orc_head_rmsnorm(float *x, int rows, int H, int dh, int row_stride, const float *g)
{
#pragma omp parallel for schedule(static)
    for (int r = 0; r < rows; ++r) {
        for (int h = 0; h < H; ++h) {
            float *v = x + (size_t)r * row_stride + (size_t)h * dh;
            double ss = 0.0;
            for (int d = 0; d < dh; ++d) ss += (double)v[d] * v[d];
            double rs = 1.0 / sqrt(ss / dh + ORC_LN_EPS);
            for (int d = 0; d < dh; ++d) v[d] = (float)((double)v[d] * rs * g[h * dh + d]);
        }
    }
}

/* Multi-head attention, softmax(q k^T / sqrt(dh)) v, per head.
 * q: [nq, *] with head h at columns q_off + h*dh (row stride q_stride);
 * k, v likewise with nk rows.  out: [nq, H*dh]. */
void orc_attention(const float *q, int q_stride, const float *k, int k_stride, const float *v,
                   int v_stride, int nq, int nk, int H, int dh, float *out)
{
    double scale = 1.0 / sqrt((double)dh);
#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * (size_t)(nk > 0 ? nk : 1));
        double *o = (double *)malloc(sizeof(double) * (size_t)dh);
#pragma omp for schedule(static) collapse(2)
        for (int h = 0; h < H; ++h) {
            for (int r = 0; r < nq; ++r) {
                const float *qr = q + (size_t)r * q_stride + (size_t)h * dh;
                double mx = -INFINITY;
                for (int j = 0; j < nk; ++j) {
                    const float *kj = k + (size_t)j * k_stride + (size_t)h * dh;
                    double acc = 0.0;
                    for (int d = 0; d < dh; ++d) acc += (double)qr[d] * (double)kj[d];
                    s[j] = acc * scale;
                    if (s[j] > mx) mx = s[j];
                }
                double l = 0.0;
                for (int j = 0; j < nk; ++j) {
                    s[j] = exp(s[j] - mx);
                    l += s[j];
                }
                for (int d = 0; d < dh; ++d) o[d] = 0.0;
                for (int j = 0; j < nk; ++j) {
                    const float *vj = v + (size_t)j * v_stride + (size_t)h * dh;
                    for (int d = 0; d < dh; ++d) o[d] += s[j] * (double)vj[d];
                }
                for (int d = 0; d < dh; ++d) out[(size_t)r * H * dh + (size_t)h * dh + d] = (float)(o[d] / l);
            }
        }
        free(s);
        free(o);
    }
}

/* Fixed 3-D sin-cos position embedding of token i's grid coordinate
 * (reading): F = W / 6 frequencies w_f = 10000^(-f/F) per axis; for axis a
 * in (d, h, w) the entries a*2F + f = sin(coord_a w_f) and
 * a*2F + F + f = cos(coord_a w_f); the last W - 6F entries are 0.         */
void orc_pos_embed(int grid, int W, int i, float *out)
{
    int F = W / 6;
    int coord[3];
    coord[0] = i / (grid * grid);
    coord[1] = (i / grid) % grid;
    coord[2] = i % grid;
    for (int n = 0; n < W; ++n) out[n] = 0.0f;
    for (int a = 0; a < 3; ++a) {
        for (int f = 0; f < F; ++f) {
            double w = pow(10000.0, -(double)f / (double)F);
            out[a * 2 * F + f] = (float)sin(coord[a] * w);
            out[a * 2 * F + F + f] = (float)cos(coord[a] * w);
        }
    }
}

/* Timestep embedding (reading, DiT style): 256-dim [cos, sin] of 1000 t at
 * frequencies exp(-ln(10000) f / 128), then Linear -> SiLU -> Linear.      */
void orc_time_embed(const void *vm, float t, float *temb)
{
    const orc_model *m = (const orc_model *)vm;
    float freq[256];
    double arg = 1000.0 * (double)t;
    for (int f = 0; f < 128; ++f) {
        double w = exp(-log(10000.0) * (double)f / 128.0);
        freq[f] = (float)cos(arg * w);
        freq[128 + f] = (float)sin(arg * w);
    }
    float *h1 = (float *)malloc(sizeof(float) * (size_t)m->W);
    orc_linear(freq, 1, 256, m->t_w1, m->t_b1, m->W, h1);
    for (int n = 0; n < m->W; ++n) h1[n] = (float)orc_silu(h1[n]);
    orc_linear(h1, 1, m->W, m->t_w2, m->t_b2, m->W, temb);
    free(h1);
}

/* Block modulation (adaLN): mod_l = Linear(SiLU(temb)) -> 6W values in the
 * order shift1, scale1, gate1, shift2, scale2, gate2 (reading: DiT adaLN).
 * block = -1 gives the final layer's (shift, scale), 2W values.           */
void orc_modulation(const void *vm, const float *temb, int block, float *mod)
{
    const orc_model *m = (const orc_model *)vm;
    int W = m->W;
    float *s = (float *)malloc(sizeof(float) * (size_t)W);
    for (int n = 0; n < W; ++n) s[n] = (float)orc_silu(temb[n]);
    if (block >= 0) orc_linear(s, 1, W, m->mod_w[block], m->mod_b[block], 6 * W, mod);
    else orc_linear(s, 1, W, m->fmod_w, m->fmod_b, 2 * W, mod);
    free(s);
}

/* Cross-attention keys / values of one sample's condition tokens for every
 * block (step-invariant: the condition does not change over the sampler). */
/* kv layout: [L][2][Nc][W] (keys then values).                            */
void orc_cond_kv(const void *vm, const uint16_t *cond, float *kv)
{
    const orc_model *m = (const orc_model *)vm;
    size_t nc = (size_t)m->Nc, W = (size_t)m->W;
    float *c = (float *)malloc(sizeof(float) * nc * (size_t)m->Dc);
    for (size_t q = 0; q < nc * (size_t)m->Dc; ++q) c[q] = bf2f(cond[q]);
    float *tmp = (float *)malloc(sizeof(float) * nc * 2 * W);
    for (int l = 0; l < m->L; ++l) {
        orc_linear(c, (int)nc, m->Dc, m->ckv_w[l], m->ckv_b[l], (int)(2 * W), tmp);
        float *kl = kv + (size_t)l * 2 * nc * W;
        float *vl = kl + nc * W;
        for (size_t r = 0; r < nc; ++r) {
            memcpy(kl + r * W, tmp + r * 2 * W, sizeof(float) * W);
            memcpy(vl + r * W, tmp + r * 2 * W + W, sizeof(float) * W);
        }
    }
    free(c);
    free(tmp);
}

/* FlowTransformer(S[I_active], t, c) (Alg. 1 step 2): embeds the a active
 * tokens of one sample, runs every block with self-attention among the
 * active tokens only (Sec. 4.2) and cross-attention to the condition, and
 * returns v_active [a, C] in the order of active_idx.
 * Block (Supp. Sec. F): h = LN(x)(1+scale1)+shift1; x += gate1 * SA(h);
 * x += CA(LN2(x) with affine, cond); h = LN(x)(1+scale2)+shift2;
 * x += gate2 * MLP(h); final: LN(x)(1+s)+sh -> Linear W -> C.             */
void orc_dit_forward(const void *vm, const float *S, const int32_t *active_idx, int a, float t,
                     const float *cond_kv, float *v_out)
{
    const orc_model *m = (const orc_model *)vm;
    const int W = m->W, C = m->C, H = m->H, dh = m->W / m->H, Wm = m->mlp * m->W, Nc = m->Nc;
    size_t aw = (size_t)a * W;
    float *x = (float *)malloc(sizeof(float) * (aw > 0 ? aw : 1));
    float *h = (float *)malloc(sizeof(float) * (aw > 0 ? aw : 1));
    float *y = (float *)malloc(sizeof(float) * (aw > 0 ? aw : 1));
    float *o = (float *)malloc(sizeof(float) * (aw > 0 ? aw : 1));
    float *qkv = (float *)malloc(sizeof(float) * (aw > 0 ? 3 * aw : 1));
    float *u = (float *)malloc(sizeof(float) * (a > 0 ? (size_t)a * Wm : 1));
    float *temb = (float *)malloc(sizeof(float) * (size_t)W);
    float *mod = (float *)malloc(sizeof(float) * (size_t)6 * W);
    float *pe = (float *)malloc(sizeof(float) * (size_t)W);

    /* input embedding of the gathered tokens: Linear C -> W plus pos-emb */
    for (int r = 0; r < a; ++r) {
        int i = active_idx[r];
        orc_pos_embed(m->grid, W, i, pe);
        for (int n = 0; n < W; ++n) {
            double acc = m->in_b[n];
            for (int c = 0; c < C; ++c) acc += (double)S[(size_t)i * C + c] * (double)m->in_w[(size_t)n * C + c];
            x[(size_t)r * W + n] = (float)(acc + (double)pe[n]);
        }
    }
    orc_time_embed(m, t, temb);

    for (int l = 0; l < m->L; ++l) {
        orc_modulation(m, temb, l, mod);
        const float *shift1 = mod, *scale1 = mod + W, *gate1 = mod + 2 * W;
        const float *shift2 = mod + 3 * W, *scale2 = mod + 4 * W, *gate2 = mod + 5 * W;

        /* self-attention among the active tokens */
        orc_layernorm(x, a, W, h);
        for (size_t q = 0; q < aw; ++q) {
            int n = (int)(q % W);
            h[q] = (float)((double)h[q] * (1.0 + (double)scale1[n]) + (double)shift1[n]);
        }
        orc_linear(h, a, W, m->qkv_w[l], m->qkv_b[l], 3 * W, qkv);
        orc_head_rmsnorm(qkv, a, H, dh, 3 * W, m->qn_g[l]);
        orc_head_rmsnorm(qkv + W, a, H, dh, 3 * W, m->kn_g[l]);
        orc_attention(qkv, 3 * W, qkv + W, 3 * W, qkv + 2 * W, 3 * W, a, a, H, dh, o);
        orc_linear(o, a, W, m->o_w[l], m->o_b[l], W, y);
        for (size_t q = 0; q < aw; ++q) x[q] = (float)((double)x[q] + (double)gate1[q % W] * (double)y[q]);

        /* cross-attention to the condition tokens */
        orc_layernorm(x, a, W, h);
        for (size_t q = 0; q < aw; ++q) {
            int n = (int)(q % W);
            h[q] = (float)((double)h[q] * (double)m->ln2_g[l][n] + (double)m->ln2_b[l][n]);
        }
        orc_linear(h, a, W, m->cq_w[l], m->cq_b[l], W, y);
        const float *kc = cond_kv + (size_t)l * 2 * Nc * W;
        const float *vc = kc + (size_t)Nc * W;
        orc_attention(y, W, kc, W, vc, W, a, Nc, H, dh, o);
        orc_linear(o, a, W, m->co_w[l], m->co_b[l], W, y);
        for (size_t q = 0; q < aw; ++q) x[q] = (float)((double)x[q] + (double)y[q]);

        /* MLP */
        orc_layernorm(x, a, W, h);
        for (size_t q = 0; q < aw; ++q) {
            int n = (int)(q % W);
            h[q] = (float)((double)h[q] * (1.0 + (double)scale2[n]) + (double)shift2[n]);
        }
        orc_linear(h, a, W, m->fc1_w[l], m->fc1_b[l], Wm, u);
        for (size_t q = 0; q < (size_t)a * Wm; ++q) u[q] = (float)orc_gelu_tanh(u[q]);
        orc_linear(u, a, Wm, m->fc2_w[l], m->fc2_b[l], W, y);
        for (size_t q = 0; q < aw; ++q) x[q] = (float)((double)x[q] + (double)gate2[q % W] * (double)y[q]);
    }

    /* final layer */
    orc_modulation(m, temb, -1, mod);
    orc_layernorm(x, a, W, h);
    for (size_t q = 0; q < aw; ++q) {
        int n = (int)(q % W);
        h[q] = (float)((double)h[q] * (1.0 + (double)mod[W + n]) + (double)mod[n]);
    }
    orc_linear(h, a, W, m->out_w, m->out_b, C, v_out);

    free(x); free(h); free(y); free(o); free(qkv); free(u); free(temb); free(mod); free(pe);
}

/* ------------------------------------------------------------------------ */
/* Convolutional stand-in decoder (reading: TRELLIS's decoder and weights   */
/* are not in the paper; Eq. 1 only needs a grid decoder O(S)).  The shape  */
/* of an upsampling 3-D convolution stack: 3x3x3 convolutions with zero     */
/* padding, ReLU, nearest-neighbour 2x upsampling in between:               */
/*   C -> 16 at D^3, x2, 16 -> 8 at (2D)^3, x2, 8 -> 1 at (4D)^3,           */
/* and sub-voxel v is occupied iff its logit > 0 ((4D)^3 = 64 N sub-voxels,  */
/* gamma_up = 64).  Each output: acc = bias, then for tap k = 0..26         */
/* ((dz, dy, dx) in {-1, 0, 1}^3, dx fastest) and input channel ci in order, */
/* acc = acc + x w with one rounding per * and +; taps outside the grid are  */
/* skipped.  Grid index (z D + y) D + x, as the tokens.                     */
/* ------------------------------------------------------------------------ */
static void orc_conv3d(const float *in, int cin, int din, int up, const uint16_t *w, const uint16_t *b, int cout,
                       int relu, float *out)
{
    const int d = din * up;
    const size_t vin = (size_t)din * din * din, vout = (size_t)d * d * d;
    for (int co = 0; co < cout; ++co)
        for (int z = 0; z < d; ++z)
            for (int y = 0; y < d; ++y)
                for (int x = 0; x < d; ++x) {
                    float acc = bf2f(b[co]);
                    for (int k = 0; k < 27; ++k) {
                        const int zz = z + k / 9 - 1, yy = y + (k / 3) % 3 - 1, xx = x + k % 3 - 1;
                        if (zz < 0 || zz >= d || yy < 0 || yy >= d || xx < 0 || xx >= d) continue;
                        const size_t src = ((size_t)(zz / up) * din + (size_t)(yy / up)) * din + (size_t)(xx / up);
                        for (int ci = 0; ci < cin; ++ci) {
                            const float p = in[(size_t)ci * vin + src] * bf2f(w[((size_t)co * cin + ci) * 27 + k]);
                            acc = acc + p;
                        }
                    }
                    out[(size_t)co * vout + ((size_t)z * d + y) * d + x] = relu ? (acc > 0.0f ? acc : 0.0f) : acc;
                }
}

void orc_decode_conv(const void *vm, const float *S, uint8_t *occ)
{
    const orc_model *m = (const orc_model *)vm;
    const int D = m->grid, C = m->C;
    const size_t N = (size_t)D * D * D;
    float *x0 = (float *)malloc(sizeof(float) * N * C);
    float *x1 = (float *)malloc(sizeof(float) * N * 16);
    float *x2 = (float *)malloc(sizeof(float) * N * 8 * 8);
    float *lg = (float *)malloc(sizeof(float) * N * 64);
    for (size_t v = 0; v < N; ++v)
        for (int c = 0; c < C; ++c) x0[(size_t)c * N + v] = S[v * C + c];
    orc_conv3d(x0, C, D, 1, m->dc1_w, m->dc1_b, 16, 1, x1);
    orc_conv3d(x1, 16, D, 2, m->dc2_w, m->dc2_b, 8, 1, x2);
    orc_conv3d(x2, 8, 2 * D, 2, m->dc3_w, m->dc3_b, 1, 0, lg);
    for (size_t q = 0; q < N * 64; ++q) occ[q] = (uint8_t)(lg[q] > 0.0f);
    free(x0); free(x1); free(x2); free(lg);
}

/* ------------------------------------------------------------------------ */
/* Data-driven PCSC slope (Supp. "Data-driven Parameter Selection"): per     */
/* instance, a RANSAC line fit of ln(dS_k) against the step index k over the */
/* intermediate steps k_lo..k_hi (8..18 in the paper), instances whose fit  */
/* is poor filtered out, and mu = the median of the remaining slopes.       */
/* Readings: the hypotheses are every pair of points (exhaustive, so the    */
/* fit is deterministic); the best pair has the most inliers (|residual| <= */
/* tol in ln units), ties to the smaller inlier sum of squared residuals,   */
/* then to the earlier pair; the slope is then the least-squares slope over */
/* its inliers; steps with dS_k = 0 carry no point; an instance is kept iff */
/* it has >= 3 points and its inliers are >= min_frac of them; the median of */
/* an even count is the mean of the middle two.                            */
/* curves: [n][T] dynamic voxels per 1-based step k at index k - 1.         */
/* slopes_out / kept_out: nullable [n].  Returns the number kept; mu_out is */
/* NaN when none is.                                                        */
/* ------------------------------------------------------------------------ */
static int orc_cmp_double(const void *a, const void *b)
{
    const double x = *(const double *)a, y = *(const double *)b;
    return (x > y) - (x < y);
}

int orc_fit_mu(const double *curves, int n, int T, int k_lo, int k_hi, double tol, double min_frac,
               double *mu_out, double *slopes_out, int *kept_out)
{
    double *kept_slopes = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    double xs[64], ys[64];
    int nk = 0;
    for (int i = 0; i < n; ++i) {
        int m = 0;
        for (int k = k_lo; k <= k_hi && k <= T && m < 64; ++k) {
            const double d = curves[(size_t)i * T + (k - 1)];
            if (d > 0.0) {
                xs[m] = (double)k;
                ys[m] = log(d);
                ++m;
            }
        }
        double slope = NAN;
        int keep = 0;
        if (m >= 3) {
            int best_cnt = -1;
            double best_sse = INFINITY;
            double best_a = 0.0, best_b = 0.0;
            for (int p = 0; p < m; ++p)
                for (int q = p + 1; q < m; ++q) {
                    const double b = (ys[q] - ys[p]) / (xs[q] - xs[p]);
                    const double a = ys[p] - b * xs[p];
                    int cnt = 0;
                    double sse = 0.0;
                    for (int j = 0; j < m; ++j) {
                        const double r = ys[j] - (a + b * xs[j]);
                        if (fabs(r) <= tol) {
                            ++cnt;
                            sse += r * r;
                        }
                    }
                    if (cnt > best_cnt || (cnt == best_cnt && sse < best_sse)) {
                        best_cnt = cnt;
                        best_sse = sse;
                        best_a = a;
                        best_b = b;
                    }
                }
            /* least squares over the best hypothesis' inliers */
            double sx = 0.0, sy = 0.0, sxx = 0.0, sxy = 0.0;
            int c = 0;
            for (int j = 0; j < m; ++j) {
                const double r = ys[j] - (best_a + best_b * xs[j]);
                if (fabs(r) <= tol) {
                    sx += xs[j];
                    sy += ys[j];
                    sxx += xs[j] * xs[j];
                    sxy += xs[j] * ys[j];
                    ++c;
                }
            }
            const double den = c * sxx - sx * sx;
            slope = den != 0.0 ? (c * sxy - sx * sy) / den : best_b;
            keep = (double)best_cnt >= min_frac * (double)m;
        }
        if (slopes_out) slopes_out[i] = slope;
        if (kept_out) kept_out[i] = keep;
        if (keep) kept_slopes[nk++] = slope;
    }
    double mu = NAN;
    if (nk > 0) {
        qsort(kept_slopes, (size_t)nk, sizeof(double), orc_cmp_double);
        mu = (nk % 2) ? kept_slopes[nk / 2] : 0.5 * (kept_slopes[nk / 2 - 1] + kept_slopes[nk / 2]);
    }
    if (mu_out) *mu_out = mu;
    free(kept_slopes);
    return nk;
}

/* ======================================================================== */
/* Algorithm 1 end to end for B independent samples.                         */
/* ======================================================================== */
/*
 * S: [B, N, C] fp32, noise in, S_0 out.  cond: [B, Nc, Dc] bf16.
 * tau, refresh_mode, hyperparameters as in orc_phase_quota / orc_tau_gate.
 * sigma_override: nullable [B]; when given, it replaces the measured sigma
 *   in the PCSC forecast (the measured value is still reported).
 * quota_schedule: nullable [T, B] phase quotas that replace the three-phase
 *   rule (the tau rule still applies on top).
 * Outputs (nullable): quota_log [T, B] effective cache quota, nact_log
 *   [T, B] active tokens, sigma_out [B] measured dynamic voxels at the
 *   anchor step (Eq. 1 between the grids before and after step k_a).
 * v_hist_out: nullable [2, B, N, C] bf16 -- (v_cache, v_prev_cache) at exit.
 * cfg_on: guide the steps k with t_k >= cfg_t_lo with strength cfg_s; the
 *   unconditional prediction sees the all-zero condition (reading: the paper
 *   names no null condition) and the same active tokens.
 * ssc_accel: 1 scores with the second difference over the last three
 *   velocities (orc_ssc_score3), 0 with the first difference of Sec. 4.1.
 * decoder: 1 decodes the grids of Eq. 1 with the convolutional stand-in
 *   (orc_decode_conv, needs G = 64), 0 with the linear one (orc_occupancy).
 * dyn_log: nullable [T, B]; Eq. 1's dS between the grids before and after
 *   every step (the curve the PCSC slope is fitted to).
 */
int orc_sample(const void *vm, int T, double eta, double rho_a, double rho_off, double mu,
               double omega, double xi, int f_corr, int tau, int refresh_mode,
               float *S, const uint16_t *cond, int B, const double *sigma_override,
               const int32_t *quota_schedule, int32_t *quota_log, int32_t *nact_log,
               double *sigma_out, uint16_t *v_hist_out, int cfg_on, double cfg_s, double cfg_t_lo,
               int ssc_accel, int decoder, int64_t *dyn_log)
{
    const orc_model *m = (const orc_model *)vm;
    const int N = m->grid * m->grid * m->grid, C = m->C, G = m->G;
    const size_t NC = (size_t)N * C;
    float *t = (float *)malloc(sizeof(float) * (size_t)(T + 1));
    orc_time_schedule(T, eta, t);
    const int ka = orc_ceil_steps(T, rho_a);

    float *kv = (float *)malloc(sizeof(float) * (size_t)m->L * 2 * m->Nc * m->W);
    uint16_t *vc = (uint16_t *)calloc(NC, sizeof(uint16_t)); /* v_cache <- 0 */
    uint16_t *vp = (uint16_t *)calloc(NC, sizeof(uint16_t)); /* v_prev_cache <- 0 */
    uint16_t *vt = (uint16_t *)malloc(sizeof(uint16_t) * NC);
    uint16_t *vpp = (uint16_t *)calloc(NC, sizeof(uint16_t)); /* v(t-3) <- 0 */
    float *score = (float *)malloc(sizeof(float) * (size_t)N);
    uint8_t *cached = (uint8_t *)malloc((size_t)N);
    int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * (size_t)N);
    float *va = (float *)malloc(sizeof(float) * NC);
    float *Sold = (float *)malloc(sizeof(float) * NC);
    uint8_t *occ_a = (uint8_t *)malloc((size_t)N * G);
    uint8_t *occ_b = (uint8_t *)malloc((size_t)N * G);
    float *kv_null = NULL, *va_c = NULL, *va_u = NULL;
    if (cfg_on) {
        uint16_t *zero = (uint16_t *)calloc((size_t)m->Nc * m->Dc, sizeof(uint16_t));
        kv_null = (float *)malloc(sizeof(float) * (size_t)m->L * 2 * m->Nc * m->W);
        orc_cond_kv(m, zero, kv_null);
        free(zero);
        va_c = (float *)malloc(sizeof(float) * NC);
        va_u = (float *)malloc(sizeof(float) * NC);
    }

    for (int b = 0; b < B; ++b) {
        float *Sb = S + (size_t)b * NC;
        orc_cond_kv(m, cond + (size_t)b * m->Nc * m->Dc, kv);
        memset(vc, 0, sizeof(uint16_t) * NC);
        memset(vp, 0, sizeof(uint16_t) * NC);
        memset(vpp, 0, sizeof(uint16_t) * NC);
        int consec = 0;
        double sigma = sigma_override ? sigma_override[b] : 0.0;
        for (int k = 1; k <= T; ++k) {
            int c;
            if (quota_schedule) {
                c = quota_schedule[(size_t)(k - 1) * B + b];
            } else {
                c = orc_phase_quota(N, T, rho_a, rho_off, mu, xi, f_corr, G, sigma, k, NULL);
            }
            c = orc_tau_gate(c, tau, refresh_mode, &consec);
            int a;
            if (c > 0) {
                orc_ssc_score3(vc, vp, ssc_accel ? vpp : NULL, N, C, omega, score);
                a = orc_select(score, N, c, cached, idx);
            } else {
                for (int i = 0; i < N; ++i) idx[i] = i;
                a = N;
            }
            if (quota_log) quota_log[(size_t)(k - 1) * B + b] = c;
            if (nact_log) nact_log[(size_t)(k - 1) * B + b] = a;
            if (a > 0) {
                if (cfg_on && (double)t[k - 1] >= cfg_t_lo) {
                    orc_dit_forward(m, Sb, idx, a, t[k - 1], kv, va_c);
                    orc_dit_forward(m, Sb, idx, a, t[k - 1], kv_null, va_u);
                    orc_cfg_combine((long long)a * C, va_c, va_u, cfg_s, va);
                } else {
                    orc_dit_forward(m, Sb, idx, a, t[k - 1], kv, va);
                }
            }
            if (k == ka || dyn_log) memcpy(Sold, Sb, sizeof(float) * NC);
            float dt = t[k - 1] - t[k];
            orc_merge_euler(N, C, idx, a, va, vc, dt, Sb, vt);
            if (k == ka || dyn_log) {
                if (decoder) {
                    orc_decode_conv(m, Sold, occ_a);
                    orc_decode_conv(m, Sb, occ_b);
                } else {
                    orc_occupancy(Sold, N, C, m->dec_w, G, occ_a);
                    orc_occupancy(Sb, N, C, m->dec_w, G, occ_b);
                }
                double meas = (double)orc_dynamic_voxels(occ_a, occ_b, (long long)N * G);
                if (dyn_log) dyn_log[(size_t)(k - 1) * B + b] = (int64_t)meas;
                if (k == ka) {
                    if (sigma_out) sigma_out[b] = meas;
                    if (!sigma_override) sigma = meas;
                }
            }
            /* v(t-3) <- v_prev_cache <- v_cache <- v_t */
            uint16_t *tmp = vpp;
            vpp = vp;
            vp = vc;
            vc = vt;
            vt = tmp;
        }
        if (v_hist_out) {
            memcpy(v_hist_out + (size_t)b * NC, vc, sizeof(uint16_t) * NC);
            memcpy(v_hist_out + (size_t)B * NC + (size_t)b * NC, vp, sizeof(uint16_t) * NC);
        }
    }
    free(t); free(kv); free(vc); free(vp); free(vt); free(vpp); free(score); free(cached); free(idx);
    free(va); free(Sold); free(occ_a); free(occ_b); free(kv_null); free(va_c); free(va_u);
    return 0;
}
