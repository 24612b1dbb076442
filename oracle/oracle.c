/*
 * CPU oracle for EmTrackMichelId hit identification.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library path may call this; only
 * the test suite, the smoke check and the benchmark's CPU-baseline leg do.  It
 * shares no code, header or table with the CUDA library.
 *
 * What it computes (arXiv:2009.04509):
 *   Sec. 2.1  For every reconstructed hit a 48x48 "patch" is cut from the
 *             hit's wire plane, centred on the hit's wire and peak time; rows
 *             are wires, columns are time intervals, a pixel is the charge in
 *             that (wire, interval).
 *   Sec. 2.2  The patch goes through a 5x5 convolution with 48 filters,
 *             stride 1, giving 48 maps of 44x44, ReLU; a dense layer of 128
 *             with ReLU; a dense layer of 32 with ReLU; then two heads: 3
 *             outputs under a softmax and 1 output under a sigmoid.  Dropout
 *             is identity at inference.  11,900,420 parameters in total.
 *
 * Readings where the paper is silent (each one is a choice; the paper fixes
 * none of them, and another reading would give other patches):
 *   - a time interval is 6 consecutive ticks on a grid fixed to the plane
 *     ([6b, 6b+6)); its value is the fp32 sum a0+a1+...+a5 taken left to
 *     right, then one IEEE fp32 division by 6.  A trailing partial interval
 *     (nticks % 6 != 0) does not exist and reads as zero;
 *   - the hit sits at row 24 / column 24 of the patch (window offsets -24..23
 *     on both axes); its interval is floor(tick / 6) with floor division;
 *   - pixels outside the plane are zero;
 *   - the convolution is a cross-correlation (no kernel flip), "valid";
 *   - the conv maps are flattened channels-last: index (y*44 + x)*48 + c;
 *   - softmax outputs are ordered (track, em, none), then the Michel sigmoid.
 *
 *   Sec. 2.1  Upstream of the patch cut, hits are found on each wire's
 *             deconvolved waveform (or_find_hits).  The paper does not give
 *             the algorithm; the reading taken: a hit is a maximal run of
 *             consecutive ticks whose value exceeds a threshold, placed at
 *             the run's largest value.
 *
 * Precision: the patch cut is fp32 by definition (it must be reproduced bit
 * for bit); everything in the network is accumulated in double.  Optional
 * emulating modes round the operands of the two large contractions (patch,
 * conv weights, conv outputs after ReLU, dense-1 weights) to bf16 or to fp16
 * before use, the points where a 16-bit tensor-core path rounds; they are a
 * diagnostic reference, not the definition.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define OR_OK 0
#define OR_ERR_ARG 1
#define OR_ERR_OOM 2

/* ------------------------------------------------------------------ helpers */

static long floor_div(long a, long b)
{
    long q = a / b;
    if ((a % b != 0) && ((a < 0) != (b < 0)))
        q -= 1;
    return q;
}

/* Round a finite float to the nearest bf16 (ties to even); returned as the
 * float whose low 16 bits are zero. */
static float round_bf16_f(float x)
{
    uint32_t u;
    memcpy(&u, &x, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);
    u &= 0xFFFF0000u;
    memcpy(&x, &u, 4);
    return x;
}

/* Round a finite float to the nearest IEEE binary16 value (ties to even,
 * gradual underflow, overflow to infinity); returned as a float. */
static float round_fp16_f(float x)
{
    if (x == 0.0f || !isfinite(x))
        return x;
    const float a = fabsf(x);
    int e;
    frexpf(a, &e);              /* a in [2^(e-1), 2^e) */
    int qexp = e - 11;          /* 11 significant bits */
    if (qexp < -24)
        qexp = -24;             /* subnormal spacing 2^-24 */
    const float q = ldexpf(1.0f, qexp);
    float r = rintf(a / q) * q; /* a / q is exact: q is a power of two */
    if (r >= 65520.0f)
        r = INFINITY;
    return copysignf(r, x);
}

/* Round a finite float to the nearest FP8 E4M3 value (sign, 4 exponent bits
 * with bias 7, 3 mantissa bits; no infinities), ties to even, gradual
 * underflow below 2^-6 (spacing 2^-9), saturating at +-448 (the largest
 * finite value); returned as a float. */
static float round_e4m3_f(float x)
{
    if (x == 0.0f || isnan(x))
        return x;
    const float a = fabsf(x);
    int e;
    frexpf(a, &e);              /* a in [2^(e-1), 2^e) */
    int qexp = e - 4;           /* 4 significant bits */
    if (qexp < -9)
        qexp = -9;              /* subnormal spacing 2^-9 */
    const float q = ldexpf(1.0f, qexp);
    float r = rintf(a / q) * q; /* a / q is exact: q is a power of two */
    if (r > 448.0f)
        r = 448.0f;
    return copysignf(r, x);
}

void or_round_e4m3(const float *in, float *out, long n)
{
    for (long i = 0; i < n; ++i)
        out[i] = round_e4m3_f(in[i]);
}

/* Power-of-two scales of the fp8 emulation: dense-1 activations are rounded
 * as e4m3(a * act_scale) / act_scale, its weights as e4m3(w * w_scale) /
 * w_scale. */
static double fp8_act_scale = 1.0, fp8_w_scale = 1.0;

void or_set_fp8_scales(double act_scale, double w_scale)
{
    fp8_act_scale = act_scale;
    fp8_w_scale = w_scale;
}

void or_round_fp16(const float *in, float *out, long n)
{
    for (long i = 0; i < n; ++i)
        out[i] = round_fp16_f(in[i]);
}

/* emulation modes: 0 none, 1 bf16, 2 fp16, 3 fp8 (bf16 conv operands, e4m3
 * dense-1 operands); round_mode covers the 16-bit roundings */
static float round_mode(float x, int mode)
{
    return (mode == 1 || mode == 3) ? round_bf16_f(x) : mode == 2 ? round_fp16_f(x) : x;
}

static float round_scaled_e4m3(float x, double scale)
{
    return (float)((double)round_e4m3_f((float)((double)x * scale)) / scale);
}

void or_round_bf16(const float *in, uint16_t *out, long n)
{
    for (long i = 0; i < n; ++i) {
        float r = round_bf16_f(in[i]);
        uint32_t u;
        memcpy(&u, &r, 4);
        out[i] = (uint16_t)(u >> 16);
    }
}

void or_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int or_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------- Sec. 2.1: patches */

/* Value of time interval b of one wire: the mean of ticks [ds*b, ds*b + ds),
 * summed in fp32 left to right, then divided once. */
static float interval_value(const float *wire_row, long b, int ds)
{
    const float *a = wire_row + b * ds;
    float s = a[0];
    for (int j = 1; j < ds; ++j)
        s = s + a[j];
    return s / (float)ds;
}

/* patches[h][r][c] = interval value of wire (w_h - psize/2 + r), interval
 * (floor(t_h/ds) - psize/2 + c); zero where the wire or the interval does not
 * exist.  hits[h] = {wire, peak tick}. */
int or_extract_patches(const float *plane, int nwires, int nticks, long ld,
                       const int32_t *hits, long nhits, int psize, int ds,
                       float *patches)
{
    if (nhits < 0 || psize <= 0 || ds <= 0 || nwires < 0 || nticks < 0 || ld < nticks)
        return OR_ERR_ARG;
    if (nhits == 0)
        return OR_OK;
    if (!plane || !hits || !patches)
        return OR_ERR_ARG;
    const long nint = nticks / ds;
    const int half = psize / 2;
    for (long h = 0; h < nhits; ++h) {
        const long wc = hits[2 * h];
        const long bc = floor_div(hits[2 * h + 1], ds);
        float *out = patches + h * (long)psize * psize;
        for (int r = 0; r < psize; ++r) {
            const long w = wc - half + r;
            for (int c = 0; c < psize; ++c) {
                const long b = bc - half + c;
                float v = 0.0f;
                if (w >= 0 && w < nwires && b >= 0 && b < nint)
                    v = interval_value(plane + w * ld, b, ds);
                out[r * psize + c] = v;
            }
        }
    }
    return OR_OK;
}

/* ---------------------------------------------------- Sec. 2.2: the network */

typedef struct {
    int P;  /* patch side (48) */
    int R;  /* conv kernel side (5) */
    int F;  /* conv filters (48) */
    int N1; /* dense-1 width (128) */
    int N2; /* dense-2 width (32) */
    int NC; /* softmax classes (3) */
} or_dims;

/* Conv + ReLU on one single-channel image.
 *   img  [P][P]
 *   w    [R][R][F]   (tap row i, tap column j, filter f)
 *   b    [F]
 *   out  [Q][Q][F]   Q = P - R + 1, out[y][x][f] = max(0, b[f] + sum_ij img[y+i][x+j] w[i][j][f]) */
void or_conv_relu(const double *img, int P, const double *w, const double *b, int R, int F,
                  double *out)
{
    const int Q = P - R + 1;
    for (int y = 0; y < Q; ++y)
        for (int x = 0; x < Q; ++x)
            for (int f = 0; f < F; ++f) {
                double s = b[f];
                for (int i = 0; i < R; ++i)
                    for (int j = 0; j < R; ++j)
                        s += img[(y + i) * P + (x + j)] * w[(i * R + j) * F + f];
                out[((long)y * Q + x) * F + f] = s > 0.0 ? s : 0.0;
            }
}

/* Dense layer: y[n] = b[n] + sum_k x[k] W[k][n], optional ReLU.  W is [K][N]. */
void or_dense(const double *x, long K, const float *W, const float *b, int N, int relu,
              double *y)
{
    for (int n = 0; n < N; ++n)
        y[n] = b ? (double)b[n] : 0.0;
    for (long k = 0; k < K; ++k) {
        const double xk = x[k];
        if (xk == 0.0)
            continue; /* adds exactly zero */
        const float *row = W + k * (long)N;
        for (int n = 0; n < N; ++n)
            y[n] += xk * (double)row[n];
    }
    if (relu)
        for (int n = 0; n < N; ++n)
            y[n] = y[n] > 0.0 ? y[n] : 0.0;
}

/* Heads: z = softmax(logits[0..NC)), m = sigmoid(logit_m). */
void or_heads(const double *logits, int NC, double logit_m, double *scores)
{
    double mx = logits[0];
    for (int c = 1; c < NC; ++c)
        if (logits[c] > mx)
            mx = logits[c];
    double s = 0.0;
    for (int c = 0; c < NC; ++c) {
        scores[c] = exp(logits[c] - mx);
        s += scores[c];
    }
    for (int c = 0; c < NC; ++c)
        scores[c] /= s;
    scores[NC] = 1.0 / (1.0 + exp(-logit_m));
}

/* Full network on n patches [n][P][P] (fp32).  Weights in the layouts of the
 * header comment, fp32.  Outputs (each [n][NC+1], double): the logits (NC
 * class logits then the Michel logit) and the scores (softmax then sigmoid).
 * emulate = 1 (bf16) or 2 (fp16) rounds patch, conv weights, post-ReLU conv
 * outputs and dense-1 weights to that format before use; 3 (fp8) rounds
 * patch and conv weights to bf16 and the post-ReLU conv outputs and dense-1
 * weights to e4m3 with the scales of or_set_fp8_scales; 0 rounds nothing. */
int or_forward(const or_dims *d, const float *patches, long n,
               const float *conv_w, const float *conv_b,
               const float *fc1_w, const float *fc1_b,
               const float *fc2_w, const float *fc2_b,
               const float *cls_w, const float *cls_b,
               const float *mic_w, const float *mic_b,
               int emulate, double *logits, double *scores)
{
    if (!d || n < 0)
        return OR_ERR_ARG;
    const int P = d->P, R = d->R, F = d->F, N1 = d->N1, N2 = d->N2, NC = d->NC;
    if (P <= 0 || R <= 0 || R > P || F <= 0 || N1 <= 0 || N2 <= 0 || NC <= 0 ||
        emulate < 0 || emulate > 3)
        return OR_ERR_ARG;
    if (n == 0)
        return OR_OK;
    const int Q = P - R + 1;
    const long K1 = (long)Q * Q * F;

    /* conv weights/bias as double (rounded to bf16 in emulation mode) */
    double *cw = (double *)malloc(sizeof(double) * R * R * F);
    double *cb = (double *)malloc(sizeof(double) * F);
    float *w1 = NULL;
    if (!cw || !cb) {
        free(cw);
        free(cb);
        return OR_ERR_OOM;
    }
    for (int i = 0; i < R * R * F; ++i)
        cw[i] = (double)round_mode(conv_w[i], emulate);
    for (int f = 0; f < F; ++f)
        cb[f] = conv_b[f];
    const float *W1 = fc1_w;
    if (emulate) {
        w1 = (float *)malloc(sizeof(float) * K1 * N1);
        if (!w1) {
            free(cw);
            free(cb);
            return OR_ERR_OOM;
        }
        for (long i = 0; i < K1 * N1; ++i)
            w1[i] = emulate == 3 ? round_scaled_e4m3(fc1_w[i], fp8_w_scale) : round_mode(fc1_w[i], emulate);
        W1 = w1;
    }

    int fail = 0;
#pragma omp parallel
    {
        double *img = (double *)malloc(sizeof(double) * P * P);
        double *act = (double *)malloc(sizeof(double) * K1);
        double *h1 = (double *)malloc(sizeof(double) * N1);
        double *h2 = (double *)malloc(sizeof(double) * N2);
        double *z = (double *)malloc(sizeof(double) * (NC + 1));
        if (!img || !act || !h1 || !h2 || !z) {
#pragma omp atomic write
            fail = 1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (long h = 0; h < n; ++h) {
                const float *p = patches + h * (long)P * P;
                for (int i = 0; i < P * P; ++i)
                    img[i] = (double)round_mode(p[i], emulate);
                or_conv_relu(img, P, cw, cb, R, F, act);
                if (emulate == 3)
                    for (long k = 0; k < K1; ++k)
                        act[k] = (double)round_scaled_e4m3((float)act[k], fp8_act_scale);
                else if (emulate)
                    for (long k = 0; k < K1; ++k)
                        act[k] = (double)round_mode((float)act[k], emulate);
                or_dense(act, K1, W1, fc1_b, N1, 1, h1);
                or_dense(h1, N1, fc2_w, fc2_b, N2, 1, h2);
                or_dense(h2, N2, cls_w, cls_b, NC, 0, z);
                or_dense(h2, N2, mic_w, mic_b, 1, 0, z + NC);
                double *lo = logits + h * (NC + 1);
                for (int c = 0; c <= NC; ++c)
                    lo[c] = z[c];
                or_heads(z, NC, z[NC], scores + h * (NC + 1));
            }
        }
        free(img);
        free(act);
        free(h1);
        free(h2);
        free(z);
    }
    free(cw);
    free(cb);
    free(w1);
    return fail ? OR_ERR_OOM : OR_OK;
}

/* ------------------------------------------------------------- hit finding */

/* Hit finding on the deconvolved waveforms (Sec. 2.1).  The paper says only
 * that hits are found on each wire's deconvolved waveform and carry a time
 * and a charge; the plainest reading is taken.  On each wire w of the plane, a hit is a maximal run of
 * consecutive ticks t (0 <= t < nticks) with plane[w][t] > threshold
 * (strictly; a NaN is never above).  For each run:
 *   start, end  its first and last tick;
 *   tick        the tick of its largest value, the earliest one on ties;
 *   peak        that value;
 *   charge      the sum of its values, accumulated in double.
 * Hits are listed wire by wire, and within a wire by start tick.  At most
 * `capacity` hits are written; the return value is the number found (which
 * may exceed `capacity`), or -1 for an invalid argument. */
static int above_threshold(float v, float threshold)
{
    return v > threshold;
}

long or_find_hits(const float *plane, int nwires, int nticks, long ld, float threshold, long capacity,
                  int32_t *wire, int32_t *tick, int32_t *start, int32_t *end, float *peak, double *charge)
{
    if (nwires < 0 || nticks < 0 || ld < nticks || capacity < 0 || (nwires > 0 && nticks > 0 && !plane))
        return -1;
    long n = 0;
    for (int w = 0; w < nwires; ++w) {
        const float *row = plane + (long)w * ld;
        int t = 0;
        while (t < nticks) {
            if (!above_threshold(row[t], threshold)) {
                ++t;
                continue;
            }
            const int first = t;
            int best = t;
            double q = 0.0;
            while (t < nticks && above_threshold(row[t], threshold)) {
                if (row[t] > row[best])
                    best = t;
                q += (double)row[t];
                ++t;
            }
            if (n < capacity) {
                wire[n] = w;
                tick[n] = best;
                start[n] = first;
                end[n] = t - 1;
                peak[n] = row[best];
                charge[n] = q;
            }
            ++n;
        }
    }
    return n;
}
