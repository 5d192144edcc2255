/*
 * dbl_oracle.c -- plain, slow, fp64 CPU reference for the ResNet-18 training
 * step of the hybrid dual-batch / cyclic-progressive scheme
 * (arXiv 2509.26092).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load this code.  It shares nothing
 * with the CUDA library: no headers, no helpers, no tables.
 *
 * Every routine is the textbook definition written out as loops, in double
 * precision, with no blocking, fusion or reordering beyond what the
 * definition states.  OpenMP only splits independent output elements (or
 * independent images for the scatter-form adjoint) across threads; each
 * output is still summed in one fixed order.
 *
 * Layouts: activations NHWC, conv weights KRSC, all row-major.
 *
 * Paper passages followed:
 *   - mini-batch SGD with the batch-mean gradient: Sec. 2.2, Eq. 1;
 *   - model-update factor (1 for large-batch workers, d_S/d_L or
 *     sqrt(d_S/d_L) for small-batch workers): Sec. 3.4;
 *   - asynchronous pushes applied by the server as they arrive: Sec. 2.4
 *     (ASP) and Sec. 3.1;
 *   - resolution changes of cyclic progressive learning: Sec. 4.1;
 *   - ResNet-18 (convolutions, BatchNorm, ReLU, residual, global pooling and
 *     one fully connected layer): Sec. 5.1.1 and Sec. 6.
 * Readings where the paper is silent (momentum form, push order, resize
 * convention, max-pool tie rule, BN epsilon) are the ones listed in the
 * design notes; each is restated at the routine that takes it.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define IDX4(a, b, c, d, B, C, D) ((((int64_t)(a) * (B) + (b)) * (C) + (c)) * (D) + (d))

static int out_dim(int in, int k, int stride, int pad) { return (in + 2 * pad - k) / stride + 1; }

/* ------------------------------------------------------------------------ */
/* bf16 storage rounding.                                                    */
/* bfloat16 keeps fp32's 8-bit exponent and 8 significand bits (7 stored).  */
/* Round-to-nearest-even of a double to that grid, written from the format's */
/* definition: normal numbers have a quantum of 2^(e-8) for |x| in          */
/* [2^(e-1), 2^e); below 2^-126 the quantum is fixed at 2^-133.             */
/* ------------------------------------------------------------------------ */
double orc_round_bf16(double x)
{
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    frexp(x, &e); /* |x| in [2^(e-1), 2^e) */
    int qexp = e - 8;
    if (e - 1 < -126) qexp = -133;
    double scaled = ldexp(x, -qexp);
    double r = nearbyint(scaled); /* default rounding mode: ties to even */
    double y = ldexp(r, qexp);
    /* overflow beyond the largest finite bf16 (0x7F7F) rounds to infinity */
    const double bmax = ldexp(255.0, 120); /* (2 - 2^-7) * 2^127 */
    if (fabs(y) > bmax) y = copysign(INFINITY, x);
    return y;
}

/* ------------------------------------------------------------------------ */
/* fp16 (IEEE 754 binary16) storage rounding, for the mixed-precision runs   */
/* of the paper's ImageNet experiments (Sec. 5.2.3).  binary16 has a 5-bit   */
/* exponent and 11 significand bits (10 stored): for |x| in [2^(e-1), 2^e)   */
/* with e - 1 >= -14 the quantum is 2^(e-11); below 2^-14 (subnormals) it is */
/* fixed at 2^-24.  Round to nearest, ties to even; the largest finite value */
/* is 65504 = (2 - 2^-10) * 2^15, and anything that rounds above it is       */
/* infinite.                                                                 */
/* ------------------------------------------------------------------------ */
double orc_round_f16(double x)
{
    if (x == 0.0 || !isfinite(x)) return x;
    int e;
    frexp(x, &e); /* |x| in [2^(e-1), 2^e) */
    int qexp = e - 11;
    if (e - 1 < -14) qexp = -24;
    double r = nearbyint(ldexp(x, -qexp)); /* ties to even */
    double y = ldexp(r, qexp);
    if (fabs(y) > 65504.0) y = copysign(INFINITY, x);
    return y;
}

void orc_round_f16_array(double* a, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) a[i] = orc_round_f16(a[i]);
}

void orc_round_bf16_array(double* a, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) a[i] = orc_round_bf16(a[i]);
}

/* ------------------------------------------------------------------------ */
/* Convolution (cross-correlation, zero padding), Sec. 5.1.1 ResNet-18.      */
/*   y[n,p,q,k] = sum_{r,s,c} x[n, p*st + r - pad, q*st + s - pad, c] w[k,r,s,c] */
/*   P = floor((H + 2 pad - R)/st) + 1.                                      */
/* ------------------------------------------------------------------------ */
void orc_conv2d_fwd(const double* x, const double* w, double* y, int N, int H, int W, int C, int K,
                    int R, int S, int st, int pad)
{
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, S, st, pad);
#pragma omp parallel for collapse(2) schedule(static)
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < P; ++p)
            for (int q = 0; q < Q; ++q)
                for (int k = 0; k < K; ++k) {
                    double acc = 0.0;
                    for (int r = 0; r < R; ++r) {
                        const int h = p * st + r - pad;
                        if (h < 0 || h >= H) continue;
                        for (int s = 0; s < S; ++s) {
                            const int ww = q * st + s - pad;
                            if (ww < 0 || ww >= W) continue;
                            const double* xp = x + IDX4(n, h, ww, 0, H, W, C);
                            const double* wp = w + IDX4(k, r, s, 0, R, S, C);
                            for (int c = 0; c < C; ++c) acc += xp[c] * wp[c];
                        }
                    }
                    y[IDX4(n, p, q, k, P, Q, K)] = acc;
                }
}

/* Data gradient: the adjoint of the forward map, written in scatter form   */
/* (each dy element sends dy*w to every input it read).  Images are         */
/* independent, so the scatter is race-free per image.                      */
void orc_conv2d_dgrad(const double* dy, const double* w, double* dx, int N, int H, int W, int C, int K,
                      int R, int S, int st, int pad)
{
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, S, st, pad);
    memset(dx, 0, sizeof(double) * (size_t)N * H * W * C);
#pragma omp parallel for schedule(static)
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < P; ++p)
            for (int q = 0; q < Q; ++q)
                for (int k = 0; k < K; ++k) {
                    const double g = dy[IDX4(n, p, q, k, P, Q, K)];
                    for (int r = 0; r < R; ++r) {
                        const int h = p * st + r - pad;
                        if (h < 0 || h >= H) continue;
                        for (int s = 0; s < S; ++s) {
                            const int ww = q * st + s - pad;
                            if (ww < 0 || ww >= W) continue;
                            double* xp = dx + IDX4(n, h, ww, 0, H, W, C);
                            const double* wp = w + IDX4(k, r, s, 0, R, S, C);
                            for (int c = 0; c < C; ++c) xp[c] += g * wp[c];
                        }
                    }
                }
}

/* Weight gradient: dw[k,r,s,c] = sum_{n,p,q} dy[n,p,q,k] x[n, p*st+r-pad, q*st+s-pad, c]. */
void orc_conv2d_wgrad(const double* x, const double* dy, double* dw, int N, int H, int W, int C, int K,
                      int R, int S, int st, int pad)
{
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, S, st, pad);
#pragma omp parallel for collapse(2) schedule(static)
    for (int k = 0; k < K; ++k)
        for (int r = 0; r < R; ++r)
            for (int s = 0; s < S; ++s)
                for (int c = 0; c < C; ++c) {
                    double acc = 0.0;
                    for (int n = 0; n < N; ++n)
                        for (int p = 0; p < P; ++p) {
                            const int h = p * st + r - pad;
                            if (h < 0 || h >= H) continue;
                            for (int q = 0; q < Q; ++q) {
                                const int ww = q * st + s - pad;
                                if (ww < 0 || ww >= W) continue;
                                acc += dy[IDX4(n, p, q, k, P, Q, K)] * x[IDX4(n, h, ww, c, H, W, C)];
                            }
                        }
                    dw[IDX4(k, r, s, c, R, S, C)] = acc;
                }
}

/* Single-element evaluators, for sampled checks at full size.               */
double orc_conv2d_fwd_at(const double* x, const double* w, int N, int H, int W, int C, int K, int R, int S,
                         int st, int pad, int n, int p, int q, int k)
{
    (void)N; (void)K;
    double acc = 0.0;
    for (int r = 0; r < R; ++r) {
        const int h = p * st + r - pad;
        if (h < 0 || h >= H) continue;
        for (int s = 0; s < S; ++s) {
            const int ww = q * st + s - pad;
            if (ww < 0 || ww >= W) continue;
            for (int c = 0; c < C; ++c) acc += x[IDX4(n, h, ww, c, H, W, C)] * w[IDX4(k, r, s, c, R, S, C)];
        }
    }
    return acc;
}

/* dx at one input element, gathered: the outputs (p,q) whose window placed  */
/* tap (r,s) on (h,w) are those with p*st = h + pad - r (exact division).    */
double orc_conv2d_dgrad_at(const double* dy, const double* w, int N, int H, int W, int C, int K, int R, int S,
                           int st, int pad, int n, int h, int ww, int c)
{
    (void)N;
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, S, st, pad);
    double acc = 0.0;
    for (int r = 0; r < R; ++r) {
        const int ph = h + pad - r;
        if (ph < 0 || ph % st) continue;
        const int p = ph / st;
        if (p >= P) continue;
        for (int s = 0; s < S; ++s) {
            const int qw = ww + pad - s;
            if (qw < 0 || qw % st) continue;
            const int q = qw / st;
            if (q >= Q) continue;
            for (int k = 0; k < K; ++k) acc += dy[IDX4(n, p, q, k, P, Q, K)] * w[IDX4(k, r, s, c, R, S, C)];
        }
    }
    return acc;
}

double orc_conv2d_wgrad_at(const double* x, const double* dy, int N, int H, int W, int C, int K, int R, int S,
                           int st, int pad, int k, int r, int s, int c)
{
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, S, st, pad);
    double acc = 0.0;
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < P; ++p) {
            const int h = p * st + r - pad;
            if (h < 0 || h >= H) continue;
            for (int q = 0; q < Q; ++q) {
                const int ww = q * st + s - pad;
                if (ww < 0 || ww >= W) continue;
                acc += dy[IDX4(n, p, q, k, P, Q, K)] * x[IDX4(n, h, ww, c, H, W, C)];
            }
        }
    return acc;
}

/* ------------------------------------------------------------------------ */
/* BatchNorm in training mode over the M = N*H*W rows of a [M, C] matrix.    */
/* mean_c = (1/M) sum y, var_c = (1/M) sum (y - mean)^2 (biased),            */
/* xhat = (y - mean)/sqrt(var + eps), out = gamma*xhat + beta [+ res],       */
/* then ReLU (max(0, .)) when relu != 0.                                     */
/* ------------------------------------------------------------------------ */
void orc_bn_fwd(const double* y, int64_t M, int C, const double* gamma, const double* beta, double eps,
                const double* res, int relu, double* out, double* mean, double* invstd)
{
#pragma omp parallel for schedule(static)
    for (int c = 0; c < C; ++c) {
        double s = 0.0;
        for (int64_t m = 0; m < M; ++m) s += y[m * C + c];
        const double mu = s / (double)M;
        double v = 0.0;
        for (int64_t m = 0; m < M; ++m) {
            const double d = y[m * C + c] - mu;
            v += d * d;
        }
        v /= (double)M;
        mean[c] = mu;
        invstd[c] = 1.0 / sqrt(v + eps);
    }
#pragma omp parallel for schedule(static)
    for (int64_t m = 0; m < M; ++m)
        for (int c = 0; c < C; ++c) {
            double o = gamma[c] * (y[m * C + c] - mean[c]) * invstd[c] + beta[c];
            if (res) o += res[m * C + c];
            if (relu && !(o > 0.0)) o = 0.0;
            out[m * C + c] = o;
        }
}

/* Backward of orc_bn_fwd.  g = (dout [+ dout2]) * [out > 0] (ReLU'(0) = 0), */
/* the gradient reaching gamma*xhat + beta [+ res].                          */
/*   dbeta = sum g, dgamma = sum g*xhat,                                     */
/*   dy = gamma*invstd*(g - dbeta/M - xhat*dgamma/M),                        */
/*   dres = g (the residual branch's gradient).                              */
void orc_bn_bwd(const double* dout, const double* dout2, const double* out, int relu, const double* y, int64_t M,
                int C, const double* gamma, const double* mean, const double* invstd, double* dy, double* dres,
                double* dgamma, double* dbeta)
{
#pragma omp parallel for schedule(static)
    for (int c = 0; c < C; ++c) {
        double sg = 0.0, sgx = 0.0;
        for (int64_t m = 0; m < M; ++m) {
            double g = dout[m * C + c] + (dout2 ? dout2[m * C + c] : 0.0);
            if (relu && !(out[m * C + c] > 0.0)) g = 0.0;
            const double xh = (y[m * C + c] - mean[c]) * invstd[c];
            sg += g;
            sgx += g * xh;
        }
        dbeta[c] = sg;
        dgamma[c] = sgx;
        for (int64_t m = 0; m < M; ++m) {
            double g = dout[m * C + c] + (dout2 ? dout2[m * C + c] : 0.0);
            if (relu && !(out[m * C + c] > 0.0)) g = 0.0;
            const double xh = (y[m * C + c] - mean[c]) * invstd[c];
            dy[m * C + c] = gamma[c] * invstd[c] * (g - sg / (double)M - xh * sgx / (double)M);
            if (dres) dres[m * C + c] = g;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* Max pooling, window R x R, stride st, padding pad (ImageNet stem: 3,2,1). */
/* Padding counts as -infinity.  Tie rule (paper silent): the first maximum  */
/* in row-major (r, s) window order is the argmax and takes all the gradient.*/
/* ------------------------------------------------------------------------ */
void orc_maxpool_fwd(const double* x, int N, int H, int W, int C, int R, int st, int pad, double* y, int32_t* arg)
{
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, R, st, pad);
#pragma omp parallel for collapse(2) schedule(static)
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < P; ++p)
            for (int q = 0; q < Q; ++q)
                for (int c = 0; c < C; ++c) {
                    double best = -INFINITY;
                    int bi = -1;
                    for (int r = 0; r < R; ++r)
                        for (int s = 0; s < R; ++s) {
                            const int h = p * st + r - pad, ww = q * st + s - pad;
                            if (h < 0 || h >= H || ww < 0 || ww >= W) continue;
                            const double v = x[IDX4(n, h, ww, c, H, W, C)];
                            if (v > best) {
                                best = v;
                                bi = r * R + s;
                            }
                        }
                    y[IDX4(n, p, q, c, P, Q, C)] = best;
                    if (arg) arg[IDX4(n, p, q, c, P, Q, C)] = bi;
                }
}

void orc_maxpool_bwd(const double* dy, const int32_t* arg, int N, int H, int W, int C, int R, int st, int pad,
                     double* dx)
{
    const int P = out_dim(H, R, st, pad), Q = out_dim(W, R, st, pad);
    memset(dx, 0, sizeof(double) * (size_t)N * H * W * C);
#pragma omp parallel for schedule(static)
    for (int n = 0; n < N; ++n)
        for (int p = 0; p < P; ++p)
            for (int q = 0; q < Q; ++q)
                for (int c = 0; c < C; ++c) {
                    const int a = arg[IDX4(n, p, q, c, P, Q, C)];
                    const int h = p * st + a / R - pad, ww = q * st + a % R - pad;
                    dx[IDX4(n, h, ww, c, H, W, C)] += dy[IDX4(n, p, q, c, P, Q, C)];
                }
}

/* ------------------------------------------------------------------------ */
/* Head: global average pooling (Sec. 6 notes the global pooling layer that  */
/* makes the network resolution-agnostic), one fully connected layer with   */
/* bias (Sec. 5.1.1), softmax cross-entropy averaged over the batch         */
/* (the 1/n of Eq. 1).                                                       */
/* ------------------------------------------------------------------------ */
void orc_avgpool_fwd(const double* x, int N, int HW, int C, double* f)
{
    for (int n = 0; n < N; ++n)
        for (int c = 0; c < C; ++c) {
            double s = 0.0;
            for (int i = 0; i < HW; ++i) s += x[((int64_t)n * HW + i) * C + c];
            f[(int64_t)n * C + c] = s / (double)HW;
        }
}

void orc_avgpool_bwd(const double* df, int N, int HW, int C, double* dx)
{
    for (int n = 0; n < N; ++n)
        for (int i = 0; i < HW; ++i)
            for (int c = 0; c < C; ++c) dx[((int64_t)n * HW + i) * C + c] = df[(int64_t)n * C + c] / (double)HW;
}

/* logits[n,j] = sum_c f[n,c] W[j,c] + b[j] */
void orc_fc_fwd(const double* f, const double* Wt, const double* b, int N, int C, int J, double* logits)
{
    for (int n = 0; n < N; ++n)
        for (int j = 0; j < J; ++j) {
            double s = b[j];
            for (int c = 0; c < C; ++c) s += f[(int64_t)n * C + c] * Wt[(int64_t)j * C + c];
            logits[(int64_t)n * J + j] = s;
        }
}

/* dW[j,c] = sum_n dl[n,j] f[n,c]; db[j] = sum_n dl[n,j]; df[n,c] = sum_j dl[n,j] W[j,c] */
void orc_fc_bwd(const double* dl, const double* f, const double* Wt, int N, int C, int J, double* dW, double* db,
                double* df)
{
    for (int j = 0; j < J; ++j) {
        double sb = 0.0;
        for (int n = 0; n < N; ++n) sb += dl[(int64_t)n * J + j];
        db[j] = sb;
        for (int c = 0; c < C; ++c) {
            double s = 0.0;
            for (int n = 0; n < N; ++n) s += dl[(int64_t)n * J + j] * f[(int64_t)n * C + c];
            dW[(int64_t)j * C + c] = s;
        }
    }
    for (int n = 0; n < N; ++n)
        for (int c = 0; c < C; ++c) {
            double s = 0.0;
            for (int j = 0; j < J; ++j) s += dl[(int64_t)n * J + j] * Wt[(int64_t)j * C + c];
            df[(int64_t)n * C + c] = s;
        }
}

/* loss = (1/N) sum_n [ log sum_j exp(l[n,j]) - l[n, label_n] ];            */
/* dlogits[n,j] = (softmax(l[n])_j - [j == label_n]) / N.                    */
double orc_softmax_ce(const double* logits, const int32_t* labels, int N, int J, double* dlogits)
{
    double loss = 0.0;
    for (int n = 0; n < N; ++n) {
        const double* l = logits + (int64_t)n * J;
        double mx = l[0];
        for (int j = 1; j < J; ++j)
            if (l[j] > mx) mx = l[j];
        double z = 0.0;
        for (int j = 0; j < J; ++j) z += exp(l[j] - mx);
        const double lse = mx + log(z);
        loss += lse - l[labels[n]];
        for (int j = 0; j < J; ++j) {
            const double p = exp(l[j] - lse);
            dlogits[(int64_t)n * J + j] = (p - (j == labels[n] ? 1.0 : 0.0)) / (double)N;
        }
    }
    return loss / (double)N;
}

/* ------------------------------------------------------------------------ */
/* Dropout before the fully connected layer.  Cyclic progressive learning   */
/* raises the dropout rate d with the resolution inside each stage          */
/* (Sec. 4.1; Tables 7 and 9 give 0.1 / 0.2 / 0.3).  The paper gives no     */
/* formula; the reading is inverted dropout on the pooled features, as in   */
/* the framework it used: each feature is kept with probability 1 - d and */
/* a kept feature is divided by 1 - d, so its expectation is unchanged.     */
/*                                                                          */
/* The random draw is the counter-based generator Philox4x64-10 (Salmon,    */
/* Moraes, Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3",    */
/* SC 2011), written from that definition: a 256-bit counter and a 128-bit  */
/* key, ten rounds, each multiplying counter words 0 and 2 by the two round */
/* multipliers (full 128-bit products), then                                */
/*     (c0, c1, c2, c3) <- (hi(M1*c2) ^ c1 ^ k0, lo(M1*c2),                 */
/*                          hi(M0*c0) ^ c3 ^ k1, lo(M0*c0)),                */
/* with the key advanced by the two Weyl constants between rounds.          */
/* ------------------------------------------------------------------------ */
static void mul_hilo64(uint64_t a, uint64_t b, uint64_t* hi, uint64_t* lo)
{
    /* schoolbook product of 32-bit halves */
    const uint64_t a0 = a & 0xffffffffu, a1 = a >> 32, b0 = b & 0xffffffffu, b1 = b >> 32;
    const uint64_t p00 = a0 * b0, p01 = a0 * b1, p10 = a1 * b0, p11 = a1 * b1;
    const uint64_t mid = (p00 >> 32) + (p01 & 0xffffffffu) + (p10 & 0xffffffffu);
    *lo = (mid << 32) | (p00 & 0xffffffffu);
    *hi = p11 + (p01 >> 32) + (p10 >> 32) + (mid >> 32);
}

void orc_philox4x64_10(const uint64_t ctr[4], const uint64_t key[2], uint64_t out[4])
{
    const uint64_t M0 = 0xD2E7470EE14C6C93ull, M1 = 0xCA5A826395121157ull;
    const uint64_t W0 = 0x9E3779B97F4A7C15ull, W1 = 0xBB67AE8584CAA73Bull;
    uint64_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3], k0 = key[0], k1 = key[1];
    for (int round = 0; round < 10; ++round) {
        if (round > 0) {
            k0 += W0;
            k1 += W1;
        }
        uint64_t hi0, lo0, hi1, lo1;
        mul_hilo64(M0, c0, &hi0, &lo0);
        mul_hilo64(M1, c2, &hi1, &lo1);
        const uint64_t n0 = hi1 ^ c1 ^ k0, n1 = lo1, n2 = hi0 ^ c3 ^ k1, n3 = lo0;
        c0 = n0;
        c1 = n1;
        c2 = n2;
        c3 = n3;
    }
    out[0] = c0;
    out[1] = c1;
    out[2] = c2;
    out[3] = c3;
}

/* keep[n,c] for N samples of C features (C a multiple of 4): feature c of   */
/* sample n takes word c % 4 of Philox4x64-10 at counter                     */
/* (n*C/4 + c/4, step, 0, 0) with key (seed, 0), and is kept when the word's */
/* upper 32 bits, as an integer, are at least floor(d * 2^32).               */
void orc_dropout_mask(int N, int C, double d, uint64_t seed, uint64_t step, uint8_t* keep)
{
    const uint64_t thr = (uint64_t)floor(d * 4294967296.0);
    const uint64_t key[2] = {seed, 0};
    for (int n = 0; n < N; ++n)
        for (int g = 0; g < C / 4; ++g) {
            const uint64_t ctr[4] = {(uint64_t)n * (uint64_t)(C / 4) + (uint64_t)g, step, 0, 0};
            uint64_t r[4];
            orc_philox4x64_10(ctr, key, r);
            for (int j = 0; j < 4; ++j) keep[(int64_t)n * C + 4 * g + j] = (uint8_t)((r[j] >> 32) >= thr);
        }
}

/* out = keep * x / (1 - d): the forward map, and (it is linear and          */
/* diagonal) also the backward map of a gradient.                           */
void orc_dropout_apply(const double* x, const uint8_t* keep, int64_t n, double d, double* out)
{
    for (int64_t i = 0; i < n; ++i) out[i] = keep[i] ? x[i] / (1.0 - d) : 0.0;
}

/* ------------------------------------------------------------------------ */
/* Parameter-server merge of the two workers' pushes (Sec. 3.4 with Eq. 1). */
/* Each push i carries its worker's batch-mean gradient g_i and is scaled by */
/* the model-update factor f_i (f_L = 1, f_S = d_S/d_L or its square root).  */
/* The server's optimizer is SGD with momentum in the form                  */
/*     u <- mu*u - lr*f_i*g_i ;  w <- w + u                                  */
/* (reduces to Eq. 1 when mu = 0).  Under ASP the server applies each push  */
/* as it arrives (Sec. 2.4):                                                 */
/*   order 0: large push, then small push (two momentum steps),             */
/*   order 1: small push, then large push,                                   */
/*   order 2: both pushes summed into one step (the synchronous reading).   */
/* A NULL gradient is a worker that did not push in this round.             */
/* ------------------------------------------------------------------------ */
void orc_ps_merge(double* w, double* u, const double* gL, const double* gS, int64_t n, double lr, double mu,
                  double fL, double fS, int order)
{
    for (int64_t i = 0; i < n; ++i) {
        double wi = w[i], ui = u[i];
        if (order == 2) {
            double g = 0.0;
            if (gL) g += fL * gL[i];
            if (gS) g += fS * gS[i];
            ui = mu * ui - lr * g;
            wi = wi + ui;
        } else {
            const double* first = order == 0 ? gL : gS;
            const double* second = order == 0 ? gS : gL;
            const double ff = order == 0 ? fL : fS, fs = order == 0 ? fS : fL;
            if (first) {
                ui = mu * ui - lr * ff * first[i];
                wi = wi + ui;
            }
            if (second) {
                ui = mu * ui - lr * fs * second[i];
                wi = wi + ui;
            }
        }
        w[i] = wi;
        u[i] = ui;
    }
}

/* The merge under mixed precision with loss scaling (Micikevicius et al.,   */
/* the method the paper cites for its fp16 runs, Sec. 5.2.3).  A worker      */
/* computes its gradient from a loss multiplied by its scale S_i, so it      */
/* pushes S_i * g_i; the server divides each push by its scale before the   */
/* momentum update above.  If any pushed value is not finite (the scaled    */
/* gradient overflowed fp16 somewhere), the server applies nothing: w and u  */
/* are left as they are.  Returns 1 when the update was applied, 0 when it  */
/* was skipped.                                                              */
int orc_ps_merge_scaled(double* w, double* u, const double* gL, const double* gS, int64_t n, double lr, double mu,
                        double fL, double fS, int order, double sL, double sS)
{
    for (int64_t i = 0; i < n; ++i)
        if ((gL && !isfinite(gL[i])) || (gS && !isfinite(gS[i]))) return 0;
    double* uL = gL ? (double*)malloc(sizeof(double) * (size_t)(n ? n : 1)) : NULL;
    double* uS = gS ? (double*)malloc(sizeof(double) * (size_t)(n ? n : 1)) : NULL;
    for (int64_t i = 0; i < n; ++i) {
        if (uL) uL[i] = gL[i] / sL;
        if (uS) uS[i] = gS[i] / sS;
    }
    orc_ps_merge(w, u, uL, uS, n, lr, mu, fL, fS, order);
    free(uL);
    free(uS);
    return 1;
}

/* Dynamic loss scale: after a step whose gradients overflowed, halve the   */
/* scale and restart the count of good steps; after `interval` good steps   */
/* in a row, double it.                                                     */
void orc_loss_scale_update(double* scale, int* good, int found_inf, int interval)
{
    if (found_inf) {
        *scale = *scale / 2.0;
        *good = 0;
        return;
    }
    *good += 1;
    if (*good >= interval) {
        *scale = *scale * 2.0;
        *good = 0;
    }
}

/* ------------------------------------------------------------------------ */
/* Bilinear downsampling for the low-resolution sub-stages (Sec. 4.1).      */
/* Convention (paper silent): half-pixel centres, no antialiasing, edge     */
/* clamp.  Output j of an axis samples source coordinate                    */
/*     src = (j + 1/2) * in/out - 1/2 = ((2j+1)*in - out) / (2*out),        */
/* taken in exact integers: i0 = floor(num/den), lambda = (num - i0*den)/den,*/
/* i1 = min(i0 + 1, in - 1).  Negative src (upsampling only) clamps to 0.   */
/* ------------------------------------------------------------------------ */
int orc_resize_taps(int in, int out, int32_t* i0, int32_t* i1, double* lam)
{
    if (in <= 0 || out <= 0) return -1;
    for (int j = 0; j < out; ++j) {
        const int64_t num = (int64_t)(2 * j + 1) * in - out;
        const int64_t den = 2 * (int64_t)out;
        int64_t a;
        double l;
        if (num <= 0) {
            a = 0;
            l = 0.0;
        } else {
            a = num / den;
            l = (double)(num - a * den) / (double)den;
        }
        if (a > in - 1) {
            a = in - 1;
            l = 0.0;
        }
        i0[j] = (int32_t)a;
        i1[j] = (int32_t)(a + 1 < in ? a + 1 : in - 1);
        lam[j] = l;
    }
    return 0;
}

/* out[n,y,x,c] = (1-ly)[(1-lx) a + lx b] + ly[(1-lx) c + lx d] */
int orc_bilinear_resize(const double* in, int N, int Hi, int Wi, int C, double* out, int Ho, int Wo)
{
    int32_t *y0 = malloc(sizeof(int32_t) * Ho), *y1 = malloc(sizeof(int32_t) * Ho);
    int32_t *x0 = malloc(sizeof(int32_t) * Wo), *x1 = malloc(sizeof(int32_t) * Wo);
    double *ly = malloc(sizeof(double) * Ho), *lx = malloc(sizeof(double) * Wo);
    int rc = -1;
    if (!y0 || !y1 || !x0 || !x1 || !ly || !lx) goto done;
    orc_resize_taps(Hi, Ho, y0, y1, ly);
    orc_resize_taps(Wi, Wo, x0, x1, lx);
    for (int n = 0; n < N; ++n)
        for (int yy = 0; yy < Ho; ++yy)
            for (int xx = 0; xx < Wo; ++xx)
                for (int c = 0; c < C; ++c) {
                    const double a = in[IDX4(n, y0[yy], x0[xx], c, Hi, Wi, C)];
                    const double b = in[IDX4(n, y0[yy], x1[xx], c, Hi, Wi, C)];
                    const double cc = in[IDX4(n, y1[yy], x0[xx], c, Hi, Wi, C)];
                    const double d = in[IDX4(n, y1[yy], x1[xx], c, Hi, Wi, C)];
                    const double top = (1.0 - lx[xx]) * a + lx[xx] * b;
                    const double bot = (1.0 - lx[xx]) * cc + lx[xx] * d;
                    out[IDX4(n, yy, xx, c, Ho, Wo, C)] = (1.0 - ly[yy]) * top + ly[yy] * bot;
                }
    rc = 0;
done:
    free(y0); free(y1); free(x0); free(x1); free(ly); free(lx);
    return rc;
}
