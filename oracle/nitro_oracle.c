/*
 * CPU oracle for NITRO-D integer-only training (arXiv 2407.11698).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * statement of what the GPU path computes.  Only the test-suite, the smoke
 * check and the CPU-baseline leg of the benchmark may load it.  It shares no
 * code, header or table with the CUDA library.
 *
 * Conventions used throughout (the paper fixes none of them):
 *   activations NHWC  a[((b*H + y)*W + x)*C + c]
 *   conv weights OHWI w[((co*3 + ky)*3 + kx)*Cin + ci]   (3x3, stride 1, pad 1)
 *   linear weights     w[o*In + i]
 *   every value is held in int64; contractions are summed modulo 2^64
 *   (uint64 arithmetic), which equals the exact sum whenever the exact sum
 *   fits int64.  The caller decides, from operand bounds, whether it does.
 *
 * Parallelism: OpenMP over independent output elements only; every output is
 * one sequential sum, so thread count never changes a result.
 */
#include <stdint.h>
#include <stddef.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Threads the contraction loops may use (reported beside CPU timings). */
int64_t nor_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ---------------------------------------------------------------------- */
/* Integer division.  The paper's \intdiv{x}{d} is floor(x / d) (Sec. 3.2,  */
/* Eq. 1 and every later use).  C's "/" truncates toward zero, so a         */
/* negative inexact quotient is moved down by one.  Requires d > 0.         */
/* ---------------------------------------------------------------------- */
int64_t nor_fdiv(int64_t x, int64_t d) {
    int64_t q = x / d;
    int64_t r = x % d;
    if (r < 0) q -= 1;
    return q;
}

/* Element-wise floor division of a vector (same rule as nor_fdiv). */
void nor_fdiv_vec(int64_t n, const int64_t* x, int64_t d, int64_t* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = nor_fdiv(x[i], d);
}

/* Division rounding toward zero: the optional IntegerSGD rounding under   */
/* which Sec. 3.3's remark "|w| < eta_inv gives a zero decay term" holds.  */
int64_t nor_tdiv(int64_t x, int64_t d) { return x / d; }

/* ---------------------------------------------------------------------- */
/* NITRO-ReLU (Sec. 3.2.2).                                                */
/* mu_int8 is the floor-average of the four segment means:                */
/*   x < -127      : floor(-127 / alpha_inv)                               */
/*   -127 <= x <= 0: floor(-127 / (2 alpha_inv))                           */
/*   0 < x <= 127  : 63                                                    */
/*   x > 127       : 127                                                   */
/* ---------------------------------------------------------------------- */
int64_t nor_relu_mu(int64_t alpha_inv) {
    int64_t m1 = nor_fdiv(-127, alpha_inv);
    int64_t m2 = nor_fdiv(-127, 2 * alpha_inv);
    int64_t m3 = 63;
    int64_t m4 = 127;
    return nor_fdiv(m1 + m2 + m3 + m4, 4);
}

/* Forward: x < 0 -> floor(max(x,-127)/alpha_inv) - mu ; x >= 0 -> min(x,127) - mu */
int64_t nor_relu(int64_t x, int64_t alpha_inv, int64_t mu) {
    if (x < 0) {
        int64_t c = x < -127 ? -127 : x;
        return nor_fdiv(c, alpha_inv) - mu;
    }
    return (x > 127 ? 127 : x) - mu;
}

/* Which of the four pieces x falls in (the split the forward definition  */
/* uses):  0: x < -127   1: -127 <= x < 0   2: 0 <= x <= 127   3: x > 127 */
int64_t nor_relu_region(int64_t x) {
    if (x < -127) return 0;
    if (x < 0) return 1;
    if (x <= 127) return 2;
    return 3;
}

/* Backward of NITRO-ReLU (not written in the paper; derivative of each   */
/* piece): saturated pieces pass nothing, the identity piece passes g, the */
/* slope-1/alpha_inv piece passes floor(g / alpha_inv).                    */
int64_t nor_relu_bwd(int64_t g, int64_t region, int64_t alpha_inv) {
    switch (region) {
        case 1: return nor_fdiv(g, alpha_inv);
        case 2: return g;
        default: return 0;
    }
}

/* Vector forms of the element-wise pieces above.                          */
void nor_scale_relu(int64_t n, const int64_t* z, int64_t sf, int64_t alpha_inv,
                    int64_t* zs, int64_t* region, int64_t* act) {
    int64_t mu = nor_relu_mu(alpha_inv);
    for (int64_t i = 0; i < n; ++i) {
        int64_t s = nor_fdiv(z[i], sf);            /* NITRO-Scaling, Eq. 1 */
        zs[i] = s;
        region[i] = nor_relu_region(s);
        act[i] = nor_relu(s, alpha_inv, mu);
    }
}

void nor_relu_bwd_vec(int64_t n, const int64_t* g, const int64_t* region,
                      int64_t alpha_inv, int64_t* out) {
    for (int64_t i = 0; i < n; ++i) out[i] = nor_relu_bwd(g[i], region[i], alpha_inv);
}

/* ---------------------------------------------------------------------- */
/* Integer square root (Sec. 3.3.1 uses the integer-square-root routine):  */
/* the largest r with r*r <= n, by bisection.                              */
/* ---------------------------------------------------------------------- */
int64_t nor_isqrt(int64_t n) {
    if (n <= 0) return 0;
    int64_t lo = 0, hi = 3037000499LL;         /* floor(sqrt(2^63 - 1)) */
    if (hi > n) hi = n;
    while (lo < hi) {
        int64_t mid = lo + (hi - lo + 1) / 2;
        if (mid <= n / mid) lo = mid; else hi = mid - 1;
    }
    return lo;
}

/* Integer Kaiming bound (Sec. 3.3.1): b = floor(128*1732 / (isqrt(fan_in)*1000)) */
int64_t nor_init_bound(int64_t fan_in) {
    return nor_fdiv(128 * 1732, nor_isqrt(fan_in) * 1000);
}

/* ---------------------------------------------------------------------- */
/* SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): the i-th output of a     */
/* generator seeded with s is mix(s + (i+1) * 0x9E3779B97F4A7C15), mix     */
/* being the published 64-bit finaliser.  Random-access form.              */
/* ---------------------------------------------------------------------- */
uint64_t nor_splitmix64_at(uint64_t seed, uint64_t index) {
    uint64_t z = seed + (index + 1ULL) * 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Weight draw for tensor `tensor_id` of a block: element e (canonical     */
/* order) takes output number tensor_id * 2^40 + e and maps it onto the    */
/* integers -b..b by u mod (2b+1) - b (the uniform law of Sec. 3.3.1).     */
void nor_init_uniform(int64_t n, int64_t bound, uint64_t seed, uint64_t tensor_id,
                      int64_t* w) {
    uint64_t span = (uint64_t)(2 * bound + 1);
    for (int64_t e = 0; e < n; ++e) {
        uint64_t u = nor_splitmix64_at(seed, (tensor_id << 40) + (uint64_t)e);
        w[e] = (int64_t)(u % span) - bound;
    }
}

/* ---------------------------------------------------------------------- */
/* 3x3 convolution, stride 1, zero padding 1 (Table 1 caption), and its    */
/* two adjoints.  The forward sum is the conv expression of Sec. 3.2.1:    */
/*   z[b,y,x,co] = sum_{ky,kx,ci} a[b, y+ky-1, x+kx-1, ci] * w[co,ky,kx,ci] */
/* ---------------------------------------------------------------------- */
void nor_conv3x3_fwd(int64_t B, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                     const int64_t* a, const int64_t* w, int64_t* z) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int64_t b = 0; b < B; ++b)
        for (int64_t y = 0; y < H; ++y)
            for (int64_t x = 0; x < W; ++x)
                for (int64_t co = 0; co < Cout; ++co) {
                    uint64_t s = 0;
                    for (int64_t ky = 0; ky < 3; ++ky)
                        for (int64_t kx = 0; kx < 3; ++kx) {
                            int64_t iy = y + ky - 1, ix = x + kx - 1;
                            if (iy < 0 || iy >= H || ix < 0 || ix >= W) continue;
                            const int64_t* ap = a + ((b * H + iy) * W + ix) * Cin;
                            const int64_t* wp = w + ((co * 3 + ky) * 3 + kx) * Cin;
                            for (int64_t ci = 0; ci < Cin; ++ci)
                                s += (uint64_t)ap[ci] * (uint64_t)wp[ci];
                        }
                    z[((b * H + y) * W + x) * Cout + co] = (int64_t)s;
                }
}

/* Input gradient: g_in[b,y,x,ci] = sum over every output (b,oy,ox,co) that */
/* read input pixel (y,x) through tap (ky,kx): oy = y-ky+1, ox = x-kx+1.    */
void nor_conv3x3_dgrad(int64_t B, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                       const int64_t* g_out, const int64_t* w, int64_t* g_in) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int64_t b = 0; b < B; ++b)
        for (int64_t y = 0; y < H; ++y)
            for (int64_t x = 0; x < W; ++x)
                for (int64_t ci = 0; ci < Cin; ++ci) {
                    uint64_t s = 0;
                    for (int64_t ky = 0; ky < 3; ++ky)
                        for (int64_t kx = 0; kx < 3; ++kx) {
                            int64_t oy = y - ky + 1, ox = x - kx + 1;
                            if (oy < 0 || oy >= H || ox < 0 || ox >= W) continue;
                            const int64_t* gp = g_out + ((b * H + oy) * W + ox) * Cout;
                            for (int64_t co = 0; co < Cout; ++co)
                                s += (uint64_t)gp[co] *
                                     (uint64_t)w[((co * 3 + ky) * 3 + kx) * Cin + ci];
                        }
                    g_in[((b * H + y) * W + x) * Cin + ci] = (int64_t)s;
                }
}

/* Weight gradient: dw[co,ky,kx,ci] = sum_{b,y,x} g_out[b,y,x,co] * a[b,y+ky-1,x+kx-1,ci] */
void nor_conv3x3_wgrad(int64_t B, int64_t H, int64_t W, int64_t Cin, int64_t Cout,
                       const int64_t* a, const int64_t* g_out, int64_t* dw) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int64_t co = 0; co < Cout; ++co)
        for (int64_t t = 0; t < 9; ++t) {
            int64_t ky = t / 3, kx = t % 3;
            for (int64_t ci = 0; ci < Cin; ++ci) {
                uint64_t s = 0;
                for (int64_t b = 0; b < B; ++b)
                    for (int64_t y = 0; y < H; ++y)
                        for (int64_t x = 0; x < W; ++x) {
                            int64_t iy = y + ky - 1, ix = x + kx - 1;
                            if (iy < 0 || iy >= H || ix < 0 || ix >= W) continue;
                            s += (uint64_t)g_out[((b * H + y) * W + x) * Cout + co] *
                                 (uint64_t)a[((b * H + iy) * W + ix) * Cin + ci];
                        }
                dw[((co * 3 + ky) * 3 + kx) * Cin + ci] = (int64_t)s;
            }
        }
}

/* ---------------------------------------------------------------------- */
/* Linear layer (Sec. 3.2.1): z[b,o] = sum_i a[b,i] * w[o,i], and adjoints. */
/* ---------------------------------------------------------------------- */
void nor_linear_fwd(int64_t B, int64_t In, int64_t Out,
                    const int64_t* a, const int64_t* w, int64_t* z) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int64_t b = 0; b < B; ++b)
        for (int64_t o = 0; o < Out; ++o) {
            uint64_t s = 0;
            for (int64_t i = 0; i < In; ++i)
                s += (uint64_t)a[b * In + i] * (uint64_t)w[o * In + i];
            z[b * Out + o] = (int64_t)s;
        }
}

void nor_linear_dgrad(int64_t B, int64_t In, int64_t Out,
                      const int64_t* g_out, const int64_t* w, int64_t* g_in) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int64_t b = 0; b < B; ++b)
        for (int64_t i = 0; i < In; ++i) {
            uint64_t s = 0;
            for (int64_t o = 0; o < Out; ++o)
                s += (uint64_t)g_out[b * Out + o] * (uint64_t)w[o * In + i];
            g_in[b * In + i] = (int64_t)s;
        }
}

void nor_linear_wgrad(int64_t B, int64_t In, int64_t Out,
                      const int64_t* a, const int64_t* g_out, int64_t* dw) {
    #pragma omp parallel for collapse(2) schedule(static)
    for (int64_t o = 0; o < Out; ++o)
        for (int64_t i = 0; i < In; ++i) {
            uint64_t s = 0;
            for (int64_t b = 0; b < B; ++b)
                s += (uint64_t)g_out[b * Out + o] * (uint64_t)a[b * In + i];
            dw[o * In + i] = (int64_t)s;
        }
}

/* ---------------------------------------------------------------------- */
/* MaxPool2D 2x2 stride 2 (Table 1 caption).  Output size floor(H/2) x     */
/* floor(W/2).  Window scan order (0,0),(0,1),(1,0),(1,1); the first       */
/* maximum wins and its position 0..3 is recorded for the backward pass.   */
/* ---------------------------------------------------------------------- */
void nor_maxpool_fwd(int64_t B, int64_t H, int64_t W, int64_t C,
                     const int64_t* a, int64_t* out, int64_t* argmax) {
    int64_t Ho = H / 2, Wo = W / 2;
    for (int64_t b = 0; b < B; ++b)
        for (int64_t y = 0; y < Ho; ++y)
            for (int64_t x = 0; x < Wo; ++x)
                for (int64_t c = 0; c < C; ++c) {
                    int64_t best = 0, bestv = 0;
                    for (int64_t k = 0; k < 4; ++k) {
                        int64_t iy = 2 * y + k / 2, ix = 2 * x + k % 2;
                        int64_t v = a[((b * H + iy) * W + ix) * C + c];
                        if (k == 0 || v > bestv) { bestv = v; best = k; }
                    }
                    out[((b * Ho + y) * Wo + x) * C + c] = bestv;
                    argmax[((b * Ho + y) * Wo + x) * C + c] = best;
                }
}

/* Routes each pooled gradient to the recorded window position; every     */
/* other input position (and the rows/columns dropped by the floor) gets 0. */
void nor_maxpool_bwd(int64_t B, int64_t H, int64_t W, int64_t C,
                     const int64_t* g_out, const int64_t* argmax, int64_t* g_in) {
    int64_t Ho = H / 2, Wo = W / 2;
    for (int64_t i = 0; i < B * H * W * C; ++i) g_in[i] = 0;
    for (int64_t b = 0; b < B; ++b)
        for (int64_t y = 0; y < Ho; ++y)
            for (int64_t x = 0; x < Wo; ++x)
                for (int64_t c = 0; c < C; ++c) {
                    int64_t o = ((b * Ho + y) * Wo + x) * C + c;
                    int64_t k = argmax[o];
                    int64_t iy = 2 * y + k / 2, ix = 2 * x + k % 2;
                    g_in[((b * H + iy) * W + ix) * C + c] = g_out[o];
                }
}

/* ---------------------------------------------------------------------- */
/* Learning-layer pooling (Sec. 3.3 training iteration: a block's output   */
/* is downsampled by a pooling layer, z^mp, before its learning layers;    */
/* App. B fixes the learning layers' input size d^lr).  A kh x kw max-pool */
/* with stride (kh, kw); output floor(H/kh) x floor(W/kw).  The window is  */
/* scanned row by row, the first maximum wins, and its position            */
/* r * kw + s (row r, column s of the window) is recorded for backward.    */
/* ---------------------------------------------------------------------- */
void nor_winpool_fwd(int64_t B, int64_t H, int64_t W, int64_t C, int64_t kh, int64_t kw,
                     const int64_t* a, int64_t* out, int64_t* argmax) {
    int64_t Ho = H / kh, Wo = W / kw;
    for (int64_t b = 0; b < B; ++b)
        for (int64_t y = 0; y < Ho; ++y)
            for (int64_t x = 0; x < Wo; ++x)
                for (int64_t c = 0; c < C; ++c) {
                    int64_t best = 0, bestv = 0;
                    for (int64_t r = 0; r < kh; ++r)
                        for (int64_t s = 0; s < kw; ++s) {
                            int64_t v = a[((b * H + y * kh + r) * W + x * kw + s) * C + c];
                            if ((r == 0 && s == 0) || v > bestv) { bestv = v; best = r * kw + s; }
                        }
                    out[((b * Ho + y) * Wo + x) * C + c] = bestv;
                    argmax[((b * Ho + y) * Wo + x) * C + c] = best;
                }
}

/* Backward of nor_winpool_fwd: each pooled gradient goes to the recorded  */
/* window position; every other position, and the rows and columns the    */
/* floor drops, get 0.                                                     */
void nor_winpool_bwd(int64_t B, int64_t H, int64_t W, int64_t C, int64_t kh, int64_t kw,
                     const int64_t* g_out, const int64_t* argmax, int64_t* g_in) {
    int64_t Ho = H / kh, Wo = W / kw;
    for (int64_t i = 0; i < B * H * W * C; ++i) g_in[i] = 0;
    for (int64_t b = 0; b < B; ++b)
        for (int64_t y = 0; y < Ho; ++y)
            for (int64_t x = 0; x < Wo; ++x)
                for (int64_t c = 0; c < C; ++c) {
                    int64_t o = ((b * Ho + y) * Wo + x) * C + c;
                    int64_t k = argmax[o];
                    int64_t iy = y * kh + k / kw, ix = x * kw + k % kw;
                    g_in[((b * H + iy) * W + ix) * C + c] = g_out[o];
                }
}

/* ---------------------------------------------------------------------- */
/* Dropout of the linear blocks (App. B, rate p_l).  The paper gives no    */
/* integer form; the reading used: a dropped activation becomes 0 (the     */
/* centre of the NITRO-ReLU output, which is shifted by mu) with no        */
/* rescaling, and passes no gradient.  p is given in units of 2^-16        */
/* (p16 in 0..65536).  Element e = b * out_features + j of forward layer   */
/* `layer` at training step t is dropped when the top 16 bits of output    */
/* 2^63 + t * 2^35 + layer * 2^31 + e of the block's SplitMix64 stream are */
/* below p16 (t is taken modulo 2^28).                                     */
/* ---------------------------------------------------------------------- */
int64_t nor_dropout_drop(uint64_t seed, uint64_t step, uint64_t layer, uint64_t e, int64_t p16) {
    uint64_t idx = (1ULL << 63) + ((step & ((1ULL << 28) - 1)) << 35) + (layer << 31) + e;
    uint64_t u = nor_splitmix64_at(seed, idx);
    return (int64_t)(u >> 48) < p16;
}

void nor_dropout_mask(int64_t n, uint64_t seed, uint64_t step, uint64_t layer, int64_t p16,
                      int64_t* drop) {
    for (int64_t e = 0; e < n; ++e) drop[e] = nor_dropout_drop(seed, step, layer, (uint64_t)e, p16);
}

/* ---------------------------------------------------------------------- */
/* IntegerSGD, Algorithm 1.  For every weight:                             */
/*   d = R(dw, gamma_inv);  if eta_inv != 0: d += R(w, eta_inv);  w -= d   */
/* R is floor division (round_mode 0, the paper's notation) or truncation  */
/* toward zero (round_mode 1).  The result is left in int64; the caller    */
/* checks that it still fits the int32 weight storage.                     */
/* ---------------------------------------------------------------------- */
void nor_integersgd(int64_t n, int64_t* w, const int64_t* dw, int64_t gamma_inv,
                    int64_t eta_inv, int64_t round_mode) {
    for (int64_t i = 0; i < n; ++i) {
        int64_t d = round_mode ? nor_tdiv(dw[i], gamma_inv) : nor_fdiv(dw[i], gamma_inv);
        if (eta_inv != 0)
            d += round_mode ? nor_tdiv(w[i], eta_inv) : nor_fdiv(w[i], eta_inv);
        w[i] = w[i] - d;
    }
}

/* ---------------------------------------------------------------------- */
/* Integer data pre-processing, App. A.  Over the n 8-bit values x of a    */
/* dataset (every element of every sample counts once):                    */
/*   mu    = floor(sum_i x_i / n)                                          */
/*   omega = floor(sum_i |x_i - mu| / n)     (mean absolute deviation)     */
/*   x_hat = floor((x_i - mu) * 51 / omega)  (51 = floor(64 * 0.8))        */
/* Readings where the appendix is silent: omega = 0 divides by 1, and      */
/* x_hat is stored as int8 clamped to [-127, 127], the interval the        */
/* appendix names as the int8 range the output is meant to fill.           */
/* ---------------------------------------------------------------------- */
void nor_prep_stats(int64_t n, const uint8_t* x, int64_t* mu, int64_t* omega) {
    int64_t s = 0;
    for (int64_t i = 0; i < n; ++i) s += x[i];
    const int64_t m = nor_fdiv(s, n);
    int64_t a = 0;
    for (int64_t i = 0; i < n; ++i) {
        const int64_t dv = (int64_t)x[i] - m;
        a += dv < 0 ? -dv : dv;
    }
    *mu = m;
    *omega = nor_fdiv(a, n);
}

void nor_prep_apply(int64_t n, const uint8_t* x, int64_t mu, int64_t omega, int8_t* out) {
    const int64_t div = omega > 0 ? omega : 1;
    for (int64_t i = 0; i < n; ++i) {
        int64_t v = nor_fdiv(((int64_t)x[i] - mu) * 51, div);
        if (v < -127) v = -127;
        if (v > 127) v = 127;
        out[i] = (int8_t)v;
    }
}
