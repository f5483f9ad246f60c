// CUDA-core kernels of the NITRO-D block step: an exact int64 implicit GEMM
// for every contraction shape (conv 3x3 fwd / dgrad / wgrad, linear fwd /
// dgrad / wgrad), and the element-wise stages fused around it (NITRO-Scaling,
// NITRO-ReLU and max-pool forward, with dropout for linear layers; max-pool,
// NITRO-ReLU backward and STE; the learning layer, its max-pool to d_lr and
// the RSS loss; IntegerSGD).
//
// The GEMM serves the contractions the tensor-core path does not take (narrow
// or small layers, linear weight and input gradients, linear forwards whose
// input width is not a multiple of 8); the learning layer (G = 10 outputs) and
// the element-wise stages always run here.
#include <cuda_bf16.h>

#include <algorithm>

#include "nitro_internal.cuh"
#include "prof.cuh"

namespace nitro {
namespace {

constexpr int kTile = 64;   // M and N tile
constexpr int kTK = 16;     // K slab
constexpr unsigned kFull = 0xffffffffu;

struct GemmParams {
    const int8_t* act;
    const int32_t* grad;
    const int32_t* wts;
    int64_t* out;
    int M, N, K;
    int B, H, W, Cin, Cout;
    int k_split;
};

// Operand element A[m][k] / B[n][k] of each contraction (see GemmMode).
template <int MODE>
__device__ __forceinline__ int32_t load_a(const GemmParams& p, int m, int k) {
    if (MODE == GM_CONV_FWD || MODE == GM_CONV_DGRAD) {
        const int hw = p.H * p.W;
        const int b = m / hw, r = m - b * hw, y = r / p.W, x = r - y * p.W;
        const int C = MODE == GM_CONV_FWD ? p.Cin : p.Cout;
        const int t = k / C, c = k - t * C, ky = t / 3, kx = t - 3 * ky;
        // forward reads input (y+ky-1, x+kx-1); dgrad reads output (y-ky+1, x-kx+1)
        const int iy = MODE == GM_CONV_FWD ? y + ky - 1 : y - ky + 1;
        const int ix = MODE == GM_CONV_FWD ? x + kx - 1 : x - kx + 1;
        if (iy < 0 || iy >= p.H || ix < 0 || ix >= p.W) return 0;
        const int64_t idx = ((int64_t)(b * p.H + iy) * p.W + ix) * C + c;
        return MODE == GM_CONV_FWD ? (int32_t)p.act[idx] : p.grad[idx];
    } else if (MODE == GM_CONV_WGRAD) {
        return p.grad[(int64_t)k * p.Cout + m];
    } else if (MODE == GM_LIN_FWD) {
        return p.act[(int64_t)m * p.Cin + k];
    } else if (MODE == GM_LIN_DGRAD) {
        return p.grad[(int64_t)m * p.Cout + k];
    } else {  // GM_LIN_WGRAD
        return p.grad[(int64_t)k * p.Cout + m];
    }
}

template <int MODE>
__device__ __forceinline__ int32_t load_b(const GemmParams& p, int n, int k) {
    if (MODE == GM_CONV_FWD) {
        return p.wts[(int64_t)n * 9 * p.Cin + k];
    } else if (MODE == GM_CONV_DGRAD) {
        const int t = k / p.Cout, co = k - t * p.Cout;
        return p.wts[((int64_t)co * 9 + t) * p.Cin + n];
    } else if (MODE == GM_CONV_WGRAD) {
        const int t = n / p.Cin, ci = n - t * p.Cin, ky = t / 3, kx = t - 3 * ky;
        const int hw = p.H * p.W;
        const int b = k / hw, r = k - b * hw, y = r / p.W, x = r - y * p.W;
        const int iy = y + ky - 1, ix = x + kx - 1;
        if (iy < 0 || iy >= p.H || ix < 0 || ix >= p.W) return 0;
        return p.act[((int64_t)(b * p.H + iy) * p.W + ix) * p.Cin + ci];
    } else if (MODE == GM_LIN_FWD) {
        return p.wts[(int64_t)n * p.Cin + k];
    } else if (MODE == GM_LIN_DGRAD) {
        return p.wts[(int64_t)k * p.Cin + n];
    } else {  // GM_LIN_WGRAD
        return p.act[(int64_t)k * p.Cin + n];
    }
}

// 64x64 output tile per CTA, 4x4 per thread, int64 accumulators.  With
// gridDim.z > 1 each CTA sums one K slice and adds it into a zeroed `out`
// with 64-bit integer atomics (exact and order-independent).
template <int MODE>
__global__ void __launch_bounds__(256) k_gemm(GemmParams p) {
    pdl_wait();
    __shared__ int32_t As[kTK][kTile + 4];
    __shared__ int32_t Bs[kTK][kTile + 4];
    const int m0 = blockIdx.y * kTile, n0 = blockIdx.x * kTile;
    const int kb = blockIdx.z * p.k_split;
    const int ke = min(p.K, kb + p.k_split);
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    int64_t acc[4][4];
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[r][c] = 0;

    for (int k0 = kb; k0 < ke; k0 += kTK) {
        for (int i = threadIdx.x; i < kTile * kTK; i += 256) {
            const int mm = i / kTK, kk = i - mm * kTK;
            const int k = k0 + kk;
            const int m = m0 + mm, n = n0 + mm;
            As[kk][mm] = (m < p.M && k < ke) ? load_a<MODE>(p, m, k) : 0;
            Bs[kk][mm] = (n < p.N && k < ke) ? load_b<MODE>(p, n, k) : 0;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < kTK; ++kk) {
            int32_t a[4], b[4];
#pragma unroll
            for (int r = 0; r < 4; ++r) a[r] = As[kk][ty + 16 * r];
#pragma unroll
            for (int c = 0; c < 4; ++c) b[c] = Bs[kk][tx + 16 * c];
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int c = 0; c < 4; ++c) acc[r][c] += (int64_t)a[r] * b[c];
        }
        __syncthreads();
    }
#pragma unroll
    for (int r = 0; r < 4; ++r)
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int m = m0 + ty + 16 * r, n = n0 + tx + 16 * c;
            if (m < p.M && n < p.N) {
                int64_t* o = p.out + (int64_t)m * p.N + n;
                if (gridDim.z > 1)
                    atomicAdd(reinterpret_cast<unsigned long long*>(o),
                              (unsigned long long)acc[r][c]);
                else
                    *o = acc[r][c];
            }
        }
}

// ---------------------------------------------------------------------------
// Forward epilogue: one thread per pooling window (or per element).
// ---------------------------------------------------------------------------
__global__ void k_fwd_epilogue(const int64_t* __restrict__ z, LayerGeom g, int B,
                               int alpha_inv, int mu, int64_t kdiv, int8_t* __restrict__ out,
                               int8_t* __restrict__ out2, int8_t* __restrict__ region,
                               int8_t* __restrict__ argmax, DropoutArgs drop) {
    pdl_wait();
    const int C = g.cout;
    if (!g.pool) {
        // dropout (linear layers): element i = b * out_features + j of this step's mask
        const uint32_t t = drop.p16 ? *drop.step : 0u;
        const int64_t n = (int64_t)B * g.h * g.w * C;
        for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
             i += (int64_t)gridDim.x * blockDim.x) {
            const int64_t zs = scale_floor(z[i], kdiv);
            int rg = relu_region(zs);
            int8_t v = (int8_t)relu_value(zs, alpha_inv, mu);
            if (drop.p16 && dropout_drop(drop.seed, t, drop.layer, (uint64_t)i, drop.p16)) {
                rg = kRegionDropped;
                v = 0;
            }
            region[i] = (int8_t)rg;
            out[i] = v;
            if (out2) out2[i] = v;
        }
        return;
    }
    // windows over ceil(h/2) x ceil(w/2); partial windows (odd edges) only
    // record region codes of the positions the floor-sized pool drops.
    const int wy_n = (g.h + 1) / 2, wx_n = (g.w + 1) / 2;
    const int64_t n = (int64_t)B * wy_n * wx_n * C;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % C);
        int64_t r = i / C;
        const int wx = (int)(r % wx_n);
        r /= wx_n;
        const int wy = (int)(r % wy_n);
        const int b = (int)(r / wy_n);
        int best = 0, bestv = 0;
        bool full = (2 * wy + 1 < g.h) && (2 * wx + 1 < g.w);
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int iy = 2 * wy + (k >> 1), ix = 2 * wx + (k & 1);
            if (iy >= g.h || ix >= g.w) continue;
            const int64_t pi = ((int64_t)(b * g.h + iy) * g.w + ix) * C + c;
            const int64_t zs = scale_floor(z[pi], kdiv);
            region[pi] = (int8_t)relu_region(zs);
            const int v = relu_value(zs, alpha_inv, mu);
            if (k == 0 || v > bestv) { bestv = v; best = k; }
        }
        if (full) {
            const int64_t oi = ((int64_t)(b * g.oh + wy) * g.ow + wx) * C + c;
            out[oi] = (int8_t)bestv;
            if (out2) out2[oi] = (int8_t)bestv;
            argmax[oi] = (int8_t)best;
        }
    }
}

// ---------------------------------------------------------------------------
// Learning layer forward + RSS loss, in one kernel.  A CTA (128-feature
// slice, 16 samples) adds its partial sums of z[b][g] = sum_j a[b][j] W_lr[g][j]
// into zsum with int64 atomics (exact, order independent).  The last CTA of
// a sample group (per-group ticket) turns that group's z into
// y_hat = floor(z / (256 d)) and grad_L = y_hat - 32 onehot and adds its part
// of the SSE; the last of those (final ticket) writes the loss.
// Tickets live behind zsum: zsum[B G + y] per group, zsum[B G + groups].
// Splitting this into a partial-sum kernel and a separate finish kernel
// (per-slice partials with plain stores, or the atomic partials with a
// one-read-per-output finish) was measured no faster: the second launch costs
// what the fence and tickets save.
// ---------------------------------------------------------------------------
constexpr int kLrSamples = 16;   // samples per CTA
constexpr int kLpSlice = 128;    // features per CTA
static_assert(kLpSlice == 16 * 8, "k_learn_partial: 16 lanes of 8 features per sample");

__global__ void __launch_bounds__(256) k_learn_partial(const int8_t* __restrict__ a,
                                                       const int32_t* __restrict__ wlr, int B,
                                                       int d, int G, int vec8,
                                                       unsigned long long* __restrict__ zsum,
                                                       FloorDiv dv, const int32_t* __restrict__ labels,
                                                       int32_t* __restrict__ grad_l,
                                                       unsigned long long* sse, int64_t* loss,
                                                       uint32_t* maxabs_gl, uint32_t* status) {
    pdl_wait();
    // thread (u, k): sample u of the group, features 8k .. 8k + 7 of the slice,
    // read as one 8-byte word when the rows allow it (vec8: d % 8 == 0 and an
    // 8-byte aligned a).  The slice of W_lr is staged in shared memory with
    // feature 8k + m at column 16m + k, so the lanes of a sample read
    // consecutive words; classes in chunks of kLpG.
    constexpr int kLpG = 16;
    __shared__ int32_t ws[kLpG][kLpSlice + 1];
    const int u = threadIdx.x >> 4, k = threadIdx.x & 15;
    const int b = blockIdx.y * kLrSamples + u;
    const int j0 = blockIdx.x * kLpSlice;
    const int jb = j0 + 8 * k;
    int av[8];
    if (vec8 && b < B && jb + 8 <= d) {
        const uint2 w = *reinterpret_cast<const uint2*>(a + (int64_t)b * d + jb);
#pragma unroll
        for (int m = 0; m < 4; ++m) {
            av[m] = (int8_t)(w.x >> (8 * m));
            av[4 + m] = (int8_t)(w.y >> (8 * m));
        }
    } else {
#pragma unroll
        for (int m = 0; m < 8; ++m) {
            const int j = jb + m;
            av[m] = (b < B && j < d) ? a[(int64_t)b * d + j] : 0;
        }
    }
    for (int gc = 0; gc < G; gc += kLpG) {
        const int ng = min(kLpG, G - gc);
        if (gc) __syncthreads();
        for (int i = threadIdx.x; i < ng * kLpSlice; i += blockDim.x) {
            const int g = i / kLpSlice, j = i - g * kLpSlice;
            ws[g][(j & 7) * 16 + (j >> 3)] = j0 + j < d ? wlr[(int64_t)(gc + g) * d + j0 + j] : 0;
        }
        __syncthreads();
        for (int g = 0; g < ng; ++g) {
            long long t = 0;
#pragma unroll
            for (int m = 0; m < 8; ++m) t += (long long)ws[g][16 * m + k] * av[m];
#pragma unroll
            for (int off = 8; off; off >>= 1) t += __shfl_xor_sync(kFull, t, off);
            if (k == 0 && b < B && t != 0)
                atomicAdd(&zsum[(int64_t)b * G + gc + g], (unsigned long long)t);
        }
    }
    __shared__ int last;
    __shared__ unsigned long long red_s[8];
    __shared__ uint32_t red_m[8];
    __shared__ int flags;
    unsigned long long* tickets = zsum + (int64_t)B * G;
    if (k == 0) __threadfence();     // the lanes that added into zsum
    __syncthreads();
    if (threadIdx.x == 0) {
        flags = 0;
        last = atomicAdd(&tickets[blockIdx.y], 1ull) == (unsigned long long)gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    // this sample group's z is complete: y_hat, grad_L, its share of the SSE
    unsigned long long ss = 0;
    uint32_t mx = 0;
    int fl = 0;
    const int nb = min(kLrSamples, B - (int)blockIdx.y * kLrSamples);
    for (int i = threadIdx.x; i < nb * G; i += blockDim.x) {
        const int bb = blockIdx.y * kLrSamples + i / G, g = i % G;
        const int lab = labels[bb];
        const bool bad = lab < 0 || lab >= G;
        if (bad && g == 0) fl |= ST_BAD_LABEL;
        // NITRO-Scaling, SF = 2^8 d: floor(floor(z / 256) / d)
        const int64_t yhat = dv.floor_div((int64_t)__ldcg(zsum + (int64_t)bb * G + g) >> 8);
        const int64_t v = yhat - ((!bad && g == lab) ? 32 : 0);
        if (!fits_i32(v)) fl |= ST_OVERFLOW;
        const int32_t sv = (int32_t)v;
        grad_l[(int64_t)bb * G + g] = sv;
        ss += (unsigned long long)((int64_t)sv * sv);
        mx = max(mx, abs_u32(sv));
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) {
        ss += __shfl_xor_sync(kFull, ss, off);
        mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    }
    if (fl) atomicOr(&flags, fl);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) { red_s[warp] = ss; red_m[warp] = mx; }
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long t = 0;
        uint32_t m = 0;
        for (int w = 0; w < 8; ++w) { t += red_s[w]; m = max(m, red_m[w]); }
        atomicAdd(sse, t);                                   // modulo 2^64
        if (m) atomicMax(maxabs_gl, m);
        if (flags) atomicOr(status, (uint32_t)flags);
        __threadfence();
        if (atomicAdd(&tickets[gridDim.y], 1ull) == (unsigned long long)gridDim.y - 1) {
            __threadfence();
            const unsigned long long tot = atomicAdd(sse, 0ull);
            if (loss) *loss = fdiv64((int64_t)tot, 2);
        }
    }
}

// dW_lr[g][j] = sum_b grad_l[b][g] * a[b][j]
__global__ void k_learn_dw(const int8_t* __restrict__ a, const int32_t* __restrict__ grad_l,
                           int B, int d, int G, int64_t* __restrict__ dwlr) {
    pdl_wait();
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const int g = blockIdx.y;
    if (j >= d) return;
    int64_t s = 0;
#pragma unroll 8
    for (int b = 0; b < B; ++b) s += (int64_t)grad_l[(int64_t)b * G + g] * a[(int64_t)b * d + j];
    dwlr[(int64_t)g * d + j] = s;
}

// ---------------------------------------------------------------------------
// Gradient at a layer output -> delta at its pre-activation.
// ---------------------------------------------------------------------------
__global__ void k_grad_to_delta(DeltaSrc src, LayerGeom g, int B, int alpha_inv,
                                const int8_t* __restrict__ region,
                                const int8_t* __restrict__ argmax, int32_t* __restrict__ delta,
                                uint32_t* maxabs_delta, uint32_t* status) {
    pdl_wait();
    const int64_t out_f = (int64_t)g.oh * g.ow * g.cout;
    const int64_t n = (int64_t)B * out_f;
    if (blockIdx.x == 0 && threadIdx.x == 0 &&
        int64_bound_exceeded(*src.maxabs_a, *src.maxabs_b, src.bound_k))
        atomicOr(status, ST_OVERFLOW);
    uint32_t mx = 0;
    bool ovf = false;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t b = i / out_f, q = i - b * out_f;
        int64_t gv;
        if (src.wlr) {
            uint64_t acc = 0;  // modulo 2^64, exact below the bound
#pragma unroll 16
            for (int k = 0; k < src.G; ++k)
                acc += (uint64_t)(int64_t)src.grad_l[b * src.G + k] *
                       (uint64_t)(int64_t)src.wlr[(int64_t)k * out_f + q];
            gv = (int64_t)acc;
        } else {
            gv = src.g64[i];
        }
        ovf |= !fits_i32(gv);
        const int32_t gs = (int32_t)gv;
        if (g.pool) {
            const int c = (int)(q % g.cout);
            const int64_t r = q / g.cout;
            const int ox = (int)(r % g.ow), oy = (int)(r / g.ow);
            const int am = argmax[i];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const int iy = 2 * oy + (k >> 1), ix = 2 * ox + (k & 1);
                const int64_t pi = ((b * g.h + iy) * g.w + ix) * g.cout + c;
                const int32_t dv = (k == am) ? relu_backward(gs, region[pi], alpha_inv) : 0;
                delta[pi] = dv;
                mx = max(mx, abs_u32(dv));
            }
        } else {
            const int32_t dv = relu_backward(gs, region[i], alpha_inv);
            delta[i] = dv;
            mx = max(mx, abs_u32(dv));
        }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    ovf = __any_sync(kFull, ovf);
    if ((threadIdx.x & 31) == 0) {
        if (mx) atomicMax(maxabs_delta, mx);
        if (ovf) atomicOr(status, ST_OVERFLOW);
    }
}

// ---------------------------------------------------------------------------
// Learning-layer max-pool (Sec. 3.3, z^mp; window from d^lr, App. B): one
// thread per pooled element, channel fastest, so a warp reads 32 consecutive
// channels of each window row.  First maximum in row-major window order.
// ---------------------------------------------------------------------------
__global__ void k_lr_pool_fwd(const int8_t* __restrict__ a, int B, int H, int W, int C, int kh,
                              int kw, int ph, int pw, int8_t* __restrict__ out,
                              uint8_t* __restrict__ am) {
    pdl_wait();
    const int64_t n = (int64_t)B * ph * pw * C;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % C);
        int64_t r = i / C;
        const int x = (int)(r % pw);
        r /= pw;
        const int y = (int)(r % ph);
        const int64_t b = r / ph;
        const int8_t* p = a + ((b * H + (int64_t)y * kh) * W + (int64_t)x * kw) * C + c;
        int best = 0, bestv = p[0];
        for (int u = 0; u < kh; ++u)
            for (int v = 0; v < kw; ++v) {
                const int val = p[((int64_t)u * W + v) * C];
                if (val > bestv) { bestv = val; best = u * kw + v; }
            }
        out[i] = (int8_t)bestv;
        am[i] = (uint8_t)best;
    }
}

// Same, four channels per thread (C % 4 == 0, 4-byte aligned buffers): signed
// SIMD byte maxima, and a window position replaced only where a later value
// is strictly greater (the first maximum wins).
__global__ void k_lr_pool_fwd4(const int8_t* __restrict__ a, int B, int H, int W, int C, int kh,
                               int kw, int ph, int pw, FloorDiv32 dv_c4, FloorDiv32 dv_pw,
                               FloorDiv32 dv_ph, int8_t* __restrict__ out,
                               uint8_t* __restrict__ am) {
    pdl_wait();
    const int C4 = C >> 2;
    const uint32_t n4 = (uint32_t)B * ph * pw * C4;
    for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += gridDim.x * blockDim.x) {
        const uint32_t pix = dv_c4.udiv(i);
        const int c = (int)(i - pix * C4) * 4;
        const uint32_t r = dv_pw.udiv(pix);
        const int x = (int)(pix - r * pw);
        const uint32_t b = dv_ph.udiv(r);
        const int y = (int)(r - b * ph);
        const int8_t* p = a + ((b * H + (uint32_t)(y * kh)) * W + (uint32_t)(x * kw)) * C + c;
        uint32_t best = *reinterpret_cast<const uint32_t*>(p), pos = 0;
        for (int u = 0; u < kh; ++u)
            for (int v = 0; v < kw; ++v) {
                const uint32_t val = *reinterpret_cast<const uint32_t*>(p + (u * W + v) * C);
                const uint32_t gt = __vcmpgts4(val, best);
                best = __vmaxs4(best, val);
                pos = (pos & ~gt) | ((uint32_t)(u * kw + v) * 0x01010101u & gt);
            }
        reinterpret_cast<uint32_t*>(out)[i] = best;
        reinterpret_cast<uint32_t*>(am)[i] = pos;
    }
}

// ---------------------------------------------------------------------------
// Learning-layer backward through the pool, into the last layer's delta.  One
// thread per pre-pool element (b, y, x, c) of that conv layer: it receives a
// gradient only if it won its 2x2 window (when the layer pools) and the
// pooled position won its learning-pool window; that thread alone forms
// delta_fw = sum_g grad_L[b][g] W_lr[g][f] of the learning feature f (modulo
// 2^64, int32 storage rule) and applies NITRO-ReLU backward.  Every element is
// written, so no clearing pass is needed.
// ---------------------------------------------------------------------------
__global__ void k_lrpool_to_delta(const int32_t* __restrict__ gl, const int32_t* __restrict__ wlr,
                                  int G, int d, LayerGeom g, LrPoolGeom lp, int B,
                                  const uint8_t* __restrict__ lam,
                                  const int8_t* __restrict__ argmax,
                                  const int8_t* __restrict__ region, FloorDiv32 alpha,
                                  int32_t* __restrict__ delta, const uint32_t* maxabs_gl,
                                  const uint32_t* maxabs_wlr, uint32_t* maxabs_delta,
                                  uint32_t* status) {
    pdl_wait();
    const int C = g.cout;
    const int64_t n = (int64_t)B * g.h * g.w * C;
    if (blockIdx.x == 0 && threadIdx.x == 0 && int64_bound_exceeded(*maxabs_gl, *maxabs_wlr, G))
        atomicOr(status, ST_OVERFLOW);
    uint32_t mx = 0;
    bool ovf = false;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % C);
        int64_t r = i / C;
        const int x = (int)(r % g.w);
        r /= g.w;
        const int y = (int)(r % g.h);
        const int64_t b = r / g.h;
        int qy = y, qx = x;
        bool hit = true;
        if (g.pool) {
            qy = y >> 1;
            qx = x >> 1;
            hit = qy < g.oh && qx < g.ow &&
                  argmax[((b * g.oh + qy) * g.ow + qx) * C + c] == (((y & 1) << 1) | (x & 1));
        }
        int32_t dv = 0;
        if (hit) {
            const int wy = qy / lp.kh, wx = qx / lp.kw;
            hit = wy < lp.ph && wx < lp.pw &&
                  lam[((b * lp.ph + wy) * lp.pw + wx) * C + c] ==
                      (qy - wy * lp.kh) * lp.kw + (qx - wx * lp.kw);
            if (hit) {
                const int64_t f = ((int64_t)wy * lp.pw + wx) * C + c;
                uint64_t acc = 0;   // modulo 2^64, exact below the bound
                for (int k = 0; k < G; ++k)
                    acc += (uint64_t)((int64_t)gl[b * G + k] * wlr[(int64_t)k * d + f]);
                const int64_t gv = (int64_t)acc;
                ovf |= !fits_i32(gv);
                const int32_t gs = (int32_t)gv;
                const int rg = region[i];
                dv = rg == 1 ? alpha.floor_div(gs) : (rg == 2 ? gs : 0);
            }
        }
        delta[i] = dv;
        mx = max(mx, abs_u32(dv));
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    ovf = __any_sync(kFull, ovf);
    if ((threadIdx.x & 31) == 0) {
        if (mx) atomicMax(maxabs_delta, mx);
        if (ovf) atomicOr(status, ST_OVERFLOW);
    }
}

// Same, four channels per thread (C % 4 == 0): one 4-byte load of each code
// array and of the region bytes, one 16-byte delta store, 32-bit index
// arithmetic (B h w C < 2^31) through invariant dividers; the pool windows
// are powers of two, so their divisions are shifts.
__global__ void k_lrpool_to_delta4(const int32_t* __restrict__ gl, const int32_t* __restrict__ wlr,
                                   int G, int d, LayerGeom g, LrPoolGeom lp, int lg_kh, int lg_kw,
                                   int B, FloorDiv32 dv_c4, FloorDiv32 dv_w, FloorDiv32 dv_h,
                                   const uint8_t* __restrict__ lam,
                                   const int8_t* __restrict__ argmax,
                                   const int8_t* __restrict__ region, FloorDiv32 alpha,
                                   int32_t* __restrict__ delta, const uint32_t* maxabs_gl,
                                   const uint32_t* maxabs_wlr, uint32_t* maxabs_delta,
                                   uint32_t* status) {
    pdl_wait();
    const int C = g.cout, C4 = g.cout >> 2;
    const uint32_t n4 = (uint32_t)B * g.h * g.w * C4;
    if (blockIdx.x == 0 && threadIdx.x == 0 && int64_bound_exceeded(*maxabs_gl, *maxabs_wlr, G))
        atomicOr(status, ST_OVERFLOW);
    uint32_t mx = 0;
    bool ovf = false;
    for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += gridDim.x * blockDim.x) {
        const uint32_t pix = dv_c4.udiv(i);
        const int c = (int)(i - pix * C4) * 4;
        const uint32_t r = dv_w.udiv(pix);
        const int x = (int)(pix - r * g.w);
        const uint32_t b = dv_h.udiv(r);
        const int y = (int)(r - b * g.h);
        int qy = y, qx = x;
        bool any = true;
        uint32_t am2 = 0, code2 = 0;
        if (g.pool) {
            qy = y >> 1;
            qx = x >> 1;
            any = qy < g.oh && qx < g.ow;
            if (any) {
                am2 = *reinterpret_cast<const uint32_t*>(argmax + ((b * g.oh + qy) * g.ow + qx) * C + c);
                code2 = (uint32_t)(((y & 1) << 1) | (x & 1));
            }
        }
        int v[4] = {0, 0, 0, 0};
        const int wy = qy >> lg_kh, wx = qx >> lg_kw;
        if (any && wy < lp.ph && wx < lp.pw) {
            const uint32_t lw =
                *reinterpret_cast<const uint32_t*>(lam + ((b * lp.ph + wy) * lp.pw + wx) * C + c);
            const uint32_t code = (uint32_t)(((qy - (wy << lg_kh)) << lg_kw) + (qx - (wx << lg_kw)));
            const uint32_t rw = *reinterpret_cast<const uint32_t*>(region + 4 * (size_t)i);
            const int f0 = (wy * lp.pw + wx) * C + c;
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const bool hit = (!g.pool || ((am2 >> (8 * j)) & 255u) == code2) &&
                                 ((lw >> (8 * j)) & 255u) == code;
                if (!hit) continue;
                uint64_t acc = 0;   // modulo 2^64, exact below the bound
                for (int k = 0; k < G; ++k)
                    acc += (uint64_t)((int64_t)gl[b * G + k] * wlr[(int64_t)k * d + f0 + j]);
                const int64_t gv = (int64_t)acc;
                ovf |= !fits_i32(gv);
                const int32_t gs = (int32_t)gv;
                const int rg = (int8_t)(rw >> (8 * j));
                v[j] = rg == 1 ? alpha.floor_div(gs) : (rg == 2 ? gs : 0);
                mx = max(mx, abs_u32(v[j]));
            }
        }
        reinterpret_cast<int4*>(delta)[i] = make_int4(v[0], v[1], v[2], v[3]);
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    ovf = __any_sync(kFull, ovf);
    if ((threadIdx.x & 31) == 0) {
        if (mx) atomicMax(maxabs_delta, mx);
        if (ovf) atomicOr(status, ST_OVERFLOW);
    }
}

// ---------------------------------------------------------------------------
// IntegerSGD (Algorithm 1); blockIdx.y selects the tensor.
// ---------------------------------------------------------------------------
__device__ __forceinline__ int32_t sgd_one(const SgdTensor& t, int round_trunc, int32_t w32,
                                           int64_t g, uint32_t& mx, bool& ovf) {
    const int64_t w = w32;
    int64_t d = round_trunc ? t.gdiv.trunc_div(g) : t.gdiv.floor_div(g);
    if (t.eta_inv != 0) d += round_trunc ? t.ediv.trunc_div(w) : t.ediv.floor_div(w);
    const int64_t nw = w - d;
    ovf |= !fits_i32(nw);
    const int32_t s = (int32_t)nw;
    mx = max(mx, abs_u32(s));
    return s;
}

// The updated weight w (element i of [Cout][9][cin]) into its four bf16 limb
// planes: limbs 0..2 the digits ((x + 128) & 255) - 128 of successive base-256
// remainders, limb 3 the rest; each limb is an integer of at most 8 bits, so
// the top half of its fp32 bits is its exact bf16.
__device__ __forceinline__ void sgd_planes(const SgdTensor& t, int64_t i, int32_t w) {
    const uint32_t q = t.cin_div.udiv((uint32_t)i);
    const int ci = (int)(i - (int64_t)q * t.cin);
    const int tap = (int)(q % 9u), co = (int)(q / 9u);
    uint16_t* p = t.planes + (int64_t)co * t.row_k + tap * t.tap_k + ci;
    int64_t x = w;
#pragma unroll
    for (int l = 0; l < 4; ++l) {
        int v;
        if (l < 3) {
            v = (int)(((x + 128) & 255) - 128);
            x = (x - v) >> 8;
        } else {
            v = (int)x;
        }
        p[l * t.plane] = (uint16_t)(__float_as_uint((float)v) >> 16);
    }
}

// Four consecutive updated weights into their limb planes when the planes are
// laid out like W (linear layers; convs with Cin a multiple of 64): the same
// split, one 8-byte store per plane at p + l * plane.
__device__ __forceinline__ void sgd_planes4(uint16_t* p, int64_t plane, int4 w) {
    int32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int l = 0; l < 4; ++l) {
        uint32_t h[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            int dg;
            if (l < 3) {
                // v = 256 q + r: digit r or r - 256, remainder q or q + 1
                const int r = v[k] & 255;
                dg = r - ((r >> 7) << 8);
                v[k] = (v[k] >> 8) + (r >> 7);
            } else {
                dg = v[k];
            }
            h[k] = __float_as_uint((float)dg) >> 16;
        }
        *reinterpret_cast<uint2*>(p + l * plane) = make_uint2(h[0] | (h[1] << 16), h[2] | (h[3] << 16));
    }
}

// Four consecutive weights per thread (16-byte loads of W, two of dW; the
// tensors are this library's own 256-byte aligned buffers), the tail singly.
__global__ void k_integersgd(SgdBatch bt) {
    pdl_wait();
    const SgdTensor t = bt.t[blockIdx.y];
    uint32_t mx = 0;
    bool ovf = false;
    const int64_t n4 = t.n / 4;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int4 w = reinterpret_cast<const int4*>(t.w)[i];
        const longlong2 g0 = reinterpret_cast<const longlong2*>(t.dw)[2 * i];
        const longlong2 g1 = reinterpret_cast<const longlong2*>(t.dw)[2 * i + 1];
        int4 o;
        o.x = sgd_one(t, bt.round_trunc, w.x, g0.x, mx, ovf);
        o.y = sgd_one(t, bt.round_trunc, w.y, g0.y, mx, ovf);
        o.z = sgd_one(t, bt.round_trunc, w.z, g1.x, mx, ovf);
        o.w = sgd_one(t, bt.round_trunc, w.w, g1.y, mx, ovf);
        reinterpret_cast<int4*>(t.w)[i] = o;
        if (t.planes && t.contig) {
            sgd_planes4(t.planes + 4 * i, t.plane, o);
        } else if (t.planes) {
            sgd_planes(t, 4 * i, o.x);
            sgd_planes(t, 4 * i + 1, o.y);
            sgd_planes(t, 4 * i + 2, o.z);
            sgd_planes(t, 4 * i + 3, o.w);
        }
    }
    for (int64_t i = 4 * n4 + blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < t.n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t nw = sgd_one(t, bt.round_trunc, t.w[i], t.dw[i], mx, ovf);
        t.w[i] = nw;
        if (t.planes) sgd_planes(t, i, nw);
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    ovf = __any_sync(kFull, ovf);
    if ((threadIdx.x & 31) == 0) {
        if (mx) atomicMax(t.maxabs_w, mx);
        if (ovf) atomicOr(bt.status, ST_OVERFLOW);
    }
    // one block step taken: advance the dropout step counter
    if (bt.step && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) *bt.step += 1u;
}

// ---------------------------------------------------------------------------
// Narrow-input 3x3 conv (Cin <= 8, e.g. image channels): forward with the
// NITRO-Scaling / NITRO-ReLU / max-pool epilogue fused, one thread per
// (pooling window or pixel, 16 output channels).  The weights sit in shared
// memory; sums are exact int64.
// ---------------------------------------------------------------------------
constexpr int kSmallCin = 8;
constexpr int kSmallCo = 16;

struct SmallFwdArgs {
    const int8_t* x;       // [B][H][W][Cin]
    const int32_t* w;      // [Cout][3][3][Cin]
    int B, H, W, Cin, Cout, pool, oh, ow;
    FloorDiv32 sf32;       // divide by 9 * Cin (after >> 8)
    int64_t z_hi, z_lo;    // saturation thresholds 128 SF and -127 SF
    FloorDiv alpha;
    int mu;
    int8_t* act;           // [B][oh][ow][Cout]
    int8_t* out2;
    int8_t* region;        // [B][H][W][Cout]
    int8_t* argmax;
    uint16_t* next_nhwc;   // bf16 copy of act, or null
};

__global__ void __launch_bounds__(256) k_conv_small_fwd(const SmallFwdArgs a) {
    pdl_wait();
    extern __shared__ int32_t wsm[];                 // Cout * 9 * Cin
    __shared__ int8_t relu_tab[256];
    const int nw = a.Cout * 9 * a.Cin;
    for (int i = threadIdx.x; i < nw; i += blockDim.x) wsm[i] = a.w[i];
    if (threadIdx.x < 255) relu_tab[threadIdx.x] = (int8_t)relu_value((int64_t)threadIdx.x - 127, a.alpha, a.mu);
    __syncthreads();
    const int step = a.pool ? 2 : 1;
    const int wy_n = (a.H + step - 1) / step, wx_n = (a.W + step - 1) / step;
    const int ngrp = a.Cout / kSmallCo;
    const int64_t total = (int64_t)a.B * wy_n * wx_n * ngrp;
    for (int64_t idx = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; idx < total;
         idx += (int64_t)gridDim.x * blockDim.x) {
        const int grp = (int)(idx % ngrp);
        int64_t r = idx / ngrp;
        const int wx = (int)(r % wx_n);
        r /= wx_n;
        const int wy = (int)(r % wy_n);
        const int b = (int)(r / wy_n);
        const int co0 = grp * kSmallCo;
        int8_t vals[4][kSmallCo];
        bool valid[4];
        for (int k = 0; k < step * step; ++k) {
            const int y = wy * step + (k >> 1), x = wx * step + (k & 1);
            valid[k] = y < a.H && x < a.W;
            if (!valid[k]) continue;
            // 3x3 x Cin input patch, zero outside the image
            int32_t patch[9 * kSmallCin];
            for (int t = 0; t < 9; ++t) {
                const int iy = y + t / 3 - 1, ix = x + t % 3 - 1;
                const bool in = iy >= 0 && iy < a.H && ix >= 0 && ix < a.W;
                const int8_t* src = a.x + (((int64_t)b * a.H + iy) * a.W + ix) * a.Cin;
                for (int c = 0; c < a.Cin; ++c) patch[t * a.Cin + c] = in ? (int32_t)src[c] : 0;
            }
            const int K = 9 * a.Cin;
            uint32_t rg[kSmallCo / 4] = {0, 0, 0, 0};
            for (int j = 0; j < kSmallCo; ++j) {
                const int32_t* wr = wsm + (co0 + j) * K;
                int64_t z = 0;
                for (int q = 0; q < K; ++q) z += (int64_t)wr[q] * patch[q];
                int reg, val;
                if (z >= a.z_hi) { reg = 3; val = relu_tab[254]; }
                else if (z < a.z_lo) { reg = 0; val = relu_tab[0]; }
                else {
                    const int zq = a.sf32.floor_div((int32_t)(z >> 8));
                    reg = zq < 0 ? 1 : 2;
                    val = relu_tab[zq + 127];
                }
                vals[k][j] = (int8_t)val;
                rg[j >> 2] |= (uint32_t)reg << (8 * (j & 3));
            }
            const int64_t pix = ((int64_t)b * a.H + y) * a.W + x;
            *reinterpret_cast<uint4*>(a.region + pix * a.Cout + co0) = make_uint4(rg[0], rg[1], rg[2], rg[3]);
        }
        int64_t o;
        int8_t outv[kSmallCo];
        uint32_t am[kSmallCo / 4] = {0, 0, 0, 0};
        if (a.pool) {
            if (!(valid[0] && valid[1] && valid[2] && valid[3])) continue;   // floor-sized pool
            for (int j = 0; j < kSmallCo; ++j) {
                int best = vals[0][j], kb = 0;                 // first maximum wins
                for (int k = 1; k < 4; ++k)
                    if (vals[k][j] > best) { best = vals[k][j]; kb = k; }
                outv[j] = (int8_t)best;
                am[j >> 2] |= (uint32_t)kb << (8 * (j & 3));
            }
            o = (((int64_t)b * a.oh + wy) * a.ow + wx) * a.Cout + co0;
            *reinterpret_cast<uint4*>(a.argmax + o) = make_uint4(am[0], am[1], am[2], am[3]);
        } else {
            for (int j = 0; j < kSmallCo; ++j) outv[j] = vals[0][j];
            o = (((int64_t)b * a.H + wy) * a.W + wx) * a.Cout + co0;
        }
        uint32_t pk[4];
        for (int q = 0; q < 4; ++q)
            pk[q] = (uint32_t)(uint8_t)outv[4 * q] | ((uint32_t)(uint8_t)outv[4 * q + 1] << 8) |
                    ((uint32_t)(uint8_t)outv[4 * q + 2] << 16) | ((uint32_t)(uint8_t)outv[4 * q + 3] << 24);
        *reinterpret_cast<uint4*>(a.act + o) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        if (a.out2) *reinterpret_cast<uint4*>(a.out2 + o) = make_uint4(pk[0], pk[1], pk[2], pk[3]);
        if (a.next_nhwc) {
            uint32_t bw[8];
            for (int q = 0; q < 8; ++q)
                bw[q] = (uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn((float)outv[2 * q])) |
                        ((uint32_t)__bfloat16_as_ushort(__float2bfloat16_rn((float)outv[2 * q + 1])) << 16);
            reinterpret_cast<uint4*>(a.next_nhwc + o)[0] = make_uint4(bw[0], bw[1], bw[2], bw[3]);
            reinterpret_cast<uint4*>(a.next_nhwc + o)[1] = make_uint4(bw[4], bw[5], bw[6], bw[7]);
        }
    }
}

// Narrow-input weight gradient: CTA = a chunk of kWgRows image rows of one
// image; delta rows and the input rows with their halo are staged in shared
// memory; each thread owns a few (co, tap, ci) entries, sums them over the
// chunk in int64 and adds them into dW with 64-bit atomics.
constexpr int kWgRows = 8;

__global__ void __launch_bounds__(256) k_conv_small_wgrad(const int8_t* __restrict__ x,
                                                          const int32_t* __restrict__ d, int B,
                                                          int H, int W, int Cin, int Cout,
                                                          unsigned long long* __restrict__ dw) {
    pdl_wait();
    extern __shared__ int32_t sm[];
    const int rows = min(kWgRows, H - blockIdx.x * kWgRows);
    const int y0 = blockIdx.x * kWgRows, b = blockIdx.y;
    int32_t* dsm = sm;                                   // [rows][W][Cout]
    int8_t* xsm = reinterpret_cast<int8_t*>(sm + kWgRows * W * Cout);   // [rows+2][W+2][Cin]
    const int nd = rows * W * Cout;
    for (int i = threadIdx.x; i < nd; i += blockDim.x)
        dsm[i] = d[((int64_t)b * H + y0) * W * Cout + i];
    const int hx = (rows + 2) * (W + 2) * Cin;
    for (int i = threadIdx.x; i < hx; i += blockDim.x) {
        const int c = i % Cin, rest = i / Cin, xx = rest % (W + 2), yy = rest / (W + 2);
        const int iy = y0 + yy - 1, ix = xx - 1;
        xsm[i] = (iy >= 0 && iy < H && ix >= 0 && ix < W) ? x[(((int64_t)b * H + iy) * W + ix) * Cin + c] : 0;
    }
    __syncthreads();
    const int nout = Cout * 9 * Cin;
    for (int e = threadIdx.x; e < nout; e += blockDim.x) {
        const int ci = e % Cin, t = (e / Cin) % 9, co = e / (9 * Cin);
        const int ky = t / 3, kx = t % 3;
        int64_t acc = 0;
        for (int yy = 0; yy < rows; ++yy) {
            const int32_t* drow = dsm + (yy * W) * Cout + co;
            const int8_t* xrow = xsm + ((yy + ky) * (W + 2) + kx) * Cin + ci;
            for (int xx = 0; xx < W; ++xx) acc += (int64_t)drow[xx * Cout] * xrow[xx * Cin];
        }
        atomicAdd(&dw[e], (unsigned long long)acc);
    }
}

// ---------------------------------------------------------------------------
// Learning-layer backward, fused, for G <= 16.  CTA: 64 features q of the
// block output x 16 samples; grad_L and the 16 x 64 slice of a are staged in
// shared memory.  dW_lr[g][q] partials over the 16 samples are dot products
// out of shared memory, added to a zeroed dW_lr with 64-bit atomics.  With a
// forward layer below (has_delta): thread (q, lane) forms delta_fw[b][q] =
// sum_g grad_L[b][g] W_lr[g][q] (int32 storage rule) for samples lane,
// lane + 4, ... and routes it through max-pool backward and NITRO-ReLU
// backward into that layer's delta; the region bytes of its four samples are
// loaded before any is used.
// ---------------------------------------------------------------------------
constexpr int kLbQ = 64;                         // features per CTA
constexpr int kLbLanes = 4;                      // sample lanes per feature
constexpr int kLbPer = 4;                        // samples per lane
constexpr int kLbSamples = kLbLanes * kLbPer;    // samples per CTA
constexpr int kLbMaxG = 16;

template <int GM>   // classes held in registers: G <= GM
__global__ void __launch_bounds__(256) k_lr_backward(const int8_t* __restrict__ a,
                                                     const int32_t* __restrict__ gl,
                                                     const int32_t* __restrict__ wlr, int B, int G,
                                                     int d, int has_delta, LayerGeom lg,
                                                     FloorDiv32 alpha,
                                                     const int8_t* __restrict__ region,
                                                     const int8_t* __restrict__ argmax,
                                                     int32_t* __restrict__ delta,
                                                     unsigned long long* __restrict__ dwlr,
                                                     const uint32_t* maxabs_gl,
                                                     const uint32_t* maxabs_wlr,
                                                     uint32_t* maxabs_delta, uint32_t* status) {
    pdl_wait();
    __shared__ int32_t gls[kLbSamples][GM];
    __shared__ int8_t as[kLbSamples][kLbQ];
    const int ql = threadIdx.x % kLbQ, sl = threadIdx.x / kLbQ;
    const int q0 = blockIdx.x * kLbQ, q = q0 + ql;
    const int b0 = blockIdx.y * kLbSamples;
    const int nb = min(kLbSamples, B - b0);
    for (int i = threadIdx.x; i < kLbSamples * GM; i += blockDim.x) {
        const int u = i / GM, g = i % GM;
        gls[u][g] = (u < nb && g < G) ? gl[(int64_t)(b0 + u) * G + g] : 0;
    }
#pragma unroll
    for (int i = 0; i < kLbPer; ++i) {
        const int u = sl + kLbLanes * i;
        as[u][ql] = (u < nb && q < d) ? a[(int64_t)(b0 + u) * d + q] : (int8_t)0;
    }
    if (has_delta && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0 &&
        int64_bound_exceeded(*maxabs_gl, *maxabs_wlr, G))
        atomicOr(status, ST_OVERFLOW);
    // loads of the delta path (W_lr column, argmax, region bytes) go out with
    // the staging loads, before the barrier
    const bool act = has_delta && q < d;
    int32_t w[GM];
    int rgv[kLbPer], am[kLbPer];
    int64_t img = 0, p00 = 0, dx = 0, dy = 0;
#pragma unroll
    for (int g = 0; g < GM; ++g) w[g] = (act && g < G) ? wlr[(int64_t)g * d + q] : 0;
    if (act) {
        // position of feature q in the (pooled) output grid
        const int c = q % lg.cout;
        const int r = q / lg.cout;
        const int ox = r % lg.ow, oy = r / lg.ow;
        // element offsets of the (up to) four pre-pool positions within one image
        img = lg.pool ? (int64_t)lg.h * lg.w * lg.cout : (int64_t)d;
        p00 = lg.pool ? ((int64_t)(2 * oy) * lg.w + 2 * ox) * lg.cout + c : q;
        dx = lg.cout;
        dy = (int64_t)lg.w * lg.cout;
    }
#pragma unroll
    for (int i = 0; i < kLbPer; ++i) {
        const int u = sl + kLbLanes * i;
        rgv[i] = 0;
        am[i] = 0;
        if (act && u < nb) {
            const int64_t base = (b0 + u) * img + p00;
            if (lg.pool) {
                // only the recorded window position receives the gradient
                am[i] = argmax[(int64_t)(b0 + u) * d + q];
                const int r0 = region[base], r1 = region[base + dx];
                const int r2 = region[base + dy], r3 = region[base + dy + dx];
                rgv[i] = am[i] == 0 ? r0 : (am[i] == 1 ? r1 : (am[i] == 2 ? r2 : r3));
            } else {
                rgv[i] = region[base];
            }
        }
    }
    __syncthreads();
    // dW_lr partials: (g, q) pairs over the CTA's samples
    for (int i = threadIdx.x; i < G * kLbQ; i += blockDim.x) {
        const int g = i / kLbQ, qq = i - g * kLbQ;
        if (q0 + qq >= d) continue;
        long long t = 0;
#pragma unroll
        for (int u = 0; u < kLbSamples; ++u) t += (long long)gls[u][g] * as[u][qq];
        if (t != 0) atomicAdd(&dwlr[(int64_t)g * d + q0 + qq], (unsigned long long)t);
    }
    if (!has_delta) return;
    uint32_t mx = 0;
    bool ovf = false;
    if (q < d) {
#pragma unroll
        for (int i = 0; i < kLbPer; ++i) {
            const int u = sl + kLbLanes * i;
            if (u >= nb) break;
            uint64_t acc = 0;     // modulo 2^64, exact below the bound
#pragma unroll
            for (int g = 0; g < GM; ++g) acc += (uint64_t)((int64_t)gls[u][g] * w[g]);
            const int64_t gv = (int64_t)acc;
            ovf |= !fits_i32(gv);
            const int32_t gs = (int32_t)gv;
            // NITRO-ReLU backward: piece 1 -> floor(g / alpha_inv), piece 2 -> g, else 0
            const int32_t dvv = rgv[i] == 1 ? alpha.floor_div(gs) : (rgv[i] == 2 ? gs : 0);
            mx = max(mx, abs_u32(dvv));
            const int64_t base = (b0 + u) * img + p00;
            if (lg.pool) {
#pragma unroll
                for (int k = 0; k < 4; ++k)
                    delta[base + (k & 1) * dx + (k >> 1) * dy] = k == am[i] ? dvv : 0;
            } else {
                delta[base] = dvv;
            }
        }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    ovf = __any_sync(kFull, ovf);
    if ((threadIdx.x & 31) == 0) {
        if (mx) atomicMax(maxabs_delta, mx);
        if (ovf) atomicOr(status, ST_OVERFLOW);
    }
}

// Same, four features per thread when the last layer's channel count is a
// multiple of 4 (four consecutive features are then four channels of one
// output position): thread (f4, u) takes features q0 + 4 f4 .. + 3 of sample
// b0 + u.  The W_lr slice is staged in shared memory; the argmax codes and
// the region bytes of the four channels are read as 4-byte words and the
// delta written with 16-byte stores.  The dW_lr partials are those of
// k_lr_backward.
template <int GM, int NS>   // NS samples per CTA, 16 NS threads
__global__ void __launch_bounds__(16 * NS) k_lr_backward4(const int8_t* __restrict__ a,
                                                      const int32_t* __restrict__ gl,
                                                      const int32_t* __restrict__ wlr, int B,
                                                      int G, int d, LayerGeom lg, FloorDiv32 alpha,
                                                      const int8_t* __restrict__ region,
                                                      const int8_t* __restrict__ argmax,
                                                      int32_t* __restrict__ delta,
                                                      unsigned long long* __restrict__ dwlr,
                                                      const uint32_t* maxabs_gl,
                                                      const uint32_t* maxabs_wlr,
                                                      uint32_t* maxabs_delta, uint32_t* status) {
    pdl_wait();
    __shared__ int32_t gls[NS][GM];
    __shared__ int8_t as[NS][kLbQ];
    __shared__ __align__(16) int32_t wsl[GM][kLbQ];
    const int f4 = threadIdx.x & 15, u = threadIdx.x >> 4;
    const int q0 = blockIdx.x * kLbQ, q = q0 + 4 * f4;
    const int b0 = blockIdx.y * NS;
    const int nb = min(NS, B - b0);
    for (int i = threadIdx.x; i < NS * GM; i += blockDim.x) {
        const int uu = i / GM, g = i % GM;
        gls[uu][g] = (uu < nb && g < G) ? gl[(int64_t)(b0 + uu) * G + g] : 0;
    }
    for (int i = threadIdx.x; i < NS * kLbQ; i += blockDim.x) {
        const int uu = i / kLbQ, qq = i % kLbQ;
        as[uu][qq] = (uu < nb && q0 + qq < d) ? a[(int64_t)(b0 + uu) * d + q0 + qq] : (int8_t)0;
    }
    for (int i = threadIdx.x; i < GM * kLbQ; i += blockDim.x) {
        const int g = i / kLbQ, qq = i % kLbQ;
        wsl[g][qq] = (g < G && q0 + qq < d) ? wlr[(int64_t)g * d + q0 + qq] : 0;
    }
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0 &&
        int64_bound_exceeded(*maxabs_gl, *maxabs_wlr, G))
        atomicOr(status, ST_OVERFLOW);
    // loads of the delta path go out with the staging loads, before the barrier
    const bool act = q < d && u < nb;      // d % 4 == 0: all four features valid
    int64_t base = 0, dx = 0, dy = 0;
    uint32_t amw = 0, r00 = 0, r01 = 0, r10 = 0, r11 = 0;
    if (act) {
        const int c = q % lg.cout;
        const int r = q / lg.cout;
        const int ox = r % lg.ow, oy = r / lg.ow;
        const int64_t img = lg.pool ? (int64_t)lg.h * lg.w * lg.cout : (int64_t)d;
        const int64_t p00 = lg.pool ? ((int64_t)(2 * oy) * lg.w + 2 * ox) * lg.cout + c : q;
        dx = lg.cout;
        dy = (int64_t)lg.w * lg.cout;
        base = (b0 + u) * img + p00;
        r00 = *reinterpret_cast<const uint32_t*>(region + base);
        if (lg.pool) {
            amw = *reinterpret_cast<const uint32_t*>(argmax + (int64_t)(b0 + u) * d + q);
            r01 = *reinterpret_cast<const uint32_t*>(region + base + dx);
            r10 = *reinterpret_cast<const uint32_t*>(region + base + dy);
            r11 = *reinterpret_cast<const uint32_t*>(region + base + dy + dx);
        }
    }
    __syncthreads();
    // dW_lr partials: (g, q) pairs over the CTA's samples
    for (int i = threadIdx.x; i < G * kLbQ; i += blockDim.x) {
        const int g = i / kLbQ, qq = i - g * kLbQ;
        if (q0 + qq >= d) continue;
        long long t = 0;
#pragma unroll
        for (int uu = 0; uu < NS; ++uu) t += (long long)gls[uu][g] * as[uu][qq];
        if (t != 0) atomicAdd(&dwlr[(int64_t)g * d + q0 + qq], (unsigned long long)t);
    }
    uint32_t mx = 0;
    bool ovf = false;
    if (act) {
        uint64_t acc[4] = {0, 0, 0, 0};    // modulo 2^64, exact below the bound
#pragma unroll
        for (int g = 0; g < GM; ++g) {
            const int4 w4 = *reinterpret_cast<const int4*>(&wsl[g][4 * f4]);
            const int64_t gv = gls[u][g];
            acc[0] += (uint64_t)(gv * w4.x);
            acc[1] += (uint64_t)(gv * w4.y);
            acc[2] += (uint64_t)(gv * w4.z);
            acc[3] += (uint64_t)(gv * w4.w);
        }
        int32_t dv[4];
        int code[4];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int64_t g64 = (int64_t)acc[j];
            ovf |= !fits_i32(g64);
            const int32_t gs = (int32_t)g64;
            // region byte at the recorded window position of channel j
            code[j] = lg.pool ? (int)((amw >> (8 * j)) & 3u) : 0;
            const uint32_t rsel = code[j] == 0 ? r00 : (code[j] == 1 ? r01 : (code[j] == 2 ? r10 : r11));
            const int rg = (int8_t)(rsel >> (8 * j));
            // NITRO-ReLU backward: piece 1 -> floor(g / alpha_inv), piece 2 -> g, else 0
            dv[j] = rg == 1 ? alpha.floor_div(gs) : (rg == 2 ? gs : 0);
            mx = max(mx, abs_u32(dv[j]));
        }
        if (lg.pool) {
#pragma unroll
            for (int k = 0; k < 4; ++k)
                *reinterpret_cast<int4*>(delta + base + (k & 1) * dx + (k >> 1) * dy) =
                    make_int4(code[0] == k ? dv[0] : 0, code[1] == k ? dv[1] : 0,
                              code[2] == k ? dv[2] : 0, code[3] == k ? dv[3] : 0);
        } else {
            *reinterpret_cast<int4*>(delta + base) = make_int4(dv[0], dv[1], dv[2], dv[3]);
        }
    }
#pragma unroll
    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(kFull, mx, off));
    ovf = __any_sync(kFull, ovf);
    if ((threadIdx.x & 31) == 0) {
        if (mx) atomicMax(maxabs_delta, mx);
        if (ovf) atomicOr(status, ST_OVERFLOW);
    }
}

inline int grid_for(int64_t n, int threads, int cap = 152 * 16) {
    int64_t g = (n + threads - 1) / threads;
    return (int)(g < 1 ? 1 : (g > cap ? cap : g));
}

}  // namespace

cudaError_t simt_gemm(int mode, const int8_t* act, const int32_t* grad, const int32_t* wts,
                      int64_t* out, int B, int H, int W, int Cin, int Cout, cudaStream_t s) {
    GemmParams p{act, grad, wts, out, 0, 0, 0, B, H, W, Cin, Cout, 0};
    const int P = B * H * W;
    switch (mode) {
        case GM_CONV_FWD: p.M = P; p.N = Cout; p.K = 9 * Cin; break;
        case GM_CONV_DGRAD: p.M = P; p.N = Cin; p.K = 9 * Cout; break;
        case GM_CONV_WGRAD: p.M = Cout; p.N = 9 * Cin; p.K = P; break;
        case GM_LIN_FWD: p.M = B; p.N = Cout; p.K = Cin; break;
        case GM_LIN_DGRAD: p.M = B; p.N = Cin; p.K = Cout; break;
        case GM_LIN_WGRAD: p.M = Cout; p.N = Cin; p.K = B; break;
        default: return cudaErrorInvalidValue;
    }
    if (p.M <= 0 || p.N <= 0) return cudaSuccess;
    const int tiles_m = (p.M + kTile - 1) / kTile, tiles_n = (p.N + kTile - 1) / kTile;
    // Split K over gridDim.z (64-bit atomics into a zeroed output, exact in any
    // order) until the grid holds about four CTAs per SM, keeping at least
    // 256 K per split.  Weight gradients always reduce over a long K; the
    // forward and input gradient need it when the output has few tiles (a
    // batch of 64 against a linear layer, a 4 x 4 conv map).
    int splits = 1;
    const int64_t tiles = (int64_t)tiles_m * tiles_n;
    if (mode == GM_CONV_WGRAD || mode == GM_LIN_WGRAD || tiles < 2 * 152) {
        const int64_t want = (4 * 152 + tiles - 1) / tiles;
        const int64_t maxs = (p.K + 255) / 256;
        splits = (int)(want < maxs ? want : maxs);
        if (splits < 1) splits = 1;
    }
    p.k_split = ((p.K + splits - 1) / splits + kTK - 1) / kTK * kTK;
    if (p.k_split == 0) p.k_split = kTK;
    splits = p.K > 0 ? (p.K + p.k_split - 1) / p.k_split : 1;
    if (splits > 1 || p.K == 0) {
        cudaError_t e = cudaMemsetAsync(out, 0, sizeof(int64_t) * (size_t)p.M * p.N, s);
        if (e != cudaSuccess) return e;
        if (p.K == 0) return cudaSuccess;
    }
    dim3 grid(tiles_n, tiles_m, splits);
    static const int kIds[6] = {K_SIMT_CONV_FWD, K_SIMT_CONV_DGRAD, K_SIMT_CONV_WGRAD,
                                K_SIMT_LIN_FWD, K_SIMT_LIN_DGRAD, K_SIMT_LIN_WGRAD};
    ProfScope ps(kIds[mode], s, 2.0 * p.M * p.N * p.K, 0.0);
    switch (mode) {
        case GM_CONV_FWD: launch_k(k_gemm<GM_CONV_FWD>, grid, 256, 0, s, p); break;
        case GM_CONV_DGRAD: launch_k(k_gemm<GM_CONV_DGRAD>, grid, 256, 0, s, p); break;
        case GM_CONV_WGRAD: launch_k(k_gemm<GM_CONV_WGRAD>, grid, 256, 0, s, p); break;
        case GM_LIN_FWD: launch_k(k_gemm<GM_LIN_FWD>, grid, 256, 0, s, p); break;
        case GM_LIN_DGRAD: launch_k(k_gemm<GM_LIN_DGRAD>, grid, 256, 0, s, p); break;
        default: launch_k(k_gemm<GM_LIN_WGRAD>, grid, 256, 0, s, p); break;
    }
    return cudaGetLastError();
}

cudaError_t simt_fwd_epilogue(const int64_t* z, const LayerGeom& g, int B, int alpha_inv,
                              int mu, int8_t* out, int8_t* out2, int8_t* region,
                              int8_t* argmax, cudaStream_t s, const DropoutArgs* drop) {
    if (B <= 0) return cudaSuccess;
    const int64_t kdiv = g.kind == NITRO_CONV3X3 ? 9LL * g.cin : (int64_t)g.cin;
    const int64_t n = g.pool ? (int64_t)B * ((g.h + 1) / 2) * ((g.w + 1) / 2) * g.cout
                             : (int64_t)B * g.h * g.w * g.cout;
    DropoutArgs da{};
    if (drop && drop->p16) {
        if (g.pool || !drop->step) return cudaErrorInvalidValue;
        da = *drop;
    }
    ProfScope ps(K_FWD_EPILOGUE, s, 0.0, 0.0);
    launch_k(k_fwd_epilogue, grid_for(n, 256), 256, 0, s, z, g, B, alpha_inv, mu, kdiv, out, out2,
                                                    region, argmax, da);
    return cudaGetLastError();
}

cudaError_t simt_lr_pool_fwd(const int8_t* a, int B, int H, int W, int C, int kh, int kw,
                             int ph, int pw, int8_t* out, uint8_t* am, cudaStream_t s) {
    const int64_t n = (int64_t)B * ph * pw * C;
    if (n <= 0) return cudaSuccess;
    if (kh < 1 || kw < 1 || ph * kh > H || pw * kw > W || kh * kw > 256) return cudaErrorInvalidValue;
    ProfScope ps(K_LR_POOL, s, 0.0, (double)B * H * W * C + 2.0 * n);
    if (C % 4 == 0 && (((uintptr_t)a | (uintptr_t)out | (uintptr_t)am) & 3) == 0)
        launch_k(k_lr_pool_fwd4, grid_for(n / 4, 256), 256, 0, s,
            a, B, H, W, C, kh, kw, ph, pw, FloorDiv32::make((uint32_t)(C / 4)),
            FloorDiv32::make((uint32_t)pw), FloorDiv32::make((uint32_t)ph), out, am);
    else
        launch_k(k_lr_pool_fwd, grid_for(n, 256), 256, 0, s, a, B, H, W, C, kh, kw, ph, pw, out, am);
    return cudaGetLastError();
}

cudaError_t simt_lrpool_to_delta(const int32_t* gl, const int32_t* wlr, int G, int d,
                                 const LayerGeom& g, const LrPoolGeom& lp, int B,
                                 const uint8_t* am, const int8_t* argmax, const int8_t* region,
                                 int alpha_inv, int32_t* delta, const uint32_t* maxabs_gl,
                                 const uint32_t* maxabs_wlr, uint32_t* maxabs_delta,
                                 uint32_t* status, cudaStream_t s) {
    const int64_t n = (int64_t)B * g.h * g.w * g.cout;
    if (n <= 0) return cudaSuccess;
    if (g.kind != NITRO_CONV3X3 || lp.ph * lp.kh > g.oh || lp.pw * lp.kw > g.ow ||
        (int64_t)lp.ph * lp.pw * g.cout != d || alpha_inv < 1)
        return cudaErrorInvalidValue;
    // bytes: region (1) and delta (4) per element, the two argmax codes per
    // pooled position, grad_L and the columns of W_lr read
    ProfScope ps(K_LRPOOL_TO_DELTA, s, 2.0 * B * d * G,
                 5.0 * n + (double)B * g.oh * g.ow * g.cout * (g.pool ? 1 : 0) + (double)B * d +
                     4.0 * G * (B + (double)d));
    int lg_kh = 0, lg_kw = 0;
    while ((1 << lg_kh) < lp.kh) ++lg_kh;
    while ((1 << lg_kw) < lp.kw) ++lg_kw;
    const bool aligned = (((uintptr_t)am | (uintptr_t)region | (uintptr_t)delta |
                           (uintptr_t)(g.pool ? argmax : region)) & 15) == 0;
    if (g.cout % 4 == 0 && aligned && (1 << lg_kh) == lp.kh && (1 << lg_kw) == lp.kw) {
        launch_k(k_lrpool_to_delta4, grid_for(n / 4, 256), 256, 0, s,
            gl, wlr, G, d, g, lp, lg_kh, lg_kw, B, FloorDiv32::make((uint32_t)(g.cout / 4)),
            FloorDiv32::make((uint32_t)g.w), FloorDiv32::make((uint32_t)g.h), am, argmax, region,
            FloorDiv32::make((uint32_t)alpha_inv), delta, maxabs_gl, maxabs_wlr, maxabs_delta,
            status);
    } else {
        launch_k(k_lrpool_to_delta, grid_for(n, 256), 256, 0, s,
            gl, wlr, G, d, g, lp, B, am, argmax, region,
            FloorDiv32::make((uint32_t)alpha_inv), delta, maxabs_gl, maxabs_wlr, maxabs_delta,
            status);
    }
    return cudaGetLastError();
}

size_t simt_learn_scratch(int max_batch, int d, int G) {
    (void)d;
    return (size_t)max_batch * G + (max_batch + kLrSamples - 1) / kLrSamples + 1;
}

cudaError_t simt_learn_fwd(const int8_t* a, const int32_t* wlr, const int32_t* labels, int B,
                           int d, int G, int64_t* zsum, int32_t* grad_l, unsigned long long* sse,
                           int64_t* loss, uint32_t* maxabs_gl, uint32_t* status, cudaStream_t s) {
    if (B <= 0) return cudaSuccess;
    const int groups = (B + kLrSamples - 1) / kLrSamples;
    // partial sums, then the per-group tickets and the final ticket
    cudaError_t e = cudaMemsetAsync(zsum, 0, sizeof(int64_t) * ((size_t)B * G + groups + 1), s);
    if (e != cudaSuccess) return e;
    dim3 grid((d + kLpSlice - 1) / kLpSlice, groups);
    ProfScope ps(K_LEARN_FWD, s, 2.0 * B * d * G, 0.0);
    const int vec8 = d % 8 == 0 && ((uintptr_t)a & 7) == 0;
    launch_k(k_learn_partial, grid, 256, 0, s, a, wlr, B, d, G, vec8,
                                         reinterpret_cast<unsigned long long*>(zsum),
                                         FloorDiv::make((uint64_t)d), labels, grad_l, sse, loss,
                                         maxabs_gl, status);
    return cudaGetLastError();
}

cudaError_t simt_learn_dw(const int8_t* a, const int32_t* grad_l, int B, int d, int G,
                          int64_t* dwlr, cudaStream_t s) {
    dim3 grid((d + 255) / 256, G);
    ProfScope ps(K_LEARN_DW, s, 2.0 * B * d * G, 0.0);
    launch_k(k_learn_dw, grid, 256, 0, s, a, grad_l, B, d, G, dwlr);
    return cudaGetLastError();
}

cudaError_t simt_grad_to_delta(const DeltaSrc& src, const LayerGeom& g, int B, int alpha_inv,
                               const int8_t* region, const int8_t* argmax, int32_t* delta,
                               uint32_t* maxabs_delta, uint32_t* status, cudaStream_t s) {
    if (B <= 0) return cudaSuccess;
    if (g.pool && ((g.h & 1) || (g.w & 1))) {
        cudaError_t e = cudaMemsetAsync(delta, 0, sizeof(int32_t) * (size_t)B * g.h * g.w * g.cout, s);
        if (e != cudaSuccess) return e;
    }
    const int64_t n = (int64_t)B * g.oh * g.ow * g.cout;
    ProfScope ps(K_GRAD_TO_DELTA, s, 0.0, 0.0);
    launch_k(k_grad_to_delta, grid_for(n, 256), 256, 0, s, src, g, B, alpha_inv, region, argmax, delta,
                                                     maxabs_delta, status);
    return cudaGetLastError();
}

cudaError_t simt_integersgd(const SgdBatch& b_in, cudaStream_t s) {
    if (b_in.count <= 0) return cudaSuccess;
    SgdBatch b = b_in;
    int64_t nmax = 0;
    for (int i = 0; i < b.count; ++i) {
        nmax = b.t[i].n > nmax ? b.t[i].n : nmax;
        if (b.t[i].gamma_inv <= 0 || b.t[i].eta_inv < 0) return cudaErrorInvalidValue;
        b.t[i].gdiv = FloorDiv::make((uint64_t)b.t[i].gamma_inv);
        b.t[i].ediv = FloorDiv::make(b.t[i].eta_inv > 0 ? (uint64_t)b.t[i].eta_inv : 1);
        if (b.t[i].planes) {
            if (b.t[i].cin < 1 || b.t[i].n >= ((int64_t)1 << 31)) return cudaErrorInvalidValue;
            b.t[i].cin_div = FloorDiv32::make((uint32_t)b.t[i].cin);
            // planes laid out like W: entry (t, ci) of row co at co 9 cin + t cin + ci,
            // 8-byte aligned for every group of four (plane stride a multiple of 4)
            b.t[i].contig = b.t[i].row_k == 9 * b.t[i].tap_k && b.t[i].tap_k == b.t[i].cin &&
                            b.t[i].plane % 4 == 0 && ((uintptr_t)b.t[i].planes & 7) == 0;
        }
    }
    dim3 grid(grid_for((nmax + 3) / 4, 256, 152 * 4), b.count);
    double bytes = 0;
    for (int i = 0; i < b.count; ++i)
        bytes += (b.t[i].planes ? 24.0 : 16.0) * b.t[i].n;   // W r+w, dW r (+ 4 bf16 planes)
    ProfScope ps(K_INTEGERSGD, s, 0.0, bytes);
    launch_k(k_integersgd, grid, 256, 0, s, b);
    return cudaGetLastError();
}


bool simt_small_conv_ok(const LayerGeom& g) {
    if (g.kind != NITRO_CONV3X3 || g.cin > kSmallCin || g.cout % kSmallCo != 0) return false;
    // weights of the forward and a row chunk of delta for the weight gradient
    // must fit in shared memory
    const int64_t fwd_smem = 4LL * g.cout * 9 * g.cin;
    const int64_t wg_smem = 4LL * kWgRows * g.w * g.cout + (int64_t)(kWgRows + 2) * (g.w + 2) * g.cin;
    return fwd_smem <= 48 * 1024 && wg_smem <= 200 * 1024;
}

cudaError_t simt_conv_small_fwd(const int8_t* x, const int32_t* w, const LayerGeom& g, int B,
                                int alpha_inv, int mu, int8_t* act, int8_t* out2, int8_t* region,
                                int8_t* argmax, uint16_t* next_nhwc, cudaStream_t s) {
    if (B <= 0) return cudaSuccess;
    SmallFwdArgs a{};
    a.x = x; a.w = w; a.B = B; a.H = g.h; a.W = g.w; a.Cin = g.cin; a.Cout = g.cout;
    a.pool = g.pool; a.oh = g.oh; a.ow = g.ow;
    a.sf32 = FloorDiv32::make(9u * (uint32_t)g.cin);
    const int64_t sf = 256LL * 9 * g.cin;
    a.z_hi = 128 * sf;
    a.z_lo = -127 * sf;
    a.alpha = FloorDiv::make((uint64_t)alpha_inv);
    a.mu = mu;
    a.act = act; a.out2 = out2; a.region = region; a.argmax = argmax; a.next_nhwc = next_nhwc;
    const int step = g.pool ? 2 : 1;
    const int64_t n = (int64_t)B * ((g.h + step - 1) / step) * ((g.w + step - 1) / step) * (g.cout / kSmallCo);
    const size_t smem = sizeof(int32_t) * (size_t)g.cout * 9 * g.cin;
    ProfScope ps(K_SIMT_CONV_FWD, s, 2.0 * B * g.h * g.w * g.cout * 9.0 * g.cin, 0.0);
    launch_k(k_conv_small_fwd, grid_for(n, 256, 152 * 32), 256, smem, s, a);
    return cudaGetLastError();
}

cudaError_t simt_conv_small_wgrad(const int8_t* x, const int32_t* d, const LayerGeom& g, int B,
                                  int64_t* dw, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(dw, 0, sizeof(int64_t) * 9 * g.cin * g.cout, s);
    if (e != cudaSuccess || B <= 0) return e;
    dim3 grid((g.h + kWgRows - 1) / kWgRows, B);
    const size_t smem = sizeof(int32_t) * (size_t)kWgRows * g.w * g.cout +
                        (size_t)(kWgRows + 2) * (g.w + 2) * g.cin + 16;
    if (smem > 200 * 1024) return cudaErrorInvalidValue;
    if (smem > 48 * 1024) {
        e = cudaFuncSetAttribute(k_conv_small_wgrad, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
    }
    ProfScope ps(K_SIMT_CONV_WGRAD, s, 2.0 * B * g.h * g.w * g.cout * 9.0 * g.cin, 0.0);
    launch_k(k_conv_small_wgrad, grid, 256, smem, s, x, d, B, g.h, g.w, g.cin, g.cout,
                                               reinterpret_cast<unsigned long long*>(dw));
    return cudaGetLastError();
}

bool simt_lr_backward_ok(int G) { return G <= kLbMaxG; }

cudaError_t simt_lr_backward(const int8_t* a, const int32_t* gl, const int32_t* wlr, int B, int G,
                             int d, const LayerGeom* lg, int alpha_inv, const int8_t* region,
                             const int8_t* argmax, int32_t* delta, int64_t* dwlr,
                             const uint32_t* maxabs_gl, const uint32_t* maxabs_wlr,
                             uint32_t* maxabs_delta, uint32_t* status, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(dwlr, 0, sizeof(int64_t) * (size_t)G * d, s);
    if (e != cudaSuccess || B <= 0) return e;
    if (lg && lg->pool && ((lg->h & 1) || (lg->w & 1))) {   // rows / columns the pool dropped
        e = cudaMemsetAsync(delta, 0, sizeof(int32_t) * (size_t)B * lg->h * lg->w * lg->cout, s);
        if (e != cudaSuccess) return e;
    }
    dim3 grid((d + kLbQ - 1) / kLbQ, (B + kLbSamples - 1) / kLbSamples);
    // the four-feature kernel takes 32 samples per CTA (half the weight-gradient
    // atomics of 16) when the batch fills them
    constexpr int kLb4Samples = 32;
    dim3 grid4((d + kLbQ - 1) / kLbQ, (B + kLb4Samples - 1) / kLb4Samples);
    ProfScope ps(K_LR_BACKWARD, s, (lg ? 4.0 : 2.0) * B * d * G, 0.0);
    const FloorDiv32 al = FloorDiv32::make((uint32_t)(alpha_inv > 0 ? alpha_inv : 1));
    auto* dw64 = reinterpret_cast<unsigned long long*>(dwlr);
    const LayerGeom g0 = lg ? *lg : LayerGeom{};
    // four features per thread: channel counts in multiples of 4 and
    // 16-byte aligned code and delta buffers (this library's own)
    const bool quad = lg && lg->cout % 4 == 0 && d % 4 == 0 &&
                      (((uintptr_t)region | (uintptr_t)delta |
                        (uintptr_t)(lg->pool ? argmax : region)) & 15) == 0;
    if (quad) {
        if (G <= 10)
            launch_k(k_lr_backward4<10, kLb4Samples>, grid4, 16 * kLb4Samples, 0, s,
                a, gl, wlr, B, G, d, g0, al, region, argmax, delta, dw64, maxabs_gl, maxabs_wlr,
                maxabs_delta, status);
        else
            launch_k(k_lr_backward4<kLbMaxG, kLb4Samples>, grid4, 16 * kLb4Samples, 0, s,
                a, gl, wlr, B, G, d, g0, al, region, argmax, delta, dw64, maxabs_gl, maxabs_wlr,
                maxabs_delta, status);
        return cudaGetLastError();
    }
    if (G <= 10)
        launch_k(k_lr_backward<10>, grid, 256, 0, s, a, gl, wlr, B, G, d, lg != nullptr, g0, al, region,
                                               argmax, delta, dw64, maxabs_gl, maxabs_wlr,
                                               maxabs_delta, status);
    else
        launch_k(k_lr_backward<kLbMaxG>, grid, 256, 0, s, a, gl, wlr, B, G, d, lg != nullptr, g0, al,
                                                    region, argmax, delta, dw64, maxabs_gl,
                                                    maxabs_wlr, maxabs_delta, status);
    return cudaGetLastError();
}

}  // namespace nitro
