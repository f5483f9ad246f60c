// Internal declarations of the GB300 NITRO-D library (not part of the ABI).
#pragma once

#include <cstdint>
#include <utility>
#include <cuda_runtime.h>

#include "nitro.h"

namespace nitro {

// ---------------------------------------------------------------------------
// Integer helpers, device and host.  fdiv is the paper's \intdiv (floor).
// ---------------------------------------------------------------------------
__host__ __device__ __forceinline__ int64_t fdiv64(int64_t x, int64_t d) {
    int64_t q = x / d;
    return (x % d < 0) ? q - 1 : q;
}
__host__ __device__ __forceinline__ int32_t fdiv32(int32_t x, int32_t d) {
    int32_t q = x / d;
    return (x % d < 0) ? q - 1 : q;
}
__host__ __device__ __forceinline__ int64_t tdiv64(int64_t x, int64_t d) { return x / d; }

// floor(z / (256 * k)) = floor(floor(z / 256) / k) for k > 0; the first step
// is an arithmetic shift.
__host__ __device__ __forceinline__ int64_t scale_floor(int64_t z, int64_t k) {
    return fdiv64(z >> 8, k);
}

// Floor division by an invariant positive integer d through a multiply-high,
// after Granlund & Montgomery, "Division by invariant integers using
// multiplication" (PLDI 1994), Fig. 4.1 (N = 64): with l = ceil(log2 d),
// m = floor(2^64 (2^l - d) / d) + 1, sh1 = min(l, 1), sh2 = max(l - 1, 0),
// floor(n / d) = (t + ((n - t) >> sh1)) >> sh2 with t = mulhi(m, n), for every
// unsigned 64-bit n.  Negative x use floor(x / d) = -floor((-x - 1) / d) - 1.
struct FloorDiv {
    uint64_t m;
    int sh1, sh2;
    __host__ static FloorDiv make(uint64_t d) {
        int l = 0;
        while (l < 64 && ((uint64_t)1 << l) < d) ++l;
        FloorDiv f;
        const unsigned __int128 two_l = (unsigned __int128)1 << l;
        f.m = (uint64_t)((((unsigned __int128)1 << 64) * (two_l - d)) / d + 1);
        f.sh1 = l < 1 ? l : 1;
        f.sh2 = l > 1 ? l - 1 : 0;
        return f;
    }
    __host__ __device__ __forceinline__ uint64_t udiv(uint64_t n) const {
#ifdef __CUDA_ARCH__
        const uint64_t t = __umul64hi(m, n);
#else
        const uint64_t t = (uint64_t)(((unsigned __int128)m * n) >> 64);
#endif
        return (t + ((n - t) >> sh1)) >> sh2;
    }
    __host__ __device__ __forceinline__ int64_t floor_div(int64_t x) const {
        if (x >= 0) return (int64_t)udiv((uint64_t)x);
        return -(int64_t)udiv((uint64_t)(-(x + 1))) - 1;
    }
    __host__ __device__ __forceinline__ int64_t trunc_div(int64_t x) const {
        if (x >= 0) return (int64_t)udiv((uint64_t)x);
        return -(int64_t)udiv((uint64_t)(-(x + 1)) + 1);
    }
};

// The same method with N = 32 for 32-bit operands (one 32-bit multiply-high).
struct FloorDiv32 {
    uint32_t m;
    int sh1, sh2;
    __host__ static FloorDiv32 make(uint32_t d) {
        int l = 0;
        while (l < 32 && ((uint64_t)1 << l) < d) ++l;
        FloorDiv32 f;
        f.m = (uint32_t)((((uint64_t)1 << 32) * (((uint64_t)1 << l) - d)) / d + 1);
        f.sh1 = l < 1 ? l : 1;
        f.sh2 = l > 1 ? l - 1 : 0;
        return f;
    }
    __host__ __device__ __forceinline__ uint32_t udiv(uint32_t n) const {
#ifdef __CUDA_ARCH__
        const uint32_t t = __umulhi(m, n);
#else
        const uint32_t t = (uint32_t)(((uint64_t)m * n) >> 32);
#endif
        return (t + ((n - t) >> sh1)) >> sh2;
    }
    // branch-free: for x < 0, ~x = -(x + 1) and ~q = -q - 1
    __host__ __device__ __forceinline__ int32_t floor_div(int32_t x) const {
        const uint32_t ux = x >= 0 ? (uint32_t)x : ~(uint32_t)x;
        const uint32_t q = udiv(ux);
        return x >= 0 ? (int32_t)q : (int32_t)~q;
    }
};

__host__ __device__ __forceinline__ bool fits_i32(int64_t v) {
    return v >= INT32_MIN && v <= INT32_MAX;
}

// NITRO-ReLU piece of x: 0 x<-127, 1 -127<=x<0, 2 0<=x<=127, 3 x>127.
__host__ __device__ __forceinline__ int relu_region(int64_t x) {
    return x < -127 ? 0 : (x < 0 ? 1 : (x <= 127 ? 2 : 3));
}
// NITRO-ReLU forward value (Sec. 3.2.2).
__host__ __device__ __forceinline__ int relu_value(int64_t x, int alpha_inv, int mu) {
    if (x < 0) {
        int c = x < -127 ? -127 : (int)x;
        return fdiv32(c, alpha_inv) - mu;
    }
    return (x > 127 ? 127 : (int)x) - mu;
}
// Same, with the slope division through a precomputed divider.
__host__ __device__ __forceinline__ int relu_value(int64_t x, const FloorDiv& alpha, int mu) {
    if (x < 0) {
        int64_t c = x < -127 ? -127 : x;
        return (int)alpha.floor_div(c) - mu;
    }
    return (x > 127 ? 127 : (int)x) - mu;
}
// NITRO-ReLU backward per piece.
__host__ __device__ __forceinline__ int32_t relu_backward(int32_t g, int region, int alpha_inv) {
    return region == 1 ? fdiv32(g, alpha_inv) : (region == 2 ? g : 0);
}

__host__ __device__ __forceinline__ uint32_t abs_u32(int32_t v) {
    return v < 0 ? (uint32_t)(-(int64_t)v) : (uint32_t)v;
}

// SplitMix64 (Steele, Lea & Flood, OOPSLA 2014), random-access form: output
// `index` of the generator seeded with `seed` is the published finaliser
// applied to seed + (index + 1) * 0x9E3779B97F4A7C15.
__host__ __device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t index) {
    uint64_t z = seed + (index + 1ULL) * 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

// Dropout of the linear forward layers (App. B, p_l): element e of forward
// layer `layer` at step t is dropped when the top 16 bits of output
// 2^63 + t 2^35 + layer 2^31 + e of the block's SplitMix64 stream are below
// p16 (rate in units of 2^-16; t modulo 2^28, layer < 16, e < 2^31).
constexpr int kRegionDropped = 4;   // region code of a dropped activation
struct DropoutArgs {
    uint64_t seed;
    uint32_t p16;           // 0 = off
    int layer;
    const uint32_t* step;   // device step counter
};
__host__ __device__ __forceinline__ bool dropout_drop(uint64_t seed, uint32_t t, int layer,
                                                      uint64_t e, uint32_t p16) {
    const uint64_t idx = (1ULL << 63) + ((uint64_t)(t & ((1u << 28) - 1)) << 35) +
                         ((uint64_t)layer << 31) + e;
    return (uint32_t)(splitmix64_at(seed, idx) >> 48) < p16;
}

// max|A| * max|B| * k >= 2^63 : int64 exactness of an int32 x int32
// contraction of length k is no longer guaranteed.
__host__ __device__ __forceinline__ bool int64_bound_exceeded(uint32_t ma, uint32_t mb, int64_t k) {
    unsigned __int128 p = (unsigned __int128)ma * mb * (unsigned __int128)k;
    return p >= ((unsigned __int128)1 << 63);
}

// ---------------------------------------------------------------------------
// Layer geometry as the kernels see it.
// ---------------------------------------------------------------------------
struct LayerGeom {
    int kind;       // NITRO_CONV3X3 / NITRO_LINEAR
    int cin, cout;  // linear: cin = in features, cout = out features
    int h, w;       // input spatial (1 for linear)
    int pool;       // 2x2 max-pool after NITRO-ReLU
    int oh, ow;     // output spatial after the optional pool
};

// Device status word bits (same values as the ABI's NITRO_STATUS_BIT_*).
enum : uint32_t { ST_OVERFLOW = 1u, ST_BAD_LABEL = 2u, ST_TIMEOUT = 4u };

// ---------------------------------------------------------------------------
// CUDA-core kernels (kernels_simt.cu).  All launch on `s`, return the launch
// error, and do nothing for empty problems.
// ---------------------------------------------------------------------------
enum GemmMode : int {
    GM_CONV_FWD = 0,    // C[p][co]      = sum_(t,ci) a[p + tap t][ci] * W[co][t][ci]
    GM_CONV_DGRAD = 1,  // C[p][ci]      = sum_(t,co) g[p - tap t][co] * W[co][t][ci]
    GM_CONV_WGRAD = 2,  // C[co][(t,ci)] = sum_p g[p][co] * a[p + tap t][ci]
    GM_LIN_FWD = 3,     // C[b][o] = sum_i a[b][i] * W[o][i]
    GM_LIN_DGRAD = 4,   // C[b][i] = sum_o g[b][o] * W[o][i]
    GM_LIN_WGRAD = 5    // C[o][i] = sum_b g[b][o] * a[b][i]
};

// Exact int64 implicit GEMM on CUDA cores.  act: int8 activations, grad:
// int32 gradients, wts: int32 weights; out: int64, row-major C (overwritten).
cudaError_t simt_gemm(int mode, const int8_t* act, const int32_t* grad, const int32_t* wts,
                      int64_t* out, int B, int H, int W, int Cin, int Cout, cudaStream_t s);

// z (int64, pre-pool NHWC) -> NITRO-Scaling -> NITRO-ReLU -> region codes,
// optional 2x2 max-pool with argmax codes, int8 outputs (out2 may be NULL).
// With drop.p16 > 0 (linear layers, no pool) dropped outputs are stored as 0
// with region code kRegionDropped.
cudaError_t simt_fwd_epilogue(const int64_t* z, const LayerGeom& g, int B, int alpha_inv,
                              int mu, int8_t* out, int8_t* out2, int8_t* region,
                              int8_t* argmax, cudaStream_t s, const DropoutArgs* drop = nullptr);

// Learning-layer max-pool (Sec. 3.3, z^mp): a [B][H][W][C] int8 -> out
// [B][ph][pw][C] over kh x kw windows with stride (kh, kw), first maximum in
// row-major window order, its position r*kw + s in am.
cudaError_t simt_lr_pool_fwd(const int8_t* a, int B, int H, int W, int C, int kh, int kw,
                             int ph, int pw, int8_t* out, uint8_t* am, cudaStream_t s);

// delta_fw = grad_l W_lr at the pooled learning features (int32 storage rule,
// int64 bound check), routed back through the learning-layer pool (window
// maximum am), the 2x2 max-pool of conv layer g (argmax) and NITRO-ReLU
// backward into g's delta [B][h][w][cout]; every element is written.
struct LrPoolGeom {
    int kh, kw, ph, pw;
};
cudaError_t simt_lrpool_to_delta(const int32_t* gl, const int32_t* wlr, int G, int d,
                                 const LayerGeom& g, const LrPoolGeom& lp, int B,
                                 const uint8_t* am, const int8_t* argmax, const int8_t* region,
                                 int alpha_inv, int32_t* delta, const uint32_t* maxabs_gl,
                                 const uint32_t* maxabs_wlr, uint32_t* maxabs_delta,
                                 uint32_t* status, cudaStream_t s);

// Learning layer forward + loss: grad_l = floor(a W^T / (256 d)) - 32 onehot,
// sse = sum grad_l^2 (mod 2^64), loss = floor(sse / 2) (if loss != NULL),
// max|grad_l| into *maxabs_gl, status bits.  scratch: int64 buffer of
// simt_learn_scratch(max_batch, d, G) words (partial sums and tickets,
// cleared by each call); *sse must be zero on entry.
size_t simt_learn_scratch(int max_batch, int d, int G);
cudaError_t simt_learn_fwd(const int8_t* a, const int32_t* wlr, const int32_t* labels, int B,
                           int d, int G, int64_t* scratch, int32_t* grad_l, unsigned long long* sse,
                           int64_t* loss, uint32_t* maxabs_gl, uint32_t* status, cudaStream_t s);

// dW_lr[g][j] = sum_b grad_l[b][g] a[b][j]
cudaError_t simt_learn_dw(const int8_t* a, const int32_t* grad_l, int B, int d, int G,
                          int64_t* dwlr, cudaStream_t s);

// Gradient at the output of layer g (post-pool) -> delta at its
// pre-activation: max-pool backward, NITRO-ReLU backward, STE.  The source
// is either delta_fw = grad_l W_lr (lr_wlr != NULL) or an int64 dgrad output.
struct DeltaSrc {
    const int32_t* grad_l;   // [B][G]   (learning-layer source)
    const int32_t* wlr;      // [G][d]
    int G;
    const uint32_t* maxabs_a;  // bound check operands: max|grad| and max|W|
    const uint32_t* maxabs_b;
    int64_t bound_k;           // contraction length for the bound
    const int64_t* g64;      // [B][out features of the layer] (dgrad source)
};
cudaError_t simt_grad_to_delta(const DeltaSrc& src, const LayerGeom& g, int B, int alpha_inv,
                               const int8_t* region, const int8_t* argmax, int32_t* delta,
                               uint32_t* maxabs_delta, uint32_t* status, cudaStream_t s);

// Narrow-input conv (Cin <= 8, Cout % 16 == 0): fused forward (writes act,
// out2, region, argmax and, if next_nhwc != null, a bf16 copy of act) and
// weight gradient (dw overwritten).
bool simt_small_conv_ok(const LayerGeom& g);
cudaError_t simt_conv_small_fwd(const int8_t* x, const int32_t* w, const LayerGeom& g, int B,
                                int alpha_inv, int mu, int8_t* act, int8_t* out2, int8_t* region,
                                int8_t* argmax, uint16_t* next_nhwc, cudaStream_t s);
cudaError_t simt_conv_small_wgrad(const int8_t* x, const int32_t* d, const LayerGeom& g, int B,
                                  int64_t* dw, cudaStream_t s);

// Learning-layer backward for G <= 16, fused: dW_lr (overwritten) and, when
// lg (geometry of the block's last forward layer) is not null, that layer's
// delta from delta_fw = grad_L W_lr (pre-update), with the int32 storage
// rule, the int64 bound check, max-pool and NITRO-ReLU backward.  d: features
// of the block output.
bool simt_lr_backward_ok(int G);
cudaError_t simt_lr_backward(const int8_t* a, const int32_t* gl, const int32_t* wlr, int B, int G,
                             int d, const LayerGeom* lg, int alpha_inv, const int8_t* region,
                             const int8_t* argmax, int32_t* delta, int64_t* dwlr,
                             const uint32_t* maxabs_gl, const uint32_t* maxabs_wlr,
                             uint32_t* maxabs_delta, uint32_t* status, cudaStream_t s);

// IntegerSGD (Algorithm 1) over up to kMaxSgdTensors tensors in one launch.
constexpr int kMaxSgdTensors = 16;
struct SgdTensor {
    int32_t* w;
    const int64_t* dw;
    int64_t n;
    int64_t gamma_inv, eta_inv;
    uint32_t* maxabs_w;
    FloorDiv gdiv, ediv;   // dividers for gamma_inv and eta_inv (filled by simt_integersgd)
    // optional bf16 limb planes of a conv weight [Cout][9][cin] that the update
    // writes itself: planes[l plane + co row_k + t tap_k + ci], all four limbs
    uint16_t* planes;
    int64_t plane;
    int row_k, tap_k, cin;
    FloorDiv32 cin_div;    // filled by simt_integersgd
    bool contig;           // planes laid out like W (filled by simt_integersgd)
};
struct SgdBatch {
    SgdTensor t[kMaxSgdTensors];
    int count;
    int round_trunc;
    uint32_t* status;
    uint32_t* step;        // block step counter, incremented once per launch (or null)
};
cudaError_t simt_integersgd(const SgdBatch& b, cudaStream_t s);


// ---------------------------------------------------------------------------
// Programmatic dependent launch.  A kernel queued with launch_k may start
// (get SMs, set up shared memory, barriers and TMEM) while the kernel before
// it in the stream is still finishing; every kernel so queued executes
// pdl_wait() in each thread before its first access to global memory, which
// blocks until the previous kernel has completed and its writes are visible.
// pdl_trigger() lets the next kernel of the stream start launching; it only
// takes effect once every CTA of this kernel has executed it or exited.
// Both are no-ops for a kernel queued without the attribute.  Only the
// contraction kernel triggers, once its MMAs are issued: an early trigger
// lets the next kernel's waiting CTAs hold SMs that kernels of the other
// block streams would use (measured slower on the VGG-style step), and the
// other kernels trigger implicitly when their CTAs exit.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Whether launch_k queues kernels with the programmatic-serialization
// attribute (on unless the environment sets NITRO_PDL=0; read once).
bool pdl_enabled();

template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t s, Args&&... args) {
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = pdl_enabled() ? 1 : 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace nitro
