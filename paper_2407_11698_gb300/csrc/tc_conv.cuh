// Tensor-core (tcgen05) path of the 3x3 conv contractions.
//
// Every operand is split exactly into signed 8-bit limbs, x = sum_l 2^(8l) x_l:
// limbs 0..2 are digits in [-128, 127], limb 3 the remainder in [-128, 128];
// a tensor with max |x| <= 127 / 32639 / 8355711 has zero limbs from index
// 1 / 2 / 3 on, so its first L planes are exact.  Each limb is held as a bf16
// value (exact).  A contraction runs one pass per (A limb, B limb) pair
// on the bf16 tensor pipe with fp32 accumulation in TMEM; every partial sum
// over at most 1024 products of magnitude <= 2^14 is an integer below 2^24 and
// therefore exact, so chunks of 1024 are drained to integers and the passes
// are combined in int64 (modulo 2^64) with shifts 8 (la + lb).
//
// Layouts (bf16, limb planes outermost):
//   act_nhwc  [B][H][W][Cin8]          forward A (K-major: pixels x taps*channels)
//                                      and wgrad A (MN-major: (tap, ci) x pixels)
//   d_nhwc    [L][B][H][W][Cout]       dgrad A (K-major) and wgrad B (MN-major)
//   w_planes  [L][Cout][9][Cin64]      forward B (K-major) and dgrad B (MN-major:
//                                      rows co, 64 consecutive ci)
// Narrow inputs (9 Cin <= 64) use im2col rows instead, see TcLayer::im2col.
// Cin8 = Cin rounded up to 8 (TMA strides are multiples of 16 bytes); Cin64 =
// Cin rounded up to 64 so that a K-block of the forward never spans two taps.  Padding holds zeros; tiles that run past
// a tensor edge read zeros (TMA out-of-bounds fill) and skip their stores.
#pragma once

#include <vector>

#include "nitro_internal.cuh"

namespace nitro {

constexpr int kMaxLimbs = 4;

struct TcLayer {
    bool fwd = false, wgrad = false, dgrad = false;   // passes that run on tcgen05
    // narrow input (9 Cin <= 64, e.g. image channels): act_nhwc holds im2col
    // rows [B][H][W][64] (entry t Cin + ci = input at tap t, zero past 9 Cin)
    // and w_planes is [L][Cout][64]; forward and wgrad see one centred tap.
    bool im2col = false;
    int cin8 = 0;     // channels of the NHWC bf16 input copy (Cin rounded up to 8; 64 for im2col)
    int cin_k = 0;    // channels per tap in the forward K index (Cin rounded up to 64)
    uint16_t* act_nhwc = nullptr;
    uint16_t* d_nhwc = nullptr;
    uint16_t* w_planes = nullptr;
    // device words holding max |W| and max |delta| of the layer: the kernels
    // take their limb counts from them
    const uint32_t* maxabs_w = nullptr;
    const uint32_t* maxabs_d = nullptr;
    // pinned host copies of the two words, refreshed asynchronously; possibly
    // stale, used only to pick a kernel variant (any choice is exact).  By
    // default the layer keeps its own copies (max_host) and refreshes them
    // itself; tc_use_external_hints points them into a caller's mirror that
    // the caller refreshes.
    uint32_t* max_host = nullptr;
    const uint32_t* hint_w = nullptr;
    const uint32_t* hint_d = nullptr;
    bool own_hints = true;
};

// Read the layer's limb-count hints from hint_w / hint_d (pinned host words
// the caller refreshes) instead of copying them from the device per layer.
inline void tc_use_external_hints(TcLayer& t, const uint32_t* hint_w, const uint32_t* hint_d) {
    t.hint_w = hint_w;
    t.hint_d = hint_d;
    t.own_hints = false;
}

// IntegerSGD folded into the weight-gradient kernel (Algorithm 1 with the
// forward layers' gamma_inv and eta_inv): the kernel updates W and its limb
// planes and atomically maxes max |W| into *maxabs_w, which the caller zeroes
// first.  The weight gradient is still written to dW.
struct TcSgd {
    int64_t gamma_inv, eta_inv;   // eta_inv = 0: no decay
    int trunc;                    // NITRO_ROUND_TRUNC
    int32_t* W;
    uint32_t* maxabs_w;
    // the weight limb planes the update writes (null: none): entry (t, ci) of
    // row co at co row_k + t tap_k + ci, or co row_k + i for a linear layer
    uint16_t* planes;
    int64_t plane;
    int row_k, tap_k;
};

// Weight gradient of a linear layer on tcgen05 (dW[o][i] = sum_b delta[b][o]
// a[b][i], the samples as K): for in and out in multiples of 8.  act_bf16 is
// the forward's bf16 copy of the layer input [max_batch][in] (kept by the
// caller); the delta limb planes are allocated here.  t.wgrad is
// false when the layer does not qualify.
bool tc_linear_init(TcLayer& t, const LayerGeom& g, int max_batch, uint16_t* act_bf16,
                    const uint32_t* maxabs_w, const uint32_t* maxabs_d,
                    std::vector<void*>& allocs, std::vector<void*>& host_allocs);

// Decides which passes of a layer run on tensor cores and allocates their
// buffers (device memory recorded in `allocs`, pinned host memory in
// `host_allocs`).  `has_dgrad`: the layer is not the block's first, so its
// input gradient is needed.  maxabs_w / maxabs_d: device words that will hold
// max |W| and max |delta| of the layer.
bool tc_layer_init(TcLayer& t, const LayerGeom& g, int max_batch, bool has_dgrad,
                   const uint32_t* maxabs_w, const uint32_t* maxabs_d,
                   std::vector<void*>& allocs, std::vector<void*>& host_allocs);

// Where IntegerSGD writes the layer's weight planes when it splits the updated
// weights itself: planes [4][Cout][row_k], plane stride, entry (t, ci) of row
// co at co row_k + t tap_k + ci.  *planes = null when the layer has none.
void tc_weight_planes(const TcLayer& t, const LayerGeom& g, uint16_t** planes, int64_t* plane,
                      int* row_k, int* tap_k);

// After such an update: refresh the host hint of max |W|.
cudaError_t tc_weights_hint(TcLayer& t, cudaStream_t s);

// Re-splits the layer's int32 weights into limb planes (after init, an update
// or a checkpoint load); the limb count follows *maxabs_w.
cudaError_t tc_refresh_weights(TcLayer& t, const LayerGeom& g, const int32_t* W,
                               const uint32_t* maxabs_w, cudaStream_t s);

// bf16 NHWC copy of the layer's int8 input for the forward and wgrad operands
// (skipped when the previous layer's epilogue wrote it).
cudaError_t tc_pack_input(TcLayer& t, const LayerGeom& g, const int8_t* x, int batch,
                          bool nhwc_done, cudaStream_t s);

// Outputs of a forward layer for the fused epilogue.
struct TcFwdOut {
    int alpha_inv, mu;
    int8_t* act;          // [B][oh][ow][Cout] int8
    int8_t* out2;         // optional copy (may be null)
    int8_t* region;       // [B][h][w][Cout] int8
    int8_t* argmax;       // [B][oh][ow][Cout] int8 if pooled
    uint16_t* next_nhwc;  // next layer's bf16 input copy, or null
};

// Forward contraction on tcgen05; *done = false if the layer does not run
// there.  With fo != null and Cout % 16 == 0 the epilogue applies
// NITRO-Scaling, NITRO-ReLU and the max-pool and writes fo's outputs
// (*fused = true); otherwise z[p][co] (int64) is written.
cudaError_t tc_conv_forward(TcLayer& t, const LayerGeom& g, int batch, int64_t* z,
                            const TcFwdOut* fo, uint32_t* status, cudaStream_t s, bool* done,
                            bool* fused);

// Splits delta into NHWC limb planes for the wgrad and dgrad passes (limb
// count from *maxabs_delta), unless planes_done (an earlier call split this
// delta already); then refreshes the host hint of max |delta|.  Writing the
// planes from the kernels that produce delta instead (the dgrad epilogue,
// the learning-layer backward) was measured slower than this pass.
cudaError_t tc_pack_delta(TcLayer& t, const LayerGeom& g, const int32_t* delta,
                          const uint32_t* maxabs_delta, int batch, cudaStream_t s,
                          bool planes_done = false);

// tc_pack_delta, then, if wgrad runs on tcgen05, dW = sum_p delta (x)
// im2col(a).  Must precede tc_conv_dgrad.
// True when the layer's weight gradient runs on tcgen05 without a K split at
// this batch, i.e. when tc_conv_wgrad can fold IntegerSGD into it.
bool tc_wgrad_fusable(const TcLayer& t, const LayerGeom& g, int batch);

// With sgd != null the kernel also applies IntegerSGD (see TcSgd) when the
// weight gradient runs on tcgen05 without a K split; *sgd_done says whether
// it did (the caller updates the layer otherwise).
cudaError_t tc_conv_wgrad(TcLayer& t, const LayerGeom& g, const int32_t* delta,
                          const uint32_t* maxabs_delta, int batch, int64_t* dW,
                          uint32_t* status, cudaStream_t s, bool* done,
                          bool planes_done = false, const TcSgd* sgd = nullptr,
                          bool* sgd_done = nullptr);

// Where the input gradient goes when the dgrad epilogue is fused: through the
// lower layer's max-pool backward and NITRO-ReLU backward into its delta.
struct TcDgradOut {
    int alpha_inv;
    const uint32_t* maxabs_delta;   // this layer's max|delta| and max|W|
    const uint32_t* maxabs_w;
    int low_h, low_w, low_pool;     // lower layer's pre-pool size and pool flag
    const int8_t* low_region;
    const int8_t* low_argmax;
    int32_t* low_delta;             // [B][low_h][low_w][Cin] int32
    uint32_t* low_maxabs;           // max|lower delta| (atomic max)
};

// g[p][ci] = sum_(t,co) delta[p - tap t][co] W[co][t][ci] on tcgen05
// (*done = false if the layer does not run there).  With fo != null and
// Cin % 16 == 0 the epilogue produces the lower layer's delta (*fused = true);
// otherwise g is written as int64 to g64.
cudaError_t tc_conv_dgrad(TcLayer& t, const LayerGeom& g, int batch, int64_t* g64,
                          const TcDgradOut* fo, uint32_t* status, cudaStream_t s, bool* done,
                          bool* fused);

// One CTA that holds TMEM and waits, through the contraction kernel's bounded
// mbarrier wait, on a barrier nothing completes: after limit_ns it raises
// ST_TIMEOUT in *status, frees TMEM and returns.
cudaError_t tc_timeout_probe(uint32_t* status, uint64_t limit_ns, cudaStream_t s);

// Helpers of the kernel-level entry points (contract.cu).
cudaError_t tc_maxabs(const int32_t* x, int64_t n, uint32_t* out, cudaStream_t s);
cudaError_t tc_pack_int8(const int8_t* x, int64_t rows, int cols, uint16_t* out, cudaStream_t s);
// n % 8 == 0; planes [4][n], limb count from *maxabs
cudaError_t tc_pack_limbs(const int32_t* x, int64_t n, const uint32_t* maxabs, uint16_t* planes,
                          cudaStream_t s);
// C[m][n] (int64) = sum_k A[m][k] B[n][k]; A bf16 [M][K] (int8 values), B limb
// planes [4][N][K] (limb count from *max_b); K % 8 == 0.
cudaError_t tc_gemm_run(const uint16_t* a_bf16, const uint16_t* b_planes, int M, int N, int K,
                        const uint32_t* max_b, int64_t* out, uint32_t* status, cudaStream_t s);

}  // namespace nitro
