// C ABI of the NITRO-D block step (declared in include/nitro.h): argument
// checks, device memory of a block, and the launch sequence of forward,
// backward and IntegerSGD on the caller's stream.
#include <cstdio>
#include <cstdlib>
#include <algorithm>
#include <cstring>
#include <new>
#include <vector>

#include "nitro_internal.cuh"
#include "tc_conv.cuh"

using namespace nitro;

namespace {

constexpr int kLearningTensorId = 255;
constexpr int kMaxLayers = kMaxSgdTensors - 1;

struct Layer {
    LayerGeom g;
    int64_t in_f, out_f, pre_f;  // per-sample sizes: input, output (post-pool), pre-pool
    int64_t wcount;
    int32_t* W = nullptr;
    int64_t* dW = nullptr;
    int8_t* act = nullptr;       // [max_batch x out_f]
    int8_t* region = nullptr;    // [max_batch x pre_f]
    int8_t* argmax = nullptr;    // [max_batch x out_f] if pool
    int32_t* delta = nullptr;    // [max_batch x pre_f]
    TcLayer tc;                  // tensor-core state (limb planes, maps)
    uint16_t* lin_a = nullptr;       // linear on tcgen05: bf16 input [max_batch x in]
    uint16_t* lin_planes = nullptr;  // and weight limb planes [4][out][in]
};

// Linear forward on the tcgen05 GEMM: rows of 16-byte multiples for TMA
// (in % 8 == 0), and large enough to beat the CUDA-core kernel.
bool lin_tc_ok(const nitro_layer_desc& l) {
    return l.kind == NITRO_LINEAR && l.cin % 8 == 0 && l.cin >= 64 &&
           (int64_t)l.cin * l.cout >= 4096 && (int64_t)l.cin * l.cout < ((int64_t)1 << 31);
}

}  // namespace

struct nitro_block {
    nitro_block_desc desc{};
    std::vector<Layer> L;
    int G = 0, mu = 0;
    int64_t d = 0;
    int32_t* Wlr = nullptr;
    int64_t* dWlr = nullptr;
    int32_t* grad_l = nullptr;      // [max_batch x G]
    int64_t* zsum = nullptr;        // learning-layer partial sums and ticket (simt_learn_scratch)
    int64_t* z64 = nullptr;         // scratch, int64 pre-activations / dgrad outputs
    size_t z64_elems = 0;
    uint32_t* words = nullptr;      // [0] status [1] step counter (dropout masks)
                                    // [2] max|W_lr| [3 + i] max|W_i|    (reset by the update)
                                    // [3 + n] max|grad_l| [4 + n + i] max|delta_i|, then the
                                    // SSE (8-byte aligned)              (reset by the backward)
    uint32_t* words_host = nullptr; // pinned copy of the words, refreshed once per step: the
                                    // limb-count hints that pick kernel variants
    uint64_t seed = 0;
    LrPoolGeom lp{1, 1, 0, 0};      // learning-layer pool window and output grid
    int8_t* zmp = nullptr;          // [max_batch x d] pooled learning input, or null
    uint8_t* lr_am = nullptr;       // [max_batch x d] its window positions
    unsigned long long* sse = nullptr;
    int batch = 0;
    std::vector<void*> allocs;
    std::vector<void*> host_allocs;
};

namespace {

uint32_t* w_status(nitro_block* b) { return b->words; }
uint32_t* w_step(nitro_block* b) { return b->words + 1; }
uint32_t* w_wlr(nitro_block* b) { return b->words + 2; }
uint32_t* w_w(nitro_block* b, int i) { return b->words + 3 + i; }
uint32_t* w_gl(nitro_block* b) { return b->words + 3 + (int)b->L.size(); }
uint32_t* w_delta(nitro_block* b, int i) { return b->words + 4 + (int)b->L.size() + i; }
int sse_word(int n_layers) { return (4 + 2 * n_layers + 1) & ~1; }   // 8-byte aligned
int n_words(int n_layers) { return sse_word(n_layers) + 2; }

template <typename T>
bool dalloc(nitro_block* b, T** p, size_t count) {
    void* q = nullptr;
    if (count == 0) count = 1;
    if (cudaMalloc(&q, count * sizeof(T)) != cudaSuccess) return false;
    b->allocs.push_back(q);
    *p = static_cast<T*>(q);
    return true;
}

void free_all(nitro_block* b) {
    for (void* p : b->allocs) cudaFree(p);
    for (void* p : b->host_allocs) cudaFreeHost(p);
    b->allocs.clear();
    b->host_allocs.clear();
}

int64_t isqrt64(int64_t n) {
    if (n <= 0) return 0;
    int64_t r = 0;
    for (int64_t bit = (int64_t)1 << 62; bit; bit >>= 2) {  // digit-by-digit
        if (n >= r + bit) { n -= r + bit; r = (r >> 1) + bit; } else { r >>= 1; }
    }
    return r;
}

// Integer Kaiming bound (Sec. 3.3.1)
int64_t kaiming_bound(int64_t fan_in) { return fdiv64(128 * 1732, isqrt64(fan_in) * 1000); }

std::vector<int32_t> draw_weights(int64_t n, int64_t fan_in, uint64_t seed, uint64_t tensor_id) {
    const int64_t b = kaiming_bound(fan_in);
    const uint64_t span = (uint64_t)(2 * b + 1);
    std::vector<int32_t> w((size_t)n);
    for (int64_t e = 0; e < n; ++e)
        w[(size_t)e] = (int32_t)((int64_t)(splitmix64_at(seed, (tensor_id << 40) + (uint64_t)e) % span) - b);
    return w;
}

// Learning-layer pooling window (Sec. 3.3 z^mp, App. B d^lr): grow a 1 x 1
// window by doubling its height, then its width, alternately, while the
// pooled C x floor(H/kh) x floor(W/kw) map holds more than d_lr values and
// the window still fits; a side that cannot double leaves the other to grow.
void lr_window(int64_t C, int H, int W, int d_lr, int* kh_out, int* kw_out) {
    int kh = 1, kw = 1;
    if (d_lr > 0) {
        while (C * (H / kh) * (W / kw) > d_lr) {
            if (kh <= kw && 2 * kh <= H) kh *= 2;
            else if (2 * kw <= W) kw *= 2;
            else if (2 * kh <= H) kh *= 2;
            else break;
        }
    }
    *kh_out = kh;
    *kw_out = kw;
}

uint32_t host_maxabs(const int32_t* p, size_t n) {
    uint32_t m = 0;
    for (size_t i = 0; i < n; ++i) m = abs_u32(p[i]) > m ? abs_u32(p[i]) : m;
    return m;
}


#define NITRO_TRY(expr)                                \
    do {                                               \
        cudaError_t _e = (expr);                       \
        if (_e != cudaSuccess) return NITRO_ERR_CUDA;  \
    } while (0)

nitro_status validate(const nitro_block_desc* d) {
    if (!d) return NITRO_ERR_ARG;
    if (d->n_layers < 0 || d->n_layers > kMaxLayers) return NITRO_ERR_ARG;
    if (d->n_layers > 0 && !d->layers) return NITRO_ERR_ARG;
    if (d->num_classes < 1 || d->num_classes > 64) return NITRO_ERR_ARG;
    if (d->alpha_inv < 2 || d->alpha_inv > (1 << 20)) return NITRO_ERR_ARG;
    if (d->gamma_inv_lr < 1 || d->gamma_inv_lr > ((int64_t)1 << 48)) return NITRO_ERR_ARG;
    if (d->eta_inv_fw < 0 || d->eta_inv_lr < 0) return NITRO_ERR_ARG;
    if (d->sgd_round != NITRO_ROUND_FLOOR && d->sgd_round != NITRO_ROUND_TRUNC) return NITRO_ERR_ARG;
    if (d->max_batch < 0 || d->max_batch > 1000000) return NITRO_ERR_ARG;
    if (d->in_features < 1 || d->in_features > (1 << 24)) return NITRO_ERR_ARG;
    if (d->d_lr < 0 || d->dropout_p16 < 0 || d->dropout_p16 > 65536) return NITRO_ERR_ARG;
    int64_t prev_out = d->in_features;
    for (int i = 0; i < d->n_layers; ++i) {
        const nitro_layer_desc& l = d->layers[i];
        if (l.cin < 1 || l.cout < 1 || l.cin > (1 << 20) || l.cout > (1 << 20)) return NITRO_ERR_ARG;
        if (l.pool2x2 != 0 && l.pool2x2 != 1) return NITRO_ERR_ARG;
        int64_t in_f, out_f, pre_f;
        if (l.kind == NITRO_CONV3X3) {
            if (l.h < 1 || l.w < 1) return NITRO_ERR_ARG;
            if (l.pool2x2 && (l.h < 2 || l.w < 2)) return NITRO_ERR_ARG;
            in_f = (int64_t)l.h * l.w * l.cin;
            pre_f = (int64_t)l.h * l.w * l.cout;
            out_f = l.pool2x2 ? (int64_t)(l.h / 2) * (l.w / 2) * l.cout : pre_f;
            // wgrad sums B*h*w terms of |delta| < 2^31 times |a| <= 2^7
            if ((int64_t)d->max_batch * l.h * l.w > ((int64_t)1 << 24)) return NITRO_ERR_ARG;
        } else if (l.kind == NITRO_LINEAR) {
            if (l.h != 1 || l.w != 1 || l.pool2x2) return NITRO_ERR_ARG;
            in_f = l.cin;
            pre_f = out_f = l.cout;
        } else {
            return NITRO_ERR_ARG;
        }
        if (in_f != prev_out) return NITRO_ERR_ARG;
        if (pre_f > (1 << 24) || in_f > (1 << 24)) return NITRO_ERR_ARG;
        if ((int64_t)d->max_batch * (pre_f > in_f ? pre_f : in_f) >= ((int64_t)1 << 31)) return NITRO_ERR_ARG;
        prev_out = out_f;
    }
    if ((int64_t)d->max_batch * prev_out >= ((int64_t)1 << 31)) return NITRO_ERR_ARG;
    if (d->n_layers > 0) {
        const nitro_layer_desc& l = d->layers[d->n_layers - 1];
        if (l.kind == NITRO_CONV3X3) {
            int kh, kw;
            lr_window(l.cout, l.pool2x2 ? l.h / 2 : l.h, l.pool2x2 ? l.w / 2 : l.w, d->d_lr, &kh, &kw);
            if (kh * kw > 256) return NITRO_ERR_UNSUPPORTED;
        }
    }
    return NITRO_OK;
}

}  // namespace

extern "C" {

const char* nitro_status_str(nitro_status s) {
    switch (s) {
        case NITRO_OK: return "ok";
        case NITRO_ERR_ARG: return "invalid argument";
        case NITRO_ERR_OVERFLOW: return "integer overflow";
        case NITRO_ERR_TIMEOUT: return "device wait timed out";
        case NITRO_ERR_CUDA: return "CUDA error";
        case NITRO_ERR_UNSUPPORTED: return "unsupported";
    }
    return "unknown status";
}

nitro_status nitro_init_block(const nitro_block_desc* desc, uint64_t seed, void* stream,
                              nitro_block** out) {
    if (!out) return NITRO_ERR_ARG;
    *out = nullptr;
    nitro_status st = validate(desc);
    if (st != NITRO_OK) return st;
    cudaStream_t s = (cudaStream_t)stream;
    nitro_block* b = new (std::nothrow) nitro_block();
    if (!b) return NITRO_ERR_CUDA;
    b->desc = *desc;
    b->desc.layers = nullptr;
    b->G = desc->num_classes;
    {
        // mu_int8: floor-average of the four segment means (Sec. 3.2.2)
        const int a = desc->alpha_inv;
        b->mu = (int)fdiv64(fdiv64(-127, a) + fdiv64(-127, 2 * a) + 63 + 127, 4);
    }
    const int MB = desc->max_batch;
    size_t z_need = 0;
    bool ok = true;
    std::vector<std::vector<int32_t>> host_w;
    for (int i = 0; i < desc->n_layers && ok; ++i) {
        const nitro_layer_desc& l = desc->layers[i];
        Layer ly;
        ly.g.kind = l.kind; ly.g.cin = l.cin; ly.g.cout = l.cout;
        ly.g.h = l.h; ly.g.w = l.w; ly.g.pool = l.pool2x2;
        ly.g.oh = l.pool2x2 ? l.h / 2 : l.h;
        ly.g.ow = l.pool2x2 ? l.w / 2 : l.w;
        ly.in_f = (int64_t)l.h * l.w * l.cin;
        ly.pre_f = (int64_t)l.h * l.w * l.cout;
        ly.out_f = (int64_t)ly.g.oh * ly.g.ow * l.cout;
        const int64_t fan_in = l.kind == NITRO_CONV3X3 ? 9LL * l.cin : (int64_t)l.cin;
        ly.wcount = (int64_t)l.cout * fan_in;
        ok = ok && dalloc(b, &ly.W, ly.wcount) && dalloc(b, &ly.dW, ly.wcount) &&
             dalloc(b, &ly.act, (size_t)MB * ly.out_f) &&
             dalloc(b, &ly.region, (size_t)MB * ly.pre_f) &&
             dalloc(b, &ly.delta, (size_t)MB * ly.pre_f);
        if (ok && l.pool2x2) ok = dalloc(b, &ly.argmax, (size_t)MB * ly.out_f);
        if (ok && lin_tc_ok(l))
            ok = dalloc(b, &ly.lin_a, (size_t)MB * l.cin) &&
                 dalloc(b, &ly.lin_planes, (size_t)kMaxLimbs * ly.wcount);
        z_need = std::max(z_need, (size_t)MB * (size_t)ly.pre_f);
        z_need = std::max(z_need, (size_t)MB * (size_t)ly.in_f);
        host_w.push_back(draw_weights(ly.wcount, fan_in, seed, (uint64_t)i));
        b->L.push_back(ly);
    }
    b->seed = seed;
    b->d = desc->n_layers ? b->L.back().out_f : desc->in_features;
    if (desc->n_layers && b->L.back().g.kind == NITRO_CONV3X3) {
        const LayerGeom& lg = b->L.back().g;
        int kh, kw;
        lr_window(lg.cout, lg.oh, lg.ow, desc->d_lr, &kh, &kw);
        if (kh * kw > 1) {
            b->lp = LrPoolGeom{kh, kw, lg.oh / kh, lg.ow / kw};
            b->d = (int64_t)b->lp.ph * b->lp.pw * lg.cout;
            ok = ok && dalloc(b, &b->zmp, (size_t)MB * b->d) && dalloc(b, &b->lr_am, (size_t)MB * b->d);
        }
    }
    ok = ok && dalloc(b, &b->Wlr, (size_t)b->G * b->d) && dalloc(b, &b->dWlr, (size_t)b->G * b->d) &&
         dalloc(b, &b->grad_l, (size_t)MB * b->G) && dalloc(b, &b->zsum, simt_learn_scratch(MB, (int)b->d, b->G)) && dalloc(b, &b->z64, z_need) &&
         dalloc(b, &b->words, n_words(desc->n_layers));
    if (ok) {
        b->sse = reinterpret_cast<unsigned long long*>(b->words + sse_word(desc->n_layers));
        void* h = nullptr;
        ok = cudaMallocHost(&h, sizeof(uint32_t) * n_words(desc->n_layers)) == cudaSuccess;
        if (ok) {
            b->host_allocs.push_back(h);
            b->words_host = static_cast<uint32_t*>(h);
        }
    }
    b->z64_elems = z_need;
    for (int i = 0; ok && i < desc->n_layers; ++i) {
        Layer& ly = b->L[i];
        ok = ly.lin_a ? tc_linear_init(ly.tc, ly.g, desc->max_batch, ly.lin_a, w_w(b, i), w_delta(b, i),
                                       b->allocs, b->host_allocs)
                      : tc_layer_init(ly.tc, ly.g, desc->max_batch, i > 0, w_w(b, i), w_delta(b, i),
                                      b->allocs, b->host_allocs);
        // one copy of all the block's words per step refreshes the layers' hints
        if (ok) tc_use_external_hints(ly.tc, b->words_host + 3 + i,
                                      b->words_host + 4 + desc->n_layers + i);
    }
    if (!ok) {
        free_all(b);
        delete b;
        return NITRO_ERR_CUDA;
    }
    std::vector<int32_t> wlr = draw_weights((int64_t)b->G * b->d, b->d, seed, kLearningTensorId);
    std::vector<uint32_t> words(n_words(desc->n_layers), 0);
    words[2] = host_maxabs(wlr.data(), wlr.size());
    cudaError_t e = cudaSuccess;
    for (int i = 0; i < desc->n_layers && e == cudaSuccess; ++i) {
        words[3 + i] = host_maxabs(host_w[i].data(), host_w[i].size());
        e = cudaMemcpyAsync(b->L[i].W, host_w[i].data(), host_w[i].size() * 4, cudaMemcpyHostToDevice, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(b->L[i].dW, 0, (size_t)b->L[i].wcount * 8, s);
    }
    if (e == cudaSuccess) e = cudaMemcpyAsync(b->Wlr, wlr.data(), wlr.size() * 4, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(b->dWlr, 0, (size_t)b->G * b->d * 8, s);
    if (e == cudaSuccess) e = cudaMemcpyAsync(b->words, words.data(), words.size() * 4, cudaMemcpyHostToDevice, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(b->sse, 0, 8, s);
    if (e == cudaSuccess)
        e = cudaMemsetAsync(b->zsum, 0, 8 * simt_learn_scratch(MB, (int)b->d, b->G), s);
    for (int i = 0; e == cudaSuccess && i < desc->n_layers; ++i) {
        e = tc_refresh_weights(b->L[i].tc, b->L[i].g, b->L[i].W, w_w(b, i), s);
        if (e == cudaSuccess && b->L[i].lin_planes)
            e = tc_pack_limbs(b->L[i].W, b->L[i].wcount, w_w(b, i), b->L[i].lin_planes, s);
    }
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess) std::memcpy(b->words_host, words.data(), words.size() * 4);
    if (e != cudaSuccess) {
        free_all(b);
        delete b;
        return NITRO_ERR_CUDA;
    }
    *out = b;
    return NITRO_OK;
}

void nitro_destroy_block(nitro_block* b) {
    if (!b) return;
    cudaDeviceSynchronize();
    free_all(b);
    delete b;
}

nitro_status nitro_block_forward(nitro_block* b, const int8_t* a_in, int batch, int8_t* a_out,
                                 void* stream) {
    if (!b || batch < 0 || batch > b->desc.max_batch) return NITRO_ERR_ARG;
    if (batch > 0 && !a_in) return NITRO_ERR_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    b->batch = batch;
    if (batch == 0) return NITRO_OK;
    const int n = (int)b->L.size();
    const int8_t* x = a_in;
    bool nhwc_done = false;
    for (int i = 0; i < n; ++i) {
        Layer& ly = b->L[i];
        const LayerGeom& g = ly.g;
        // the fused epilogues store 16 bytes at a time: an unaligned a_out
        // is filled by a copy after the last layer instead
        int8_t* out2 = (i == n - 1 && ((uintptr_t)a_out & 15) == 0) ? a_out : nullptr;
        bool done = false, fused = false;
        NITRO_TRY(tc_pack_input(ly.tc, g, x, batch, nhwc_done, s));
        // the epilogue also writes the next layer's bf16 forward operand
        uint16_t* next_nhwc = nullptr;
        if (i + 1 < n && b->L[i + 1].tc.act_nhwc && !b->L[i + 1].tc.im2col &&
            b->L[i + 1].tc.cin8 == g.cout)
            next_nhwc = b->L[i + 1].tc.act_nhwc;
        TcFwdOut fo{b->desc.alpha_inv, b->mu, ly.act, out2, ly.region, ly.argmax, next_nhwc};
        NITRO_TRY(tc_conv_forward(ly.tc, g, batch, b->z64, &fo, w_status(b), s, &done, &fused));
        if (ly.lin_planes) {
            // linear: z = a W^T on the tcgen05 GEMM (weight planes kept by IntegerSGD)
            NITRO_TRY(tc_pack_int8(x, batch, g.cin, ly.lin_a, s));
            NITRO_TRY(tc_gemm_run(ly.lin_a, ly.lin_planes, batch, g.cout, g.cin, w_w(b, i), b->z64,
                                  w_status(b), s));
            done = true;
        }
        if (!done && simt_small_conv_ok(g)) {
            // narrow input (image channels): fused CUDA-core forward
            NITRO_TRY(simt_conv_small_fwd(x, ly.W, g, batch, b->desc.alpha_inv, b->mu, ly.act, out2,
                                          ly.region, ly.argmax, next_nhwc, s));
            done = fused = true;
        }
        if (!done) {
            const int mode = g.kind == NITRO_CONV3X3 ? GM_CONV_FWD : GM_LIN_FWD;
            NITRO_TRY(simt_gemm(mode, x, nullptr, ly.W, b->z64, batch, g.h, g.w, g.cin, g.cout, s));
        }
        if (!fused) {
            // dropout of the linear layers (App. B, p_l)
            DropoutArgs da{b->seed, (uint32_t)b->desc.dropout_p16, i, w_step(b)};
            const bool drop = g.kind == NITRO_LINEAR && b->desc.dropout_p16 > 0;
            NITRO_TRY(simt_fwd_epilogue(b->z64, g, batch, b->desc.alpha_inv, b->mu, ly.act, out2,
                                        ly.region, ly.argmax, s, drop ? &da : nullptr));
        }
        nhwc_done = fused && next_nhwc != nullptr;
        x = ly.act;
    }
    if (n > 0 && a_out && ((uintptr_t)a_out & 15) != 0)
        NITRO_TRY(cudaMemcpyAsync(a_out, b->L[n - 1].act, (size_t)batch * b->d,
                                  cudaMemcpyDeviceToDevice, s));
    return NITRO_OK;
}

}  // extern "C"

namespace {

// The block's backward (Sec. 3.3, second phase).  With `updated` != null the
// layers whose weight gradient runs on tcgen05 also apply IntegerSGD inside
// that kernel (their input gradient, which needs the pre-update weights, runs
// first) and are marked in *updated; the caller updates the rest.
nitro_status block_backward(nitro_block* b, const int8_t* a_in, const int32_t* labels, int batch,
                            int64_t* loss_dev, void* stream, std::vector<char>* updated) {
    if (!b || batch < 0 || batch != b->batch) return NITRO_ERR_ARG;
    if (updated) updated->assign(b->L.size(), 0);
    if (batch > 0 && (!labels || !a_in)) return NITRO_ERR_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    const int n = (int)b->L.size();
    const int G = b->G;
    const int64_t d = b->d;
    // reset the per-step range words and the SSE (one contiguous range)
    NITRO_TRY(cudaMemsetAsync(w_gl(b), 0, 4 * (size_t)(n_words(n) - (3 + n)), s));
    if (batch == 0) {
        NITRO_TRY(cudaMemsetAsync(b->dWlr, 0, (size_t)G * d * 8, s));
        for (int i = 0; i < n; ++i) NITRO_TRY(cudaMemsetAsync(b->L[i].dW, 0, (size_t)b->L[i].wcount * 8, s));
        if (loss_dev) NITRO_TRY(cudaMemsetAsync(loss_dev, 0, 8, s));
        return NITRO_OK;
    }
    const int8_t* a_last = n ? b->L[n - 1].act : a_in;
    if (b->zmp) {
        // z^mp: the block output max-pooled for the learning layer (Sec. 3.3)
        const LayerGeom& lg = b->L[n - 1].g;
        NITRO_TRY(simt_lr_pool_fwd(a_last, batch, lg.oh, lg.ow, lg.cout, b->lp.kh, b->lp.kw,
                                   b->lp.ph, b->lp.pw, b->zmp, b->lr_am, s));
        a_last = b->zmp;
    }
    NITRO_TRY(simt_learn_fwd(a_last, b->Wlr, labels, batch, (int)d, G, b->zsum, b->grad_l, b->sse,
                             loss_dev, w_gl(b), w_status(b), s));
    if (b->zmp) {
        // learning-weight gradient from z^mp, then delta_fw back through the
        // learning pool into the last layer's delta (pre-update W_lr)
        if (simt_lr_backward_ok(G))
            NITRO_TRY(simt_lr_backward(a_last, b->grad_l, b->Wlr, batch, G, (int)d, nullptr,
                                       b->desc.alpha_inv, nullptr, nullptr, nullptr, b->dWlr,
                                       w_gl(b), w_wlr(b), nullptr, w_status(b), s));
        else
            NITRO_TRY(simt_learn_dw(a_last, b->grad_l, batch, (int)d, G, b->dWlr, s));
        Layer& ly = b->L[n - 1];
        NITRO_TRY(simt_lrpool_to_delta(b->grad_l, b->Wlr, G, (int)d, ly.g, b->lp, batch, b->lr_am,
                                       ly.argmax, ly.region, b->desc.alpha_inv, ly.delta, w_gl(b),
                                       w_wlr(b), w_delta(b, n - 1), w_status(b), s));
    } else if (simt_lr_backward_ok(G)) {
        // learning-weight gradient and (below a forward layer) delta_fw -> that
        // layer's delta in one pass
        Layer* ly = n ? &b->L[n - 1] : nullptr;
        NITRO_TRY(simt_lr_backward(a_last, b->grad_l, b->Wlr, batch, G, (int)d, ly ? &ly->g : nullptr,
                                   b->desc.alpha_inv, ly ? ly->region : nullptr,
                                   ly ? ly->argmax : nullptr, ly ? ly->delta : nullptr, b->dWlr,
                                   w_gl(b), w_wlr(b), n ? w_delta(b, n - 1) : nullptr, w_status(b), s));
    } else {
        NITRO_TRY(simt_learn_dw(a_last, b->grad_l, batch, (int)d, G, b->dWlr, s));
    }
    if (n == 0) return NITRO_OK;
    // delta_fw = grad_L W_lr (pre-update), into the last layer
    if (!b->zmp && !simt_lr_backward_ok(G)) {
        Layer& ly = b->L[n - 1];
        DeltaSrc src{};
        src.grad_l = b->grad_l; src.wlr = b->Wlr; src.G = G;
        src.maxabs_a = w_gl(b); src.maxabs_b = w_wlr(b); src.bound_k = G;
        NITRO_TRY(simt_grad_to_delta(src, ly.g, batch, b->desc.alpha_inv, ly.region, ly.argmax,
                                     ly.delta, w_delta(b, n - 1), w_status(b), s));
    }
    const int64_t gamma_fw = 64LL * b->G * b->desc.gamma_inv_lr;
    for (int i = n - 1; i >= 0; --i) {
        Layer& ly = b->L[i];
        const LayerGeom& g = ly.g;
        const int8_t* x = i ? b->L[i - 1].act : a_in;
        bool done = false;
        // fused update: the input gradient reads the pre-update weights, so it
        // runs first (after the delta split), then the weight gradient with
        // IntegerSGD; otherwise weight gradient first, as the split requires
        const bool fuse_sgd = updated && tc_wgrad_fusable(ly.tc, g, batch);
        auto wgrad = [&]() -> nitro_status {
            if (fuse_sgd) {
                NITRO_TRY(cudaMemsetAsync(w_w(b, i), 0, 4, s));
                TcSgd sg{gamma_fw, b->desc.eta_inv_fw, b->desc.sgd_round == NITRO_ROUND_TRUNC, ly.W,
                         w_w(b, i), nullptr, 0, 0, 0};
                if (ly.lin_planes) {
                    // linear weight planes [4][out][in]
                    sg.planes = ly.lin_planes;
                    sg.plane = ly.wcount;
                    sg.row_k = g.cin;
                } else {
                    tc_weight_planes(ly.tc, g, &sg.planes, &sg.plane, &sg.row_k, &sg.tap_k);
                }
                bool sgd_done = false;
                NITRO_TRY(tc_conv_wgrad(ly.tc, g, ly.delta, w_delta(b, i), batch, ly.dW, w_status(b), s,
                                        &done, true, &sg, &sgd_done));
                (*updated)[i] = done && sgd_done;

            } else {
                NITRO_TRY(tc_conv_wgrad(ly.tc, g, ly.delta, w_delta(b, i), batch, ly.dW, w_status(b), s,
                                        &done));
            }
            if (!done && simt_small_conv_ok(g)) {
                NITRO_TRY(simt_conv_small_wgrad(x, ly.delta, g, batch, ly.dW, s));
                done = true;
            }
            if (!done) {
                const int mode = g.kind == NITRO_CONV3X3 ? GM_CONV_WGRAD : GM_LIN_WGRAD;
                NITRO_TRY(simt_gemm(mode, x, ly.delta, nullptr, ly.dW, batch, g.h, g.w, g.cin, g.cout, s));
            }
            return NITRO_OK;
        };
        if (fuse_sgd) {
            NITRO_TRY(tc_pack_delta(ly.tc, g, ly.delta, w_delta(b, i), batch, s));
        } else {
            nitro_status st = wgrad();
            if (st != NITRO_OK) return st;
        }
        if (i == 0) {
            if (fuse_sgd) {
                nitro_status st = wgrad();
                if (st != NITRO_OK) return st;
            }
            break;
        }
        done = false;
        bool fused = false;
        Layer& lo = b->L[i - 1];
        TcDgradOut fo{b->desc.alpha_inv, w_delta(b, i), w_w(b, i), lo.g.h, lo.g.w, lo.g.pool,
                      lo.region, lo.argmax, lo.delta, w_delta(b, i - 1)};
        // the fused epilogue needs the lower layer to be a conv on the same grid
        const bool can_fuse = lo.g.kind == NITRO_CONV3X3 && lo.g.oh == g.h && lo.g.ow == g.w;
        NITRO_TRY(tc_conv_dgrad(ly.tc, g, batch, b->z64, can_fuse ? &fo : nullptr, w_status(b), s,
                                &done, &fused));
        if (!done) {
            const int mode = g.kind == NITRO_CONV3X3 ? GM_CONV_DGRAD : GM_LIN_DGRAD;
            NITRO_TRY(simt_gemm(mode, nullptr, ly.delta, ly.W, b->z64, batch, g.h, g.w, g.cin, g.cout, s));
        }
        if (!fused) {
            DeltaSrc src{};
            src.g64 = b->z64;
            src.maxabs_a = w_delta(b, i); src.maxabs_b = w_w(b, i);
            src.bound_k = g.kind == NITRO_CONV3X3 ? 9LL * g.cout : (int64_t)g.cout;
            NITRO_TRY(simt_grad_to_delta(src, lo.g, batch, b->desc.alpha_inv, lo.region, lo.argmax,
                                         lo.delta, w_delta(b, i - 1), w_status(b), s));
        }
        if (fuse_sgd) {
            nitro_status st = wgrad();
            if (st != NITRO_OK) return st;
        }
    }
    return NITRO_OK;
}

// IntegerSGD of every tensor of the block not yet updated (skip[i] marks a
// forward layer updated inside its weight-gradient kernel).
nitro_status block_sgd(nitro_block* b, void* stream, const std::vector<char>* skip) {
    if (!b) return NITRO_ERR_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    const int n = (int)b->L.size();
    // gamma_inv^fw = AF * gamma_inv^lr, AF = 2^6 * G (Sec. 3.3.5)
    const int64_t gamma_fw = 64LL * b->G * b->desc.gamma_inv_lr;
    SgdBatch bt{};
    bt.round_trunc = b->desc.sgd_round == NITRO_ROUND_TRUNC;
    bt.status = w_status(b);
    bt.step = w_step(b);
    for (int i = 0; i < n; ++i) {
        if (skip && (*skip)[i]) continue;
        // the update also writes the tensor-core weight planes of the layer
        SgdTensor st{b->L[i].W, b->L[i].dW, b->L[i].wcount, gamma_fw, b->desc.eta_inv_fw,
                     w_w(b, i), {}, {}, nullptr, 0, 0, 0, 0, {}};
        tc_weight_planes(b->L[i].tc, b->L[i].g, &st.planes, &st.plane, &st.row_k, &st.tap_k);
        st.cin = b->L[i].g.cin;
        if (b->L[i].lin_planes) {
            // linear planes [4][out][in]: element o*in + k at row o*9*in + tap*in with
            // the update's (row, tap) = (o / 9, o % 9) decomposition
            st.planes = b->L[i].lin_planes;
            st.plane = b->L[i].wcount;
            st.row_k = 9 * b->L[i].g.cin;
            st.tap_k = b->L[i].g.cin;
        }
        if (skip) NITRO_TRY(cudaMemsetAsync(w_w(b, i), 0, 4, s));
        bt.t[bt.count++] = st;
    }
    bt.t[bt.count++] = SgdTensor{b->Wlr, b->dWlr, (int64_t)b->G * b->d, b->desc.gamma_inv_lr,
                                 b->desc.eta_inv_lr, w_wlr(b), {}, {}, nullptr, 0, 0, 0, 0, {}};
    // max |W_lr| and every updated layer's max |W| start from zero: one range
    // unless some layers were updated in their weight-gradient kernels
    NITRO_TRY(cudaMemsetAsync(w_wlr(b), 0, 4 * (size_t)(skip ? 1 : 1 + n), s));
    NITRO_TRY(simt_integersgd(bt, s));
    // the kernel-variant hints of the next step: one copy of all the words
    NITRO_TRY(cudaMemcpyAsync(b->words_host, b->words, 4 * (size_t)n_words(n), cudaMemcpyDeviceToHost, s));
    return NITRO_OK;
}

}  // namespace

extern "C" {

nitro_status nitro_block_backward(nitro_block* b, const int8_t* a_in, const int32_t* labels,
                                  int batch, int64_t* loss_dev, void* stream) {
    return block_backward(b, a_in, labels, batch, loss_dev, stream, nullptr);
}

nitro_status nitro_block_backward_update(nitro_block* b, const int8_t* a_in, const int32_t* labels,
                                         int batch, int64_t* loss_dev, void* stream) {
    std::vector<char> updated;
    nitro_status st = block_backward(b, a_in, labels, batch, loss_dev, stream, &updated);
    if (st != NITRO_OK) return st;
    return block_sgd(b, stream, &updated);
}

nitro_status nitro_block_set_hyper(nitro_block* b, int64_t gamma_inv_lr, int64_t eta_inv_fw,
                                   int64_t eta_inv_lr) {
    if (!b) return NITRO_ERR_ARG;
    nitro_block_desc d = b->desc;
    d.gamma_inv_lr = gamma_inv_lr;
    d.eta_inv_fw = eta_inv_fw;
    d.eta_inv_lr = eta_inv_lr;
    if (d.gamma_inv_lr < 1 || d.gamma_inv_lr > ((int64_t)1 << 48) || d.eta_inv_fw < 0 ||
        d.eta_inv_lr < 0)
        return NITRO_ERR_ARG;
    b->desc = d;
    return NITRO_OK;
}

nitro_status nitro_block_set_dropout(nitro_block* b, int dropout_p16) {
    if (!b || dropout_p16 < 0 || dropout_p16 > 65536) return NITRO_ERR_ARG;
    b->desc.dropout_p16 = dropout_p16;
    return NITRO_OK;
}

nitro_status nitro_integersgd_step(nitro_block* b, void* stream) {
    return block_sgd(b, stream, nullptr);
}

nitro_status nitro_block_diag_timeout(nitro_block* b, int wait_us, void* stream) {
    if (!b || wait_us < 1 || wait_us > 2000000) return NITRO_ERR_ARG;
    NITRO_TRY(tc_timeout_probe(w_status(b), (uint64_t)wait_us * 1000ull, (cudaStream_t)stream));
    return NITRO_OK;
}

nitro_status nitro_block_tensor_bytes(const nitro_block* b, int which, int layer, size_t* bytes) {
    if (!b || !bytes) return NITRO_ERR_ARG;
    const int n = (int)b->L.size();
    const bool per_layer = which == NITRO_T_W || which == NITRO_T_DW || which == NITRO_T_ACT ||
                           which == NITRO_T_REGION || which == NITRO_T_ARGMAX || which == NITRO_T_DELTA;
    if (per_layer && (layer < 0 || layer >= n)) return NITRO_ERR_ARG;
    if (!per_layer && layer != 0) return NITRO_ERR_ARG;
    if ((which == NITRO_T_LR_IN || which == NITRO_T_LR_ARGMAX) && !b->zmp) return NITRO_ERR_ARG;
    const size_t B = (size_t)b->batch;
    switch (which) {
        case NITRO_T_W: *bytes = (size_t)b->L[layer].wcount * 4; break;
        case NITRO_T_DW: *bytes = (size_t)b->L[layer].wcount * 8; break;
        case NITRO_T_WLR: *bytes = (size_t)b->G * b->d * 4; break;
        case NITRO_T_DWLR: *bytes = (size_t)b->G * b->d * 8; break;
        case NITRO_T_ACT: *bytes = B * b->L[layer].out_f; break;
        case NITRO_T_REGION: *bytes = B * b->L[layer].pre_f; break;
        case NITRO_T_ARGMAX:
            if (!b->L[layer].g.pool) return NITRO_ERR_ARG;
            *bytes = B * b->L[layer].out_f;
            break;
        case NITRO_T_DELTA: *bytes = B * b->L[layer].pre_f * 4; break;
        case NITRO_T_GRAD_L: *bytes = B * b->G * 4; break;
        case NITRO_T_SSE: *bytes = 8; break;
        case NITRO_T_LR_IN:
        case NITRO_T_LR_ARGMAX: *bytes = B * b->d; break;
        case NITRO_T_STEP: *bytes = 4; break;
        default: return NITRO_ERR_ARG;
    }
    return NITRO_OK;
}

static const void* tensor_ptr(nitro_block* b, int which, int layer) {
    switch (which) {
        case NITRO_T_W: return b->L[layer].W;
        case NITRO_T_DW: return b->L[layer].dW;
        case NITRO_T_WLR: return b->Wlr;
        case NITRO_T_DWLR: return b->dWlr;
        case NITRO_T_ACT: return b->L[layer].act;
        case NITRO_T_REGION: return b->L[layer].region;
        case NITRO_T_ARGMAX: return b->L[layer].argmax;
        case NITRO_T_DELTA: return b->L[layer].delta;
        case NITRO_T_GRAD_L: return b->grad_l;
        case NITRO_T_SSE: return b->sse;
        case NITRO_T_LR_IN: return b->zmp;
        case NITRO_T_LR_ARGMAX: return b->lr_am;
        case NITRO_T_STEP: return w_step(b);
    }
    return nullptr;
}

nitro_status nitro_block_grad_device(nitro_block* b, int which, int layer, void** dev_ptr,
                                     size_t* bytes) {
    if (!b || !dev_ptr) return NITRO_ERR_ARG;
    *dev_ptr = nullptr;
    if (which != NITRO_T_DW && which != NITRO_T_DWLR) return NITRO_ERR_ARG;
    size_t need = 0;
    nitro_status st = nitro_block_tensor_bytes(b, which, layer, &need);
    if (st != NITRO_OK) return st;
    *dev_ptr = const_cast<void*>(tensor_ptr(b, which, layer));
    if (bytes) *bytes = need;
    return NITRO_OK;
}

static nitro_status latched(uint32_t bits) {
    if (bits & ST_TIMEOUT) return NITRO_ERR_TIMEOUT;
    if (bits & ST_OVERFLOW) return NITRO_ERR_OVERFLOW;
    if (bits & ST_BAD_LABEL) return NITRO_ERR_ARG;
    return NITRO_OK;
}

uint32_t nitro_block_status_bits(nitro_block* b) {
    if (!b) return 0;
    uint32_t bits = 0;
    if (cudaDeviceSynchronize() != cudaSuccess) return 0xffffffffu;
    if (cudaMemcpy(&bits, b->words, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return 0xffffffffu;
    return bits;
}

nitro_status nitro_block_status(nitro_block* b, int clear) {
    if (!b) return NITRO_ERR_ARG;
    const uint32_t bits = nitro_block_status_bits(b);
    if (bits == 0xffffffffu) return NITRO_ERR_CUDA;
    if (clear && cudaMemset(b->words, 0, 4) != cudaSuccess) return NITRO_ERR_CUDA;
    if (clear && cudaDeviceSynchronize() != cudaSuccess) return NITRO_ERR_CUDA;
    return latched(bits);
}

nitro_status nitro_block_get_tensor(nitro_block* b, int which, int layer, void* host_dst,
                                    size_t bytes) {
    size_t need = 0;
    nitro_status st = nitro_block_tensor_bytes(b, which, layer, &need);
    if (st != NITRO_OK) return st;
    if (bytes != need || (need && !host_dst)) return NITRO_ERR_ARG;
    if (cudaDeviceSynchronize() != cudaSuccess) return NITRO_ERR_CUDA;
    if (need && cudaMemcpy(host_dst, tensor_ptr(b, which, layer), need, cudaMemcpyDeviceToHost) != cudaSuccess)
        return NITRO_ERR_CUDA;
    uint32_t bits = 0;
    if (cudaMemcpy(&bits, b->words, 4, cudaMemcpyDeviceToHost) != cudaSuccess) return NITRO_ERR_CUDA;
    return latched(bits);
}

nitro_status nitro_block_set_tensor(nitro_block* b, int which, int layer, const void* host_src,
                                    size_t bytes) {
    if (which != NITRO_T_W && which != NITRO_T_DW && which != NITRO_T_WLR && which != NITRO_T_DWLR &&
        which != NITRO_T_STEP)
        return NITRO_ERR_ARG;
    size_t need = 0;
    nitro_status st = nitro_block_tensor_bytes(b, which, layer, &need);
    if (st != NITRO_OK) return st;
    if (bytes != need || !host_src) return NITRO_ERR_ARG;
    if (cudaDeviceSynchronize() != cudaSuccess) return NITRO_ERR_CUDA;
    if (cudaMemcpy((void*)tensor_ptr(b, which, layer), host_src, need, cudaMemcpyHostToDevice) != cudaSuccess)
        return NITRO_ERR_CUDA;
    if (which == NITRO_T_W || which == NITRO_T_WLR) {
        const uint32_t m = host_maxabs(static_cast<const int32_t*>(host_src), need / 4);
        uint32_t* word = which == NITRO_T_W ? w_w(b, layer) : w_wlr(b);
        if (cudaMemcpy(word, &m, 4, cudaMemcpyHostToDevice) != cudaSuccess) return NITRO_ERR_CUDA;
        if (which == NITRO_T_W &&
            tc_refresh_weights(b->L[layer].tc, b->L[layer].g, b->L[layer].W, word, 0) != cudaSuccess)
            return NITRO_ERR_CUDA;
        if (which == NITRO_T_W && b->L[layer].lin_planes &&
            tc_pack_limbs(b->L[layer].W, b->L[layer].wcount, word, b->L[layer].lin_planes, 0) !=
                cudaSuccess)
            return NITRO_ERR_CUDA;
    }
    if (cudaDeviceSynchronize() != cudaSuccess) return NITRO_ERR_CUDA;
    // the kernel-variant hints follow the new weights
    if (cudaMemcpy(b->words_host, b->words, 4 * (size_t)n_words((int)b->L.size()), cudaMemcpyDeviceToHost) !=
        cudaSuccess)
        return NITRO_ERR_CUDA;
    return NITRO_OK;
}

}  // extern "C"
