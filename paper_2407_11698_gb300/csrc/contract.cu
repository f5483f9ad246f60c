// Kernel-level entry points: one 3x3 conv contraction (forward, weight
// gradient or input gradient) or one integer GEMM, on caller buffers, through
// the same limb packing and tcgen05 kernels the block step uses (CUDA-core
// kernels where the tensor-core path does not apply).  Results are the exact
// int64 sums, modulo 2^64.
#include <new>
#include <vector>

#include "nitro_internal.cuh"
#include "tc_conv.cuh"

using namespace nitro;

struct nitro_conv {
    LayerGeom g{};
    TcLayer t;
    int max_batch = 0;
    uint32_t* words = nullptr;   // [0] max|W| [1] max|delta| [2] status
    std::vector<void*> allocs;
    std::vector<void*> host_allocs;
};

struct nitro_gemm {
    int max_m = 0, max_n = 0, max_k = 0;
    uint16_t* a = nullptr;       // bf16 [M][K]
    uint16_t* b = nullptr;       // bf16 limb planes [4][N][K]
    uint32_t* words = nullptr;   // [0] max|B| [1] status
    std::vector<void*> allocs;
};

namespace {

template <typename T>
bool dalloc(std::vector<void*>& allocs, T** p, size_t count) {
    void* q = nullptr;
    if (cudaMalloc(&q, (count ? count : 1) * sizeof(T)) != cudaSuccess) return false;
    allocs.push_back(q);
    *p = static_cast<T*>(q);
    return true;
}

void free_all(std::vector<void*>& allocs) {
    for (void* p : allocs) cudaFree(p);
    allocs.clear();
}

void free_host(std::vector<void*>& allocs) {
    for (void* p : allocs) cudaFreeHost(p);
    allocs.clear();
}

nitro_status latched(uint32_t bits) {
    if (bits & ST_TIMEOUT) return NITRO_ERR_TIMEOUT;
    if (bits & ST_OVERFLOW) return NITRO_ERR_OVERFLOW;
    return NITRO_OK;
}

#define TRY(expr)                                      \
    do {                                               \
        if ((expr) != cudaSuccess) return NITRO_ERR_CUDA; \
    } while (0)

}  // namespace

extern "C" {

nitro_status nitro_conv3x3_create(int max_batch, int h, int w, int cin, int cout,
                                  nitro_conv** out) {
    if (!out) return NITRO_ERR_ARG;
    *out = nullptr;
    if (max_batch < 1 || h < 1 || w < 1 || cin < 1 || cout < 1 || cin > (1 << 16) ||
        cout > (1 << 16) || (int64_t)max_batch * h * w > ((int64_t)1 << 24) ||
        (int64_t)max_batch * h * w * (cin > cout ? cin : cout) >= ((int64_t)1 << 31))
        return NITRO_ERR_ARG;
    nitro_conv* c = new (std::nothrow) nitro_conv();
    if (!c) return NITRO_ERR_CUDA;
    c->g = LayerGeom{NITRO_CONV3X3, cin, cout, h, w, 0, h, w};
    c->max_batch = max_batch;
    bool ok = dalloc(c->allocs, &c->words, 4) &&
              tc_layer_init(c->t, c->g, max_batch, true, c->words, c->words + 1, c->allocs,
                            c->host_allocs);
    if (ok) ok = cudaMemset(c->words, 0, 16) == cudaSuccess;
    if (!ok) {
        free_all(c->allocs);
        free_host(c->host_allocs);
        delete c;
        return NITRO_ERR_CUDA;
    }
    *out = c;
    return NITRO_OK;
}

nitro_status nitro_conv3x3_contract(nitro_conv* c, int mode, const void* x, const int32_t* y,
                                    int batch, int64_t* out, void* stream) {
    if (!c || batch < 0 || batch > c->max_batch) return NITRO_ERR_ARG;
    if (mode != NITRO_CONTRACT_FWD && mode != NITRO_CONTRACT_WGRAD && mode != NITRO_CONTRACT_DGRAD)
        return NITRO_ERR_ARG;
    if (batch > 0 && (!x || !y || !out)) return NITRO_ERR_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    const LayerGeom& g = c->g;
    uint32_t* status = c->words + 2;
    if (batch == 0) {
        if (mode == NITRO_CONTRACT_WGRAD)
            TRY(cudaMemsetAsync(out, 0, sizeof(int64_t) * 9 * g.cin * g.cout, s));
        return NITRO_OK;
    }
    bool done = false, fused = false;
    if (mode == NITRO_CONTRACT_FWD) {
        const int8_t* a = static_cast<const int8_t*>(x);
        TRY(tc_maxabs(y, (int64_t)g.cout * 9 * g.cin, c->words, s));
        TRY(tc_refresh_weights(c->t, g, y, c->words, s));
        TRY(tc_pack_input(c->t, g, a, batch, false, s));
        TRY(tc_conv_forward(c->t, g, batch, out, nullptr, status, s, &done, &fused));
        if (!done) TRY(simt_gemm(GM_CONV_FWD, a, nullptr, y, out, batch, g.h, g.w, g.cin, g.cout, s));
    } else if (mode == NITRO_CONTRACT_WGRAD) {
        const int8_t* a = static_cast<const int8_t*>(x);
        TRY(tc_pack_input(c->t, g, a, batch, false, s));
        TRY(tc_maxabs(y, (int64_t)batch * g.h * g.w * g.cout, c->words + 1, s));
        TRY(tc_conv_wgrad(c->t, g, y, c->words + 1, batch, out, status, s, &done));
        if (!done) TRY(simt_gemm(GM_CONV_WGRAD, a, y, nullptr, out, batch, g.h, g.w, g.cin, g.cout, s));
    } else {
        const int32_t* d = static_cast<const int32_t*>(x);
        TRY(tc_maxabs(y, (int64_t)g.cout * 9 * g.cin, c->words, s));
        TRY(tc_refresh_weights(c->t, g, y, c->words, s));
        TRY(tc_maxabs(d, (int64_t)batch * g.h * g.w * g.cout, c->words + 1, s));
        TRY(tc_pack_delta(c->t, g, d, c->words + 1, batch, s));
        TRY(tc_conv_dgrad(c->t, g, batch, out, nullptr, status, s, &done, &fused));
        if (!done) TRY(simt_gemm(GM_CONV_DGRAD, nullptr, d, y, out, batch, g.h, g.w, g.cin, g.cout, s));
    }
    return NITRO_OK;
}

nitro_status nitro_conv3x3_status(nitro_conv* c) {
    if (!c) return NITRO_ERR_ARG;
    uint32_t bits = 0;
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(&bits, c->words + 2, 4, cudaMemcpyDeviceToHost) != cudaSuccess)
        return NITRO_ERR_CUDA;
    return latched(bits);
}

void nitro_conv3x3_destroy(nitro_conv* c) {
    if (!c) return;
    cudaDeviceSynchronize();
    free_all(c->allocs);
    free_host(c->host_allocs);
    delete c;
}

nitro_status nitro_gemm_create(int max_m, int max_n, int max_k, nitro_gemm** out) {
    if (!out) return NITRO_ERR_ARG;
    *out = nullptr;
    if (max_m < 1 || max_n < 1 || max_k < 1 || max_k > (1 << 20) || max_m > (1 << 24) ||
        max_n > (1 << 24) || (int64_t)max_m * max_k >= ((int64_t)1 << 34) ||
        (int64_t)max_n * max_k >= ((int64_t)1 << 34))
        return NITRO_ERR_ARG;
    nitro_gemm* g = new (std::nothrow) nitro_gemm();
    if (!g) return NITRO_ERR_CUDA;
    g->max_m = max_m;
    g->max_n = max_n;
    g->max_k = max_k;
    bool ok = dalloc(g->allocs, &g->a, (size_t)max_m * max_k) &&
              dalloc(g->allocs, &g->b, (size_t)kMaxLimbs * max_n * max_k) &&
              dalloc(g->allocs, &g->words, 2);
    if (ok) ok = cudaMemset(g->words, 0, 8) == cudaSuccess;
    if (!ok) {
        free_all(g->allocs);
        delete g;
        return NITRO_ERR_CUDA;
    }
    *out = g;
    return NITRO_OK;
}

nitro_status nitro_gemm_run(nitro_gemm* g, const int8_t* a, const int32_t* b, int m, int n, int k,
                            int64_t* c, void* stream) {
    if (!g || m < 0 || n < 0 || k < 0 || m > g->max_m || n > g->max_n || k > g->max_k)
        return NITRO_ERR_ARG;
    if (m == 0 || n == 0) return NITRO_OK;
    if (!a || !b || !c) return NITRO_ERR_ARG;
    cudaStream_t s = (cudaStream_t)stream;
    if (k == 0) {
        TRY(cudaMemsetAsync(c, 0, sizeof(int64_t) * (size_t)m * n, s));
        return NITRO_OK;
    }
    if (k % 8 != 0) {
        // TMA rows must be multiples of 16 bytes: CUDA-core kernel instead
        TRY(simt_gemm(GM_LIN_FWD, a, nullptr, b, c, m, 1, 1, k, n, s));
        return NITRO_OK;
    }
    TRY(tc_pack_int8(a, m, k, g->a, s));
    TRY(tc_maxabs(b, (int64_t)n * k, g->words, s));
    TRY(tc_pack_limbs(b, (int64_t)n * k, g->words, g->b, s));
    TRY(tc_gemm_run(g->a, g->b, m, n, k, g->words, c, g->words + 1, s));
    return NITRO_OK;
}

nitro_status nitro_gemm_status(nitro_gemm* g) {
    if (!g) return NITRO_ERR_ARG;
    uint32_t bits = 0;
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(&bits, g->words + 1, 4, cudaMemcpyDeviceToHost) != cudaSuccess)
        return NITRO_ERR_CUDA;
    return latched(bits);
}

void nitro_gemm_destroy(nitro_gemm* g) {
    if (!g) return;
    cudaDeviceSynchronize();
    free_all(g->allocs);
    delete g;
}

}  // extern "C"
