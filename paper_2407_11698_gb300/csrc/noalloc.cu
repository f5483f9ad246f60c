// Forward of one 3x3 conv layer that performs no device allocation.
//
// Some callers cannot call cudaMalloc once they are running: code embedded in
// a host program that owns the whole device-memory budget (a serving process
// or game engine with its own arena), real-time loops where allocation after
// start-up is not allowed, and code that must not stall the device (cudaMalloc
// and cudaFree may synchronise it).  For them this entry point runs one conv
// layer's forward on the CUDA-core kernels that nitro_block_forward uses for
// layers off the tensor path (same results), but keeps the layer's int64
// pre-activations in a fixed array that is part of the library image instead
// of in a block's workspace.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds kNoallocScratchElems * 8 bytes (16 MiB) until the process
// exits.  Host code cannot use its name as a device address, so on the first
// call on each device the entry point looks the address up with
// cudaGetSymbolAddress (with that device current) and caches it for the life
// of the process; a cudaDeviceReset of that device is therefore not supported
// between calls.
#include <mutex>

#include "nitro_internal.cuh"

namespace {

constexpr int64_t kNoallocScratchElems = (int64_t)1 << 21;   // int64 values
constexpr int kMaxDevices = 64;

static __device__ __align__(256) int64_t g_noalloc_scratch[kNoallocScratchElems];

std::mutex g_mu;
int64_t* g_scratch_addr[kMaxDevices] = {};

// Device address of the scratch array for the current device, looked up once.
cudaError_t scratch_for_current_device(int64_t** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_scratch_addr[dev] = static_cast<int64_t*>(p);
    }
    *out = g_scratch_addr[dev];
    return cudaSuccess;
}

}  // namespace

using namespace nitro;

extern "C" nitro_status nitro_conv3x3_forward_noalloc(
    const int8_t* a_in, const int32_t* weights, int batch, int h, int w, int cin, int cout,
    int pool2x2, int alpha_inv, int8_t* a_out, int8_t* region, int8_t* argmax, void* stream) {
    if (batch < 0 || h < 1 || w < 1 || cin < 1 || cout < 1 || cin > (1 << 20) ||
        (pool2x2 != 0 && pool2x2 != 1) || alpha_inv < 2 || alpha_inv > (1 << 20))
        return NITRO_ERR_ARG;
    if (pool2x2 && (h < 2 || w < 2)) return NITRO_ERR_ARG;
    const int64_t elems = (int64_t)batch * h * w * cout;
    if (elems > kNoallocScratchElems) return NITRO_ERR_ARG;   // larger than the fixed array
    if (batch == 0) return NITRO_OK;
    if (!a_in || !weights || !a_out || !region || (pool2x2 && !argmax)) return NITRO_ERR_ARG;
    int64_t* z = nullptr;
    if (scratch_for_current_device(&z) != cudaSuccess) return NITRO_ERR_CUDA;
    cudaStream_t s = (cudaStream_t)stream;
    LayerGeom g{NITRO_CONV3X3, cin, cout, h, w, pool2x2, pool2x2 ? h / 2 : h, pool2x2 ? w / 2 : w};
    // mu_int8 of NITRO-ReLU: floor-average of the four segment means
    const int mu = (int)fdiv64(fdiv64(-127, alpha_inv) + fdiv64(-127, 2 * alpha_inv) + 63 + 127, 4);
    // The GEMM overwrites every element of z (directly, or by clearing it
    // before adding K-split partial sums), so the array needs no clearing here.
    if (simt_gemm(GM_CONV_FWD, a_in, nullptr, weights, z, batch, h, w, cin, cout, s) != cudaSuccess)
        return NITRO_ERR_CUDA;
    if (simt_fwd_epilogue(z, g, batch, alpha_inv, mu, a_out, nullptr, region, argmax, s) !=
        cudaSuccess)
        return NITRO_ERR_CUDA;
    return NITRO_OK;
}
