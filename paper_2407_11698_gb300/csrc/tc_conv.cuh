// Tensor-core (tcgen05) path of the conv contractions: state kept per layer
// and per block, and the entry points the ABI calls.  Each entry point sets
// *done = false when it does not take the layer, and the caller then runs the
// CUDA-core kernels.
#pragma once

#include <vector>

#include "nitro_internal.cuh"

namespace nitro {

struct TcLayer {
    bool fwd = false, wgrad = false, dgrad = false;   // which passes run on tcgen05
};

struct TcWorkspace {
    int max_batch = 0;
};

bool tc_block_init(TcWorkspace& ws, std::vector<void*>& allocs, int max_batch);
bool tc_layer_init(TcLayer& t, const LayerGeom& g, int max_batch, TcWorkspace& ws,
                   std::vector<void*>& allocs);
cudaError_t tc_refresh_weights(TcLayer& t, const LayerGeom& g, const int32_t* W,
                               const uint32_t* maxabs_w, cudaStream_t s);
cudaError_t tc_conv_forward(TcLayer& t, const LayerGeom& g, const int8_t* x, int batch,
                            int alpha_inv, int mu, int8_t* act, int8_t* out2, int8_t* region,
                            int8_t* argmax, TcWorkspace& ws, cudaStream_t s, bool* done);
cudaError_t tc_conv_wgrad(TcLayer& t, const LayerGeom& g, const int8_t* x, const int32_t* delta,
                          const uint32_t* maxabs_delta, int batch, int64_t* dW, TcWorkspace& ws,
                          cudaStream_t s, bool* done);
cudaError_t tc_conv_dgrad(TcLayer& t, const LayerGeom& g, const int32_t* delta,
                          const uint32_t* maxabs_delta, int batch, int64_t* g64, TcWorkspace& ws,
                          cudaStream_t s, bool* done);

}  // namespace nitro
