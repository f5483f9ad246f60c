// Tensor-core conv path (tcgen05).  Not yet enabled: every entry declines.
#include "tc_conv.cuh"

namespace nitro {

bool tc_block_init(TcWorkspace& ws, std::vector<void*>&, int max_batch) {
    ws.max_batch = max_batch;
    return true;
}
bool tc_layer_init(TcLayer&, const LayerGeom&, int, TcWorkspace&, std::vector<void*>&) { return true; }
cudaError_t tc_refresh_weights(TcLayer&, const LayerGeom&, const int32_t*, const uint32_t*, cudaStream_t) {
    return cudaSuccess;
}
cudaError_t tc_conv_forward(TcLayer&, const LayerGeom&, const int8_t*, int, int, int, int8_t*, int8_t*,
                            int8_t*, int8_t*, TcWorkspace&, cudaStream_t, bool* done) {
    *done = false;
    return cudaSuccess;
}
cudaError_t tc_conv_wgrad(TcLayer&, const LayerGeom&, const int8_t*, const int32_t*, const uint32_t*,
                          int, int64_t*, TcWorkspace&, cudaStream_t, bool* done) {
    *done = false;
    return cudaSuccess;
}
cudaError_t tc_conv_dgrad(TcLayer&, const LayerGeom&, const int32_t*, const uint32_t*, int, int64_t*,
                          TcWorkspace&, cudaStream_t, bool* done) {
    *done = false;
    return cudaSuccess;
}

}  // namespace nitro
