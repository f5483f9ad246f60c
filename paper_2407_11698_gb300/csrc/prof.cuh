// Launch accounting and optional per-kernel CUDA-event timing.
//
// Every kernel launch of the library goes through a ProfScope: it counts the
// launch, and when profiling is on it brackets the launch with a pair of CUDA
// events recorded on the launching stream, tagged with the kernel's class and
// its algorithmic work (integer ops = 2 x MACs, or HBM bytes).
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace nitro {

enum KernelId : int {
    K_SIMT_CONV_FWD = 0,
    K_SIMT_CONV_DGRAD,
    K_SIMT_CONV_WGRAD,
    K_SIMT_LIN_FWD,
    K_SIMT_LIN_DGRAD,
    K_SIMT_LIN_WGRAD,
    K_FWD_EPILOGUE,
    K_LEARN_FWD,
    K_LEARN_DW,
    K_GRAD_TO_DELTA,
    K_INTEGERSGD,
    K_FINISH_LOSS,
    K_TC_CONV_FWD,
    K_TC_CONV_WGRAD,
    K_TC_CONV_DGRAD,
    K_TC_PACK,
    K_TC_FINISH,
    K_TC_GEMM,
    K_LR_BACKWARD,
    K_TC_PACK_W,
    K_TC_PACK_X,
    K_TC_PACK_D,
    K_PREP_SUM,
    K_PREP_MAD,
    K_PREP_APPLY,
    K_LR_POOL,
    K_LRPOOL_TO_DELTA,
    K_TC_PROBE,
    K_TC_LIN_WGRAD,
    K_COUNT
};

const char* kernel_name(int id);

class ProfScope {
  public:
    // ops: algorithmic integer ops of this launch; bytes: algorithmic HBM bytes.
    ProfScope(int id, cudaStream_t s, double ops, double bytes);
    ~ProfScope();

  private:
    int slot_;
    cudaStream_t s_;
};

}  // namespace nitro
