/*
 * nitro.h - C ABI of the GB300 library for the NITRO-D local-loss block
 * training step (arXiv 2407.11698, Sec. 3.2 architecture, Sec. 3.3 learning
 * algorithm).
 *
 * One handle = one integer local-loss block: its forward layers (3x3 conv or
 * linear, each followed by NITRO-Scaling, NITRO-ReLU and an optional 2x2
 * max-pool) and its learning layer (IntLinear to G classes + NITRO-Scaling,
 * trained on the RSS loss).  A block with zero forward layers is the network's
 * output block.  A network is a chain of handles; the caller runs every
 * block's forward, then every block's backward (they are independent, Sec.
 * 3.3), then every block's IntegerSGD step.  Handles share no state, so each
 * block may run on its own stream: block i+1's forward needs only block i's
 * output, and block i's backward and update may overlap the blocks after it.
 *
 * Conventions
 *   activations   int8, NHWC  a[((b*H + y)*W + x)*C + c]; linear: a[b*In + i]
 *   conv weights  int32, OHWI w[((co*3 + ky)*3 + kx)*Cin + ci]
 *   linear / learning weights int32 w[o*In + i]; learning input is the block
 *                 output flattened in (h, w, c) order
 *   weight gradients int64, same layout as the weights
 *   gradients delta and the loss gradient int32
 *   labels        int32 in [0, G)
 *   streams       `stream` is a cudaStream_t passed as void* (NULL = legacy
 *                 default stream)
 *
 * Ownership: the caller owns every pointer argument and the stream; device
 * pointers must stay valid until the work queued on `stream` has run.  The
 * library owns everything inside a handle (weights, weight gradients, cached
 * forward state, workspace), allocated once by nitro_init_block for
 * `max_batch` samples and freed by nitro_destroy_block.
 *
 * Errors: every call checks its arguments on the host and returns
 * NITRO_ERR_ARG / NITRO_ERR_UNSUPPORTED before queuing anything.  Compute
 * calls are asynchronous: conditions found on the device (a value that does
 * not fit its storage type, a label outside [0, G), a bounded wait that gave
 * up) are latched in a per-block device status word and reported by
 * nitro_block_status or nitro_block_get_tensor, which synchronise.  No
 * exception crosses the ABI and no call traps the device.
 */
#ifndef NITRO_H
#define NITRO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    NITRO_OK = 0,
    NITRO_ERR_ARG = 1,          /* bad argument, or a label outside [0, G) */
    NITRO_ERR_OVERFLOW = 2,     /* a value did not fit its storage type     */
    NITRO_ERR_TIMEOUT = 3,      /* a bounded device wait gave up            */
    NITRO_ERR_CUDA = 4,         /* a CUDA runtime call failed               */
    NITRO_ERR_UNSUPPORTED = 5   /* valid but not supported by the library   */
} nitro_status;

typedef enum { NITRO_ROUND_FLOOR = 0, NITRO_ROUND_TRUNC = 1 } nitro_round;
typedef enum { NITRO_CONV3X3 = 0, NITRO_LINEAR = 1 } nitro_layer_kind;

/* Bits of the device status word (nitro_block_status_bits). */
#define NITRO_STATUS_BIT_OVERFLOW  1u
#define NITRO_STATUS_BIT_BAD_LABEL 2u
#define NITRO_STATUS_BIT_TIMEOUT   4u

/* One forward layer (Sec. 3.2.1, Table 1): 3x3 conv with stride 1 and zero
 * padding 1, or linear; then NITRO-Scaling with SF = 2^8*9*cin (conv) or
 * 2^8*cin (linear), NITRO-ReLU, and a 2x2 stride-2 max-pool if pool2x2
 * (conv only; output size floor(h/2) x floor(w/2)).  h, w: input size
 * (1, 1 for linear).  A linear layer after a conv layer reads its input
 * flattened in (h, w, c) order, so cin = h'*w'*c of that output. */
typedef struct {
    int kind;        /* nitro_layer_kind */
    int cin, cout;
    int h, w;
    int pool2x2;
} nitro_layer_desc;

/* One local-loss block (Sec. 3.2, Sec. 3.3; hyper-parameters of App. B). */
typedef struct {
    int n_layers;                    /* 0 = output block                     */
    const nitro_layer_desc* layers;  /* n_layers entries, copied at init     */
    int in_features;                 /* flattened input size per sample      */
    int num_classes;                 /* G, 1..64                             */
    int alpha_inv;                   /* NITRO-ReLU 1/alpha, >= 2             */
    int64_t gamma_inv_lr;            /* learning / output layers; forward
                                        layers use AF*gamma_inv_lr with
                                        AF = 2^6*G (Sec. 3.3.5)              */
    int64_t eta_inv_fw, eta_inv_lr;  /* weight-decay thresholds, 0 = off     */
    int sgd_round;                   /* nitro_round for IntegerSGD           */
    int max_batch;                   /* workspace is sized for this          */
    int d_lr;                        /* learning-layer input size d^lr; 0 =
                                        no learning-layer pooling            */
    int dropout_p16;                 /* dropout rate of the linear forward
                                        layers, in units of 2^-16 (0..65536) */
} nitro_block_desc;

/* Learning-layer pooling (Sec. 3.3: the block output is downsampled by a
 * pooling layer to z^mp before the learning layers; App. B: d^lr input
 * features).  When d_lr > 0 and the last forward layer's output C x H' x W'
 * holds more than d_lr values, the learning layer reads a kh x kw max-pool
 * of it (stride (kh, kw), output floor(H'/kh) x floor(W'/kw) x C, first
 * maximum in row-major window order, position r*kw + s recorded).  The paper
 * states no rule for the window; this library takes: from 1 x 1, double kh,
 * then kw, alternately, while C*floor(H'/kh)*floor(W'/kw) > d_lr and the
 * window fits the map (a side that cannot double leaves the other to grow).
 * The learning layer then has d = C*floor(H'/kh)*floor(W'/kw) inputs (its
 * fan-in for the initialisation).  Windows above 256 positions return
 * NITRO_ERR_UNSUPPORTED.  Linear outputs (1 x 1) and output blocks never
 * pool.
 *
 * Dropout (App. B, rate p_l of the linear blocks).  With dropout_p16 > 0,
 * every nitro_block_forward drops outputs of the block's linear forward
 * layers: a dropped activation is stored as 0, its NITRO-ReLU region code
 * becomes 4, and it passes no gradient.  The paper gives no integer form of
 * dropout; no rescaling is applied.  Element e = b*out_features + j of forward
 * layer l is dropped at step t when the top 16 bits of output
 * 2^63 + t*2^35 + l*2^31 + e of SplitMix64 seeded with the block's seed are
 * below dropout_p16.  t is the block's step counter (NITRO_T_STEP): the
 * number of nitro_integersgd_step calls so far, modulo 2^28.  Set the rate
 * to 0 (nitro_block_set_dropout) for inference. */

typedef struct nitro_block nitro_block;

/* Creates a block on the current CUDA device and initialises every weight
 * tensor with the integer Kaiming rule (Sec. 3.3.1): b = floor(128*1732 /
 * (isqrt(fan_in)*1000)), weights uniform on {-b..b}.  Element e of tensor t
 * (t = layer index, 255 for the learning layer) is -b + u mod (2b+1), u being
 * output number t*2^40 + e of SplitMix64 seeded with `seed`.  Weights are
 * uploaded on `stream`.  Returns NITRO_ERR_ARG for inconsistent shapes,
 * NITRO_ERR_CUDA if allocation fails (nothing is leaked). */
nitro_status nitro_init_block(const nitro_block_desc* desc, uint64_t seed, void* stream,
                              nitro_block** out);

/* Forward layers of the block (Sec. 3.3, first phase): for each layer
 * z = conv/linear(a, W) (exact integer sum), z* = floor(z / SF) (Eq. 1),
 * NITRO-ReLU (Sec. 3.2.2), optional max-pool.  a_in: device int8
 * [batch x in_features]; a_out: device int8 [batch x out_features] of the
 * last layer, or NULL.  Caches what backward needs.  0 <= batch <= max_batch.
 * For an output block this only records the batch. */
nitro_status nitro_block_forward(nitro_block* blk, const int8_t* a_in, int batch,
                                 int8_t* a_out, void* stream);

/* Local backward of the block (Sec. 3.3, second phase): learning layer
 * y_hat = floor(a W_lr^T / (2^8 d)), scaled one-hot target y (32 at the label,
 * Sec. 3.3.4 and App. A), grad_L = y_hat - y, RSS loss; weight gradient of
 * the learning layer; delta_fw = grad_L W_lr (pre-update W_lr, Sec. 3.3.5);
 * then through each forward layer, last to first: max-pool backward (to the
 * recorded window maximum), NITRO-ReLU backward (per piece), straight-through
 * NITRO-Scaling (Sec. 3.2.1), weight gradient, input gradient.  Must follow
 * nitro_block_forward with the same a_in and batch.  labels: device int32
 * [batch]; loss_dev: device int64 [1] receiving floor(SSE/2), or NULL. */
nitro_status nitro_block_backward(nitro_block* blk, const int8_t* a_in, const int32_t* labels,
                                  int batch, int64_t* loss_dev, void* stream);

/* IntegerSGD (Algorithm 1) on every weight tensor of the block using the
 * weight gradients of the last backward: d = R(dW, gamma_inv), plus
 * R(W, eta_inv) if eta_inv != 0, W -= d; R = floor or trunc per sgd_round.
 * Forward layers use gamma_inv^fw = 2^6*G*gamma_inv_lr and eta_inv_fw; the
 * learning layer gamma_inv_lr and eta_inv_lr. */
nitro_status nitro_integersgd_step(nitro_block* blk, void* stream);

/* nitro_block_backward followed by nitro_integersgd_step, with the same
 * results bit for bit (Sec. 3.3: a block's backward and its update depend on
 * no other block).  The conv layers whose weight gradient runs on the tensor
 * cores apply Algorithm 1 inside that kernel, to each output tile once its
 * sum is final: their new weights and limb planes are written without a
 * second pass over the gradients, and their input gradient (which reads the
 * pre-update weights) runs before the update.  The weight gradients stay
 * readable (nitro_block_get_tensor) after the call.  A data-parallel
 * exchange of the gradients needs the two separate calls instead.
 * Errors: as nitro_block_backward. */
nitro_status nitro_block_backward_update(nitro_block* blk, const int8_t* a_in,
                                         const int32_t* labels, int batch, int64_t* loss_dev,
                                         void* stream);

/* Replaces the IntegerSGD hyper-parameters of a block (Algorithm 1):
 * gamma_inv_lr (the forward layers use 2^6*G*gamma_inv_lr, Sec. 3.3.5),
 * eta_inv_fw and eta_inv_lr.  App. B multiplies the inverse learning rate by 3
 * each time the test accuracy reaches a plateau; this is the call that applies
 * such a change.  Host-only: it takes effect at the next nitro_integersgd_step
 * call, while a CUDA graph that captured an earlier step keeps the values it
 * was captured with until it is captured again.  Range checks as in
 * nitro_init_block (1 <= gamma_inv_lr <= 2^48, eta >= 0); on NITRO_ERR_ARG
 * nothing changes. */
nitro_status nitro_block_set_hyper(nitro_block* blk, int64_t gamma_inv_lr, int64_t eta_inv_fw,
                                   int64_t eta_inv_lr);

/* Replaces the dropout rate of the block's linear forward layers (0..65536,
 * units of 2^-16; 0 = off, e.g. for inference).  Host-only: it takes effect
 * at the next nitro_block_forward call; a CUDA graph that captured an earlier
 * forward keeps the rate it was captured with.  NITRO_ERR_ARG if out of
 * range (nothing changes). */
nitro_status nitro_block_set_dropout(nitro_block* blk, int dropout_p16);

/* Tensors readable / writable through get/set_tensor.  Batch-shaped tensors
 * hold the last forward/backward batch. */
typedef enum {
    NITRO_T_W = 0,       /* layer weights, int32                               */
    NITRO_T_DW = 1,      /* layer weight gradient, int64                       */
    NITRO_T_WLR = 2,     /* learning/output weights [G x d], int32 (layer = 0) */
    NITRO_T_DWLR = 3,    /* learning weight gradient, int64 (layer = 0)        */
    NITRO_T_ACT = 4,     /* layer output after pool, int8 [batch x out]        */
    NITRO_T_REGION = 5,  /* NITRO-ReLU piece 0..3 per pre-pool output, int8;
                            4 = dropped by dropout                             */
    NITRO_T_ARGMAX = 6,  /* max-pool window position 0..3 per output, int8     */
    NITRO_T_DELTA = 7,   /* gradient at the layer's pre-activation, int32      */
    NITRO_T_GRAD_L = 8,  /* loss gradient [batch x G], int32 (layer = 0)       */
    NITRO_T_SSE = 9,     /* sum of squared errors, int64 [1] (layer = 0)       */
    NITRO_T_LR_IN = 10,  /* pooled learning-layer input z^mp [batch x d], int8
                            (layer = 0; blocks with learning-layer pooling,
                            NITRO_ERR_ARG for the others)                      */
    NITRO_T_LR_ARGMAX = 11, /* window position r*kw + s of each z^mp value,
                            uint8 [batch x d] (same blocks)                    */
    NITRO_T_STEP = 12    /* step counter of the dropout masks, uint32 [1]
                            (layer = 0); writable, for resuming                */
} nitro_tensor;

/* Size in bytes of tensor (which, layer) at the current batch. */
nitro_status nitro_block_tensor_bytes(const nitro_block* blk, int which, int layer,
                                      size_t* bytes);

/* Synchronises the device, copies the tensor to host memory host_dst (which
 * must hold exactly `bytes` = nitro_block_tensor_bytes), and returns the
 * latched device status (NITRO_OK if none). */
nitro_status nitro_block_get_tensor(nitro_block* blk, int which, int layer, void* host_dst,
                                    size_t bytes);

/* Synchronises the device and overwrites a weight tensor (NITRO_T_W,
 * NITRO_T_DW, NITRO_T_WLR, NITRO_T_DWLR) or the step counter (NITRO_T_STEP)
 * from host memory; used to resume from a checkpoint.  Bit-exact: all state
 * is integer. */
nitro_status nitro_block_set_tensor(nitro_block* blk, int which, int layer,
                                    const void* host_src, size_t bytes);

/* Device address of the block's int64 weight gradient (NITRO_T_DW of a
 * layer, or NITRO_T_DWLR with layer 0) and its size in bytes, for a
 * data-parallel exchange step between nitro_block_backward and
 * nitro_integersgd_step (Algorithm 1 applied once to the gradient summed over
 * replicas: the sum of int64 gradients is exact modulo 2^64 in any order, and
 * the floor of the update comes after it).  The memory stays owned by the
 * block and valid until nitro_destroy_block; the caller may read and
 * overwrite it in stream order between those two calls.  Does not
 * synchronise.  Errors: NITRO_ERR_ARG for a null handle or pointer, another
 * tensor, or a layer out of range. */
nitro_status nitro_block_grad_device(nitro_block* blk, int which, int layer, void** dev_ptr,
                                     size_t* bytes);

/* Synchronises the device and returns the latched status as nitro_status
 * (TIMEOUT before OVERFLOW before a bad label = ARG); clears it if clear. */
nitro_status nitro_block_status(nitro_block* blk, int clear);

/* Synchronises the device and returns the raw NITRO_STATUS_BIT_* word. */
uint32_t nitro_block_status_bits(nitro_block* blk);

/* Releases every device buffer of the block.  NULL is ignored. */
void nitro_destroy_block(nitro_block* blk);

/* ---- Kernel-level contractions ----------------------------------------------
 * One contraction of a 3x3 conv layer (stride 1, zero padding 1; Sec. 3.2.1
 * conv expression and its two adjoints) or one integer GEMM, on caller-owned
 * device buffers, through the same operand split and kernels as the block
 * step.  Outputs are the exact integer sums modulo 2^64, as int64:
 *   NITRO_CONTRACT_FWD   x = int8 a [B][H][W][Cin],  y = int32 W [Cout][3][3][Cin]
 *                        out = z [B][H][W][Cout],  z = sum_(ky,kx,ci) a[y+ky-1][x+kx-1][ci] W
 *   NITRO_CONTRACT_WGRAD x = int8 a,                 y = int32 d [B][H][W][Cout]
 *                        out = dW [Cout][3][3][Cin] = sum_(b,y,x) d[b,y,x,co] a[b,y+ky-1,x+kx-1,ci]
 *   NITRO_CONTRACT_DGRAD x = int32 d [B][H][W][Cout], y = int32 W
 *                        out = g [B][H][W][Cin] = sum_(ky,kx,co) d[b,y-ky+1,x-kx+1,co] W
 * Asynchronous on `stream`; the handle owns its packing workspace (sized at
 * create for max_batch) and must not be used by two streams at once.  Buffers
 * need only the alignment of their element type (here and in the block calls). */
typedef enum { NITRO_CONTRACT_FWD = 0, NITRO_CONTRACT_WGRAD = 1, NITRO_CONTRACT_DGRAD = 2 } nitro_contract_mode;
typedef struct nitro_conv nitro_conv;
nitro_status nitro_conv3x3_create(int max_batch, int h, int w, int cin, int cout, nitro_conv** out);
nitro_status nitro_conv3x3_contract(nitro_conv* c, int mode, const void* x, const int32_t* y,
                                    int batch, int64_t* out, void* stream);
nitro_status nitro_conv3x3_status(nitro_conv* c);   /* synchronises; latched TIMEOUT */
void nitro_conv3x3_destroy(nitro_conv* c);

/* C[m][n] = sum_k A[m][k] B[n][k]: A int8 [M][K], B int32 [N][K], C int64
 * [M][N], row-major.  The integer matrix product the linear layers reduce to
 * (Sec. 3.2.1 linear expression). */
typedef struct nitro_gemm nitro_gemm;
nitro_status nitro_gemm_create(int max_m, int max_n, int max_k, nitro_gemm** out);
nitro_status nitro_gemm_run(nitro_gemm* g, const int8_t* a, const int32_t* b, int m, int n, int k,
                            int64_t* c, void* stream);
nitro_status nitro_gemm_status(nitro_gemm* g);      /* synchronises; latched TIMEOUT */
void nitro_gemm_destroy(nitro_gemm* g);

/* ---- Allocation-free layer forward ----------------------------------------
 * The paper has no counterpart to this call: it exists for callers that
 * cannot allocate device memory once running - code inside a host program
 * that owns the whole device-memory budget, real-time loops that forbid
 * allocation after start-up, or code that must not let cudaMalloc/cudaFree
 * synchronise the device.
 *
 * Runs the forward of ONE 3x3 conv layer exactly as nitro_block_forward does
 * (conv, NITRO-Scaling, NITRO-ReLU, optional 2x2 max-pool) on caller-owned
 * buffers: a_in int8 NHWC [batch x h x w x cin], weights int32 OHWI, a_out
 * int8 [batch x h' x w' x cout], region int8 [batch x h x w x cout], argmax
 * int8 [batch x h' x w' x cout] (pool2x2 only, else may be NULL), where
 * h' = pool2x2 ? floor(h / 2) : h and w' = pool2x2 ? floor(w / 2) : w (an odd
 * last row or column is dropped by the pool, as in the block path).  It calls no
 * cudaMalloc, cudaFree or allocating library routine: the int64
 * pre-activations go to a fixed 16 MiB array inside the library, so
 * batch*h*w*cout may be at most 2^21; larger sizes return NITRO_ERR_ARG and
 * queue nothing.  Every GPU that loads the library holds that array until the
 * process exits.  The first call on each device looks up the array's address
 * (cudaGetSymbolAddress, with that device current) and keeps it for the life
 * of the process; make that first call before any stream capture.  Calls
 * after a cudaDeviceReset of that device are not supported (the library image
 * may be reloaded elsewhere).  All calls share the one array: calls whose work
 * overlaps on the GPU (different streams, or different host threads) race
 * and give wrong results; serialise them, e.g. on one stream. */
nitro_status nitro_conv3x3_forward_noalloc(const int8_t* a_in, const int32_t* weights, int batch,
                                           int h, int w, int cin, int cout, int pool2x2,
                                           int alpha_inv, int8_t* a_out, int8_t* region,
                                           int8_t* argmax, void* stream);

/* ---- Integer data pre-processing (App. A) ---------------------------------
 * Maps a dataset of n 8-bit values x (every element of every sample, e.g.
 * image bytes) to int8 values centred on 0 with a spread of about 64:
 *   mu    = floor(sum x / n)
 *   omega = floor(sum |x - mu| / n)          (mean absolute deviation)
 *   x_hat = floor((x - mu) * 51 / omega), clamped to [-127, 127]
 * 51 = floor(64 * 0.8), since the MAD of Gaussian data is ~0.8 sigma.  The
 * appendix leaves omega = 0 undefined: it is read as a divisor of 1.
 *
 * nitro_prep_fit computes mu and omega of one device buffer x [n] (two
 * passes over it) and keeps them in the handle with the 256-entry map they
 * define; nitro_prep_apply maps any device buffer x [n] to out [n] (int8) with
 * the statistics of the last fit, so a test set can be mapped with the
 * training set's.  out may equal x (in place) but must not overlap it
 * otherwise.  Both calls are asynchronous on `stream` and may be captured into
 * a CUDA graph; the handle must not be used by two streams at once.
 * nitro_prep_stats synchronises the device and returns the statistics of the
 * last fit.  Buffers need no alignment; x and out at the same offset from a
 * 16-byte boundary take 16-byte vector accesses.
 * Errors: NITRO_ERR_ARG for a null handle or pointer, n < 1 in fit (n < 0 in
 * apply, where 0 queues nothing), n > 2^48, or apply / stats before a fit;
 * NITRO_ERR_CUDA for a failed allocation or launch. */
typedef struct nitro_prep nitro_prep;
nitro_status nitro_prep_create(nitro_prep** out);
nitro_status nitro_prep_fit(nitro_prep* p, const uint8_t* x, int64_t n, void* stream);
nitro_status nitro_prep_apply(nitro_prep* p, const uint8_t* x, int64_t n, int8_t* out,
                              void* stream);
nitro_status nitro_prep_stats(nitro_prep* p, int64_t* mu, int64_t* omega);
void nitro_prep_destroy(nitro_prep* p);

/* ---- Diagnostics (not part of the training step) -------------------------
 * Every kernel launch of the library is counted.  With profiling on, each
 * launch is also bracketed by CUDA events recorded on its own stream and
 * tagged with its kernel class and algorithmic work (integer ops = 2 x MACs;
 * bytes for the HBM-bound update).  Profile eager calls only: events are not
 * recorded into CUDA-graph captures. */
uint64_t nitro_kernel_launches(void);            /* launches issued since load */
void nitro_profile_enable(int on);
void nitro_profile_reset(void);                  /* drops recorded launches  */
int nitro_profile_kernel_count(void);            /* number of kernel classes */
const char* nitro_profile_kernel_name(int id);   /* static string            */
/* Synchronises on the recorded events of class `id` and returns their count,
 * summed device time (ms) and summed algorithmic ops and bytes. */
nitro_status nitro_profile_read(int id, uint64_t* launches, double* ms, double* ops,
                                double* bytes);
/* Launches recorded since the last reset, and launch i (0-based, in launch
 * order): its kernel class, device time (ms), algorithmic ops and bytes.
 * Synchronises on that launch's events; NITRO_ERR_ARG for i out of range. */
int nitro_profile_record_count(void);
nitro_status nitro_profile_record(int i, int* kernel, double* ms, double* ops, double* bytes);

/* Failure-path check of the bounded device waits (the library's TIMEOUT
 * status; the paper has no counterpart: its failure model is integer overflow).
 * Queues on `stream` one CTA that allocates TMEM as the contraction kernels do
 * and waits, through their bounded mbarrier wait, on a barrier that nothing
 * ever completes.  After wait_us microseconds the wait gives up: the kernel
 * latches the TIMEOUT bit in b's status word, the CTA's other waiting warps
 * see its abort flag and leave, TMEM is freed and the kernel returns, so the
 * CUDA context stays usable and the block keeps its state.  The next
 * nitro_block_status / nitro_block_get_tensor returns NITRO_ERR_TIMEOUT until
 * the status is cleared (nitro_block_status(b, 1)).
 * Errors: NITRO_ERR_ARG for a null handle or wait_us outside [1, 2000000];
 * NITRO_ERR_CUDA for a failed launch. */
nitro_status nitro_block_diag_timeout(nitro_block* b, int wait_us, void* stream);

/* Static, human-readable name of a status code. */
const char* nitro_status_str(nitro_status s);

#ifdef __cplusplus
}
#endif

#endif /* NITRO_H */
