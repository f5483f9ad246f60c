// tcgen05 implicit-GEMM kernels for the 3x3 conv forward, weight gradient
// and input gradient, plus the kernels that split operands into bf16 limb
// planes.  See tc_conv.cuh for the exactness argument and the layouts.
//
// A persistent CTA computes 128 x N output tiles, each over a range of
// K-blocks (64 elements each).  Warp 0 issues TMA loads into an S-stage shared-memory ring,
// warp 1 allocates TMEM and issues the MMAs, warps 2..17 drain the fp32 TMEM
// accumulator every <= 16 K-blocks into int64 registers (four warps per TMEM
// lane quadrant, each owning a quarter of the N columns).  Four TMEM accumulators
// rotate so the MMAs run up to three chunks ahead of the drain.
// Every wait on an mbarrier is bounded in time; on expiry the kernel raises
// the TIMEOUT status bit, lets the other roles leave, frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "prof.cuh"
#include "tc_conv.cuh"

namespace nitro {
namespace {

enum TcMode : int { TC_FWD = 0, TC_WGRAD = 1, TC_DGRAD = 2, TC_GEMM = 3 };

constexpr int kBM = 128;              // rows per tile (TMEM lanes)
constexpr int kBK = 64;               // K elements per block (one 128-byte row)
constexpr int kChunkBlocks = 16;      // 16 x 64 = 1024 products per exact chunk
// Warp roles: warpgroup 0 = TMA warp, MMA warp and two idle warps; warpgroups
// 1 to 4 = the epilogue, four warps per TMEM lane quadrant, each holding a
// quarter of the N columns as int64 accumulators.  The epilogue is bound by
// memory latency, so it gets as many warps as the register file allows; the
// warpgroups split it with setmaxnreg: 128 x kRegsProducer + 32 x kEpiWarps x
// kRegsEpilogue must not exceed kThreads x the registers the kernel is
// launched with (checked on the host before the first launch).  A layout with
// eight epilogue warps (half the N columns each, 224 registers, no spills) was
// measured slower: 175k against 257k images/s on the VGG-style step.
constexpr int kEpiWarp0 = 4;          // first epilogue warp
constexpr int kEpiWarps = 16;         // 4 per TMEM lane quadrant
constexpr int kThreads = 32 * (kEpiWarp0 + kEpiWarps);
constexpr int kRegsProducer = 32, kRegsEpilogue = 112;
constexpr uint64_t kWaitNs = 2000000000ull;   // 2 s bound on any wait

// ------------------------------------------------------------------ PTX
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
        " selp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Bounded wait: false when the time limit passed (TIMEOUT raised) or another
// role of this CTA gave up.  Inlined: a function call cannot sit inside the
// register-split (setmaxnreg) regions of the contraction kernel.
__device__ __forceinline__ bool mbar_wait_slow(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                            uint32_t* status, uint64_t limit_ns) {
    const uint64_t t0 = global_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63) == 0) {
            if (*abort_flag) return false;
            if (global_ns() - t0 > limit_ns) {
                *abort_flag = 1;
                atomicOr(status, ST_TIMEOUT);
                return false;
            }
        }
    }
}
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                          uint32_t* status, uint64_t limit_ns = kWaitNs) {
    return mbar_try_wait(bar, parity) || mbar_wait_slow(bar, parity, abort_flag, status, limit_ns);
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                            int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1)
        : "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                            int c0, int c1, int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
        : "memory");
}
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                            int c0, int c1, int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}
__device__ __forceinline__ void tma_load_5d(uint32_t dst, const CUtensorMap* m, uint32_t bar,
                                            int c0, int c1, int c2, int c3, int c4) {
    asm volatile(
        "cp.async.bulk.tensor.5d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6, %7}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(m)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3),
        "r"(c4)
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor, K-major operand, 128-byte swizzle: rows of
// 128 bytes, 8-row groups 1024 bytes apart (stride byte offset), version 1.
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)1 << 16;               // leading byte offset (unused here)
    d |= (uint64_t)(1024 >> 4) << 32;     // stride byte offset
    d |= (uint64_t)1 << 46;               // descriptor version
    d |= (uint64_t)2 << 61;               // 128-byte swizzle
    return d;
}

// MN-major operand, 128-byte swizzle: rows of 128 bytes run along K, each
// holding 64 consecutive M (or N) elements; 64-element blocks along M/N lie
// `mn_stride` bytes apart (leading byte offset), 8-row groups along K 1024
// bytes apart (stride byte offset).
__device__ __forceinline__ uint64_t desc_sw128_mn(uint32_t saddr, uint32_t mn_stride) {
    uint64_t d = 0;
    d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((mn_stride >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)(1024 >> 4) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor: kind::f16, A = B = bf16, D = f32; A (bit 15) and B
// (bit 16) K-major unless marked MN-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n, bool a_mn = false, bool b_mn = false) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (a_mn ? (1u << 15) : 0u) | (b_mn ? (1u << 16) : 0u) |
           ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void umma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                          uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
        : "memory");
}

__device__ __forceinline__ void tmem_ld16_nowait(uint32_t taddr, uint32_t* r) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, "
        "%11, %12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}

// Wait for this thread's outstanding tcgen05.ld, then mark the n destination
// registers as written here, so that no use of them is placed before the wait.
__device__ __forceinline__ void reg_touch16(uint32_t* r) {
    asm volatile(""
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                   "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                   "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]));
}
template <int n>
__device__ __forceinline__ void tmem_wait_ld(uint32_t* r) {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int j = 0; j < n / 16; ++j) reg_touch16(r + 16 * j);
}

// Limbs of a tensor with max |x| = m.  The split is canonical: limbs 0..2 are
// the digits ((x + 128) & 255) - 128 of successive base-256 remainders and
// limb 3 takes the rest (in [-128, 128] for int32).  With the thresholds below
// every limb at index >= L is zero, so the first L planes of the 4-limb split
// are exact and producers may write all four without knowing L.
__host__ __device__ __forceinline__ int limb_count(uint32_t m) {
    return m <= 127u ? 1 : (m <= 32639u ? 2 : (m <= 8355711u ? 3 : 4));
}

// ------------------------------------------------------------------ kernel
struct TcArgs {
    int B, H, W, Cin, Cout, Bp;
    int cin_k;             // channels per tap in the K index (Cin rounded up to 64)
    int taps;              // 9, or 1 for im2col input (forward / wgrad: no tap shift)
    int ntx, nty;          // pixel tiles along x and y (forward / dgrad)
    int wb, hb, bb;        // pixel box (forward / dgrad): wb * hb * bb = 128
    int tiles_m, tiles_n, total_tiles;
    // dividers for the tile decode (filled at launch): tiles_n, tiles_m, ntx, nty;
    // pixel-box sides are powers of two: log2 wb, log2 hb
    FloorDiv32 dv_tn, dv_tm, dv_ntx, dv_nty;
    int lg_wb, lg_hb;
    int kb_total, kb_per_split;
    int ncols;             // valid output columns (Cout for fwd/wgrad, Cin for dgrad)
    const uint32_t* max_a;  // max |operand| words setting the limb counts (nullptr = 1 limb)
    const uint32_t* max_b;
    int64_t* out;
    uint32_t* status;
    int atomic_out;
    int out_vec;           // out is 16-byte aligned: pairs of int64 stored together
    // forward with fused NITRO-Scaling / NITRO-ReLU / max-pool epilogue
    int fuse;
    FloorDiv alpha;        // divide by alpha_inv
    FloorDiv32 sf32;       // divide by 9 * Cin (after the shift by 8)
    int64_t z_hi, z_lo;    // z >= 128 SF: piece 3; z < -127 SF: piece 0
    int mu, pool, oh, ow;
    int8_t* act;           // layer output (post-pool) int8 NHWC
    int8_t* out2;          // optional second copy of the output (caller's buffer)
    int8_t* region;        // NITRO-ReLU piece per pre-pool output
    int8_t* argmax;        // window position per pooled output
    uint16_t* next_nhwc;   // bf16 copy of the output for the next layer's forward, or null
    // dgrad with fused max-pool / NITRO-ReLU backward into the lower layer's delta
    FloorDiv32 alpha32;
    const uint32_t* bound_a;   // max|delta| and max|W| of this layer (int64 exactness bound)
    const uint32_t* bound_b;
    int low_h, low_w, low_pool;
    const int8_t* low_region;
    const int8_t* low_argmax;
    int32_t* low_delta;
    uint32_t* low_maxabs;
    // weight gradient: valid rows (taps == 1) and the row stride of dW / W
    int rows;
    int64_t cstride;
    // weight gradient with IntegerSGD applied to the finished sums (no K split)
    int sgd;
    int32_t* wt;               // the layer's weights [Cout][9][Cin]
    uint16_t* wp;              // weight limb planes [4][Cout][row_k], or null
    int64_t w_plane;
    int row_k, tap_k;
    FloorDiv gdiv, ediv;       // gamma_inv, eta_inv (eta_inv = 0: no decay)
    int decay, trunc;
    uint32_t* maxabs_w;        // max |new W| (atomic max, zeroed by the caller)
};

// 16 int8 values (4 packed words) -> one 16-byte store
__device__ __forceinline__ void st16(int8_t* dst, const uint32_t* w) {
    *reinterpret_cast<uint4*>(dst) = make_uint4(w[0], w[1], w[2], w[3]);
}
// 16 int8 values (4 packed words) -> 16 bf16 values (two 16-byte stores),
// through the 256-entry table of bf16 bits indexed by byte ^ 0x80
__device__ __forceinline__ void st16_bf16(uint16_t* dst, const uint32_t* w, const uint16_t* tab) {
    uint32_t o[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
        const uint32_t lo = (w[k >> 1] >> (16 * (k & 1))) & 255u;
        const uint32_t hi = (w[k >> 1] >> (16 * (k & 1) + 8)) & 255u;
        o[k] = (uint32_t)tab[lo ^ 0x80u] | ((uint32_t)tab[hi ^ 0x80u] << 16);
    }
    reinterpret_cast<uint4*>(dst)[0] = make_uint4(o[0], o[1], o[2], o[3]);
    reinterpret_cast<uint4*>(dst)[1] = make_uint4(o[4], o[5], o[6], o[7]);
}

// PB = B-operand limbs carried per stage: one A tile feeds PB limb tiles of B
// and PB accumulators, so wide B operands do not re-stream A once per limb.
template <int N, int PB>
struct TcCfg {
    static constexpr int A_BYTES = kBM * kBK * 2;
    static constexpr int B_BYTES = N * kBK * 2;
    static constexpr int STAGE = A_BYTES + PB * B_BYTES;
    static constexpr int S_FIT = (230912 - 1536) / STAGE;   // ~225 KB of shared memory
    // at most 6 stages: deeper rings gave no gain in the training step and lost
    // up to 14% in the kernel-level contractions (more TMA writes in flight
    // compete with the MMA's shared-memory reads)
    static constexpr int S = S_FIT > 6 ? 6 : S_FIT;
    static constexpr int SMEM = 1024 + S * STAGE + 1024;
    static constexpr int NBUF = (512 / (PB * N)) > 4 ? 4 : (512 / (PB * N));   // accumulator sets
    static constexpr int TCOLS = NBUF * PB * N;                                  // 256 or 512
};

struct Tile {
    int mt, nt, kb0, kb1;
};
__device__ __forceinline__ int udiv32(const FloorDiv32& f, int x) { return (int)f.udiv((uint32_t)x); }

__device__ __forceinline__ Tile decode_tile(const TcArgs& a, int tile) {
    Tile t;
    const int r = udiv32(a.dv_tn, tile);
    t.nt = tile - r * a.tiles_n;
    const int split = udiv32(a.dv_tm, r);
    t.mt = r - split * a.tiles_m;
    t.kb0 = split * a.kb_per_split;
    t.kb1 = min(a.kb_total, t.kb0 + a.kb_per_split);
    return t;
}

// Persistent: CTA c handles tiles c, c + gridDim.x, ...; the TMA ring, the
// MMA chunk sequence and the two TMEM accumulators run on across tiles, so
// one tile's epilogue overlaps the next tile's loads and MMAs.
template <int MODE, int N, int PB>
__global__ void __launch_bounds__(kThreads, 1)
    k_tc_gemm(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
              const TcArgs args) {
    using C = TcCfg<N, PB>;
    constexpr int S = C::S;
    constexpr int NH = N / 4;            // columns per epilogue warp
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + S * C::STAGE);
    // bars[0..S) full, [S..2S) empty, then NBUF tmem-full and NBUF tmem-empty
    constexpr int NBUF = C::NBUF;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * S + 2 * NBUF);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int* hiskip_slot = reinterpret_cast<int*>(tmem_slot + 2);
    int8_t* relu_tab = reinterpret_cast<int8_t*>(smem + S * C::STAGE + 256);   // 255 entries
    // bf16 bits of every int8 value v, at index (v + 128) = byte ^ 0x80
    uint16_t* bf16_tab = reinterpret_cast<uint16_t*>(smem + S * C::STAGE + 512);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (S + s); };
    auto tfull_bar = [&](int b) { return bar0 + 8u * (2 * S + b); };
    auto tempty_bar = [&](int b) { return bar0 + 8u * (2 * S + NBUF + b); };

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_bar(s), 1);
            mbar_init(empty_bar(s), 1);
        }
        for (int b = 0; b < NBUF; ++b) {
            mbar_init(tfull_bar(b), 1);
            mbar_init(tempty_bar(b), kEpiWarps);
        }
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    // NITRO-ReLU value of every z* in [-127, 127] (fused forward epilogue)
    if (MODE == TC_FWD && args.fuse) {
        for (int i = threadIdx.x; i < 255; i += kThreads)
            relu_tab[i] = (int8_t)relu_value((int64_t)i - 127, args.alpha, args.mu);
        for (int i = threadIdx.x; i < 256; i += kThreads)
            bf16_tab[i] = __bfloat16_as_ushort(__float2bfloat16_rn((float)(i - 128)));
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(tmem_slot)),
                     "r"(C::TCOLS)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (warp == 0 && lane == 0) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
    }
    // The set-up above touches only shared memory, TMEM and the kernel's own
    // tensor maps, so it may overlap the end of the previous kernel in the
    // stream; from here on the kernel reads what that kernel wrote.
    pdl_wait();
    if (threadIdx.x == 0) {
        // Fused input gradient: the lower delta is stored as the low 32 bits of
        // the exact sum, and limb pairs with la + lb >= 4 only add multiples
        // of 2^32.  They matter only for deciding OVERFLOW, so once that bit
        // is latched they are skipped.  Read once per CTA so that all roles
        // walk the same passes (CTAs may differ; each result is the same).
        *hiskip_slot = (MODE == TC_DGRAD && args.fuse)
            ? ((*reinterpret_cast<volatile uint32_t*>(args.status) & ST_OVERFLOW) != 0) : 0;
    }
    // int32 x int32 contraction: flag when max|delta| max|W| 9 Cout >= 2^63
    if (MODE == TC_DGRAD && args.fuse && blockIdx.x == 0 && threadIdx.x == 64 &&
        int64_bound_exceeded(*args.bound_a, *args.bound_b, 9LL * args.Cout))
        atomicOr(args.status, ST_OVERFLOW);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const int LA = args.max_a ? limb_count(*args.max_a) : 1;
    const int LB = args.max_b ? limb_count(*args.max_b) : 1;
    const int hiskip = *hiskip_slot;
    // B limbs that pair with A limb la: all, or those with la + lb <= 3
    auto lb_limit = [&](int la) { return hiskip ? min(LB, 4 - la) : LB; };

    if (warp < kEpiWarp0) {
    // warpgroup 0 gives registers back, then splits into its roles
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsProducer));
    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer
            int it = 0;
            for (int tile = blockIdx.x; tile < args.total_tiles; tile += gridDim.x) {
                const Tile T = decode_tile(args, tile);
                const int n0 = T.nt * N;
                const int mq = udiv32(args.dv_ntx, T.mt), tb = udiv32(args.dv_nty, mq);
                const int tx = T.mt - mq * args.ntx, ty = mq - tb * args.nty;
                const int x0 = tx * args.wb, y0 = ty * args.hb, b0 = tb * args.bb;
                // weight gradient: the tile's two 64-row blocks of (tap, ci) rows
                // are fixed for the tile (channel start, tap offsets)
                int wa_ci[2] = {0, 0}, wa_dx[2] = {0, 0}, wa_dy[2] = {0, 0};
                if (MODE == TC_WGRAD) {
#pragma unroll
                    for (int j = 0; j < 2; ++j) {
                        const int m = T.mt * kBM + j * 64;
                        int t = m / args.cin_k, ci0 = m - t * args.cin_k;
                        if (t >= args.taps) { t = 0; ci0 = args.cin_k; }   // past the last tap: zeros
                        if (args.taps == 1) t = 4;                         // im2col rows: centre tap
                        wa_ci[j] = ci0;
                        wa_dx[j] = t % 3 - 1;
                        wa_dy[j] = t / 3 - 1;
                    }
                }
                for (int la = 0; la < LA; ++la)
                for (int lb0 = 0; lb0 < lb_limit(la); lb0 += PB) {
                    const int nb = min(PB, lb_limit(la) - lb0);
                    // weight gradient: K-block kb = pixel box (xt, yt) of image bk,
                    // walked incrementally
                    int wxt = 0, wyt = 0, wbk = 0;
                    if (MODE == TC_WGRAD) {
                        wxt = T.kb0 % args.ntx;
                        wyt = (T.kb0 / args.ntx) % args.nty;
                        wbk = T.kb0 / (args.ntx * args.nty);
                    }
                    // forward / input gradient: K-block kb = (tap t, 64-channel block cb),
                    // cb fastest, walked incrementally
                    const int knc = MODE == TC_FWD ? args.cin_k / kBK : (args.Cout + kBK - 1) / kBK;
                    int kt = 0, kcb = 0;
                    if (MODE == TC_FWD || MODE == TC_DGRAD) {
                        kt = T.kb0 / knc;
                        kcb = T.kb0 - kt * knc;
                    }
                    for (int kb = T.kb0; kb < T.kb1; ++kb, ++it) {
                        const int s = it % S;
                        if (!mbar_wait(empty_bar(s), ((it / S) & 1) ^ 1, abort_flag, args.status))
                            goto producer_done;
                        const uint32_t fb = full_bar(s);
                        const uint32_t a_dst = smem_u32(smem + s * C::STAGE);
                        const uint32_t b_dst = a_dst + C::A_BYTES;
                        // the B box spans PB limb planes (past the last limb: zeros or
                        // planes the MMA does not read)
                        mbar_expect_tx(fb, C::A_BYTES + (MODE == TC_GEMM ? nb : PB) * C::B_BYTES);
                        if (MODE == TC_GEMM) {
                            tma_load_2d(a_dst, &tmA, fb, kb * kBK, T.mt * kBM);
                            for (int j = 0; j < nb; ++j)
                                tma_load_3d(b_dst + j * C::B_BYTES, &tmB, fb, kb * kBK, n0, lb0 + j);
                        } else if (MODE == TC_FWD) {
                            const int t = kt, cb = kcb;
                            const int tc = args.taps == 1 ? 4 : t;   // im2col rows: centre tap
                            const int ky = tc / 3, kx = tc - 3 * ky;
                            tma_load_4d(a_dst, &tmA, fb, cb * kBK, x0 + kx - 1, y0 + ky - 1, b0);
                            // PB limb tiles [limb][N rows][64 k], one box
                            tma_load_3d(b_dst, &tmB, fb, t * args.cin_k + cb * kBK, n0, lb0);
                            if (++kcb == knc) { kcb = 0; ++kt; }
                        } else if (MODE == TC_DGRAD) {
                            const int t = kt, cb = kcb, ky = t / 3, kx = t - 3 * ky;
                            if (++kcb == knc) { kcb = 0; ++kt; }
                            tma_load_5d(a_dst, &tmA, fb, cb * kBK, x0 - kx + 1, y0 - ky + 1, b0, la);
                            // B MN-major from the forward planes [L][Cout][9][Cin64]:
                            // rows co (K) of 64 consecutive ci (N) for tap t; one box per
                            // 64-channel block h brings PB limbs, stored [h][limb]
#pragma unroll
                            for (int h = 0; h < N / 64; ++h)
                                tma_load_4d(b_dst + h * (PB * 64 * 128), &tmB, fb, n0 + 64 * h, t,
                                            cb * kBK, lb0);
                        } else {  // TC_WGRAD: rows (tap, ci), K = a 64-pixel box (wb x hb)
                            // of one image; both operands MN-major from the NHWC
                            // copies (channels contiguous), the tap shift on x / y.
                            const int px = wxt * args.wb, py = wyt * args.hb, bk = wbk;
#pragma unroll
                            for (int j = 0; j < 2; ++j)
                                tma_load_4d(a_dst + j * (64 * 128), &tmA, fb, wa_ci[j], px + wa_dx[j],
                                            py + wa_dy[j], bk);
                            // one box per 64-channel block h brings PB limbs, stored [h][limb]
#pragma unroll
                            for (int h = 0; h < N / 64; ++h)
                                tma_load_5d(b_dst + h * (PB * 64 * 128), &tmB, fb, n0 + 64 * h, px,
                                            py, bk, lb0);
                            if (++wxt == args.ntx) {
                                wxt = 0;
                                if (++wyt == args.nty) {
                                    wyt = 0;
                                    ++wbk;
                                }
                            }
                        }
                    }
                }
            }
        producer_done:;
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer
            // the nb limb tiles of B lie back to back in shared memory and their
            // accumulators side by side in TMEM: one MMA of width nb * N covers them
            uint32_t idesc_nb[PB + 1];
#pragma unroll
            for (int j = 1; j <= PB; ++j)
                idesc_nb[j] = idesc_bf16(kBM, j * N, MODE == TC_WGRAD, MODE == TC_WGRAD || MODE == TC_DGRAD);
            // K-major: a K-step of 16 is 32 bytes along each row; MN-major: 16
            // rows, two 1024-byte row groups, and 64-wide blocks along M / N 8 KB
            // apart.  Only the address field (bytes / 16, below 2^14 since shared
            // memory is below 256 KB) moves per K-step and per ring stage, so the
            // descriptors of stage 0 are built once and offset per K-block.
            constexpr bool a_mn = MODE == TC_WGRAD;
            constexpr bool b_mn = MODE == TC_WGRAD || MODE == TC_DGRAD;
            constexpr uint32_t kStepA = a_mn ? 2048 / 16 : 32 / 16;
            constexpr uint32_t kStepB = b_mn ? 2048 / 16 : 32 / 16;
            constexpr uint32_t kStageD = C::STAGE / 16;
            const uint32_t s0 = smem_u32(smem);
            const uint64_t da_base = a_mn ? desc_sw128_mn(s0, 64 * 128) : desc_sw128(s0);
            int st = 0;          // ring stage of the next K-block
            uint32_t ph = 0;     // and the parity of the phase it waits for
            int chunk = 0;
            for (int tile = blockIdx.x; tile < args.total_tiles; tile += gridDim.x) {
                const Tile T = decode_tile(args, tile);
                // chunks of equal length (at most kChunkBlocks K-blocks each), so
                // that no short chunk costs a full drain for little MMA work
                const int cpp = (T.kb1 - T.kb0 + kChunkBlocks - 1) / kChunkBlocks;
                const int csz = cpp ? (T.kb1 - T.kb0 + cpp - 1) / cpp : 0;
                for (int la = 0; la < LA; ++la)
                for (int lb0 = 0; lb0 < lb_limit(la); lb0 += PB) {
                    const int nb = min(PB, lb_limit(la) - lb0);
                    // one MMA of width nb * N over the pass's limb tiles.  MN-major B
                    // holds [64-channel block h][PB limbs] in 8 KB blocks: the first
                    // nb limbs of a 64-wide tile are adjacent; with two channel blocks
                    // and nb < PB the used blocks are PB * 8 KB apart (leading byte
                    // offset), and their accumulators land side by side.
                    const uint32_t idesc = idesc_nb[nb];
                    const uint32_t b_lbo = (N > 64 && nb < PB) ? PB * 64 * 128 : 64 * 128;
                    const uint64_t db_base = b_mn ? desc_sw128_mn(s0 + C::A_BYTES, b_lbo)
                                                  : desc_sw128(s0 + C::A_BYTES);
                    for (int c = 0; c < cpp; ++c, ++chunk) {
                        const int buf = chunk % NBUF;
                        if (!mbar_wait(tempty_bar(buf), ((chunk / NBUF) & 1) ^ 1, abort_flag,
                                       args.status))
                            goto mma_done;
                        tc_fence_after();
                        const uint32_t d = tmem + (uint32_t)(buf * PB * N);
                        const int c0 = T.kb0 + c * csz;
                        const int c1 = min(T.kb1, c0 + csz);
                        for (int kb = c0; kb < c1; ++kb) {
                            if (!mbar_wait(full_bar(st), ph, abort_flag, args.status))
                                goto mma_done;
                            tc_fence_after();
                            const uint64_t so = (uint64_t)((uint32_t)st * kStageD);
                            const uint64_t da0 = da_base + so, db0 = db_base + so;
                            umma_bf16(d, da0, db0, idesc, kb > c0 ? 1u : 0u);
#pragma unroll
                            for (int k = 1; k < kBK / 16; ++k)
                                umma_bf16(d, da0 + k * kStepA, db0 + k * kStepB, idesc, 1u);
                            umma_commit(empty_bar(st));
                            if (++st == S) {
                                st = 0;
                                ph ^= 1u;
                            }
                        }
                        umma_commit(tfull_bar(buf));
                    }
                }
            }
        mma_done:;
            // every MMA of this CTA is issued: the next kernel in the stream
            // may start launching (its CTAs take SMs as this kernel's CTAs exit)
            pdl_trigger();
        }
    }
    } else {
        // ---------------- epilogue: warpgroups 1 and 2
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsEpilogue));
        const int q = warp & 3;                     // TMEM lane quadrant this warp may read
        const int half = (warp - kEpiWarp0) >> 2;   // which quarter of the N columns
        int chunk = 0;
        for (int tile = blockIdx.x; tile < args.total_tiles; tile += gridDim.x) {
            const Tile T = decode_tile(args, tile);
            const int cpp = (T.kb1 - T.kb0 + kChunkBlocks - 1) / kChunkBlocks;
            uint64_t acc[NH];
#pragma unroll
            for (int i = 0; i < NH; ++i) acc[i] = 0;
            for (int la = 0; la < LA; ++la)
            for (int lb0 = 0; lb0 < lb_limit(la); lb0 += PB) {
                const int nb = min(PB, lb_limit(la) - lb0);
                const int pbw = nb < PB ? nb : PB;   // MN-major: limb blocks per channel block
                const int shift0 = 8 * (la + lb0);
                for (int c = 0; c < cpp; ++c, ++chunk) {
                    const int buf = chunk % NBUF;
                    if (!mbar_wait(tfull_bar(buf), (chunk / NBUF) & 1, abort_flag, args.status))
                        goto epi_done;
                    tc_fence_after();
                    // K-major B: limb-major columns; MN-major B: 64-column blocks
                    // ordered [channel block][limb of this pass]
                    auto limb_base = [&](int jb) -> uint32_t {
                        const int hb = (half * NH) / 64;
                        const int colj = (MODE == TC_WGRAD || MODE == TC_DGRAD)
                            ? (hb * pbw + jb) * 64 + (half * NH - hb * 64)
                            : jb * N + half * NH;
                        return tmem + ((uint32_t)(32 * q) << 16) + (uint32_t)(buf * PB * N + colj);
                    };
                    // acc += v 2^shift: one 32 x 32 -> 64 multiply-add below 2^32, an
                    // add to the high word above (shift is a multiple of 8)
                    auto accumulate = [&](const uint32_t* r, int j, int shift) {
                        if (shift < 32) {
                            const int m = 1 << shift;
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                const int v = __float2int_rz(__uint_as_float(r[i]));   // exact integer
                                acc[16 * j + i] += (uint64_t)((long long)v * (long long)m);
                            }
                        } else {
#pragma unroll
                            for (int i = 0; i < 16; ++i) {
                                const int v = __float2int_rz(__uint_as_float(r[i]));
                                acc[16 * j + i] += (uint64_t)((uint32_t)v << (shift - 32)) << 32;
                            }
                        }
                    };
                    // 32 values per TMEM round trip: two loads issued back to
                    // back, then one wait (16 columns: two limbs at once)
                    if (NH == 16) {
                        for (int jb = 0; jb < nb; jb += 2) {
                            uint32_t r[32];
                            tmem_ld16_nowait(limb_base(jb), r);
                            if (jb + 1 < nb) tmem_ld16_nowait(limb_base(jb + 1), r + 16);
                            tmem_wait_ld<32>(r);
                            accumulate(r, 0, shift0 + 8 * jb);
                            if (jb + 1 < nb) accumulate(r + 16, 0, shift0 + 8 * (jb + 1));
                        }
                    } else {
                        for (int jb = 0; jb < nb; ++jb) {
                            const uint32_t base = limb_base(jb);
#pragma unroll
                            for (int j2 = 0; j2 < NH / 32; ++j2) {
                                uint32_t r[32];
                                tmem_ld16_nowait(base + 32 * j2, r);
                                tmem_ld16_nowait(base + 32 * j2 + 16, r + 16);
                                tmem_wait_ld<32>(r);
                                accumulate(r, 2 * j2, shift0 + 8 * jb);
                                accumulate(r + 16, 2 * j2 + 1, shift0 + 8 * jb);
                            }
                        }
                    }
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(tempty_bar(buf));
                }
            }
            {
                const int r = 32 * q + lane;   // output row of this thread
                const int col0 = T.nt * N + half * NH;
                if (MODE == TC_GEMM) {
                    const int m = T.mt * kBM + r;      // C[m][n], M rows in args.B
                    if (m < args.B) {
                        int64_t* o = args.out + (int64_t)m * args.ncols + col0;
#pragma unroll
                        for (int i = 0; i < NH; ++i) {
                            if (col0 + i >= args.ncols) break;
                            if (args.atomic_out)       // K split: exact 64-bit sums
                                atomicAdd(reinterpret_cast<unsigned long long*>(o + i),
                                          (unsigned long long)acc[i]);
                            else
                                o[i] = (int64_t)acc[i];
                        }
                    }
                } else if (MODE == TC_WGRAD) {
                    const int m = T.mt * kBM + r;
                    const int t = m / args.cin_k, ci = m - t * args.cin_k;
                    // im2col rows: row m is already the (tap, ci) index t Cin + ci
                    const bool ok = args.taps == 1 ? m < args.rows : (t < 9 && ci < args.Cin);
                    const int64_t wrow = args.taps == 1 ? (int64_t)m : (int64_t)t * args.Cin + ci;
                    const int64_t cstride = args.cstride;
                    if (ok) {
                        int64_t* o = args.out + wrow;
#pragma unroll
                        for (int i = 0; i < NH; ++i) {
                            if (col0 + i >= args.ncols) break;
                            unsigned long long* dst = reinterpret_cast<unsigned long long*>(
                                o + (int64_t)(col0 + i) * cstride);
                            if (args.atomic_out) atomicAdd(dst, (unsigned long long)acc[i]);
                            else *dst = acc[i];
                        }
                    }
                    if (args.sgd) {
                        // IntegerSGD (Algorithm 1) on this thread's row of NH columns,
                        // from the final sums in the accumulators (no K split)
                        {
                            uint32_t mx = 0;
                            bool ovf = false;
                            if (ok) {
                                const int tt = args.taps == 1 ? 0 : t;
                                const int64_t pcol = args.taps == 1 ? (int64_t)m : (int64_t)tt * args.tap_k + ci;
                                // 16 columns at a time: all loads of a group are issued
                                // before any store, so a group costs one memory round trip
#pragma unroll
                                for (int i0 = 0; i0 < NH; i0 += 16) {
                                    if (col0 + i0 >= args.ncols) break;   // uniform across the warp
                                    int64_t gv[16];
                                    int32_t wv[16];
#pragma unroll
                                    for (int i = 0; i < 16; ++i) {
                                        const int co = min(col0 + i0 + i, args.ncols - 1);
                                        const int64_t e = (int64_t)co * cstride + wrow;
                                        gv[i] = (int64_t)acc[i0 + i];
                                        wv[i] = args.wt[e];
                                    }
#pragma unroll
                                    for (int i = 0; i < 16; ++i) {
                                        const int co = col0 + i0 + i;
                                        if (co >= args.ncols) break;
                                        const int64_t e = (int64_t)co * cstride + wrow;
                                        const int64_t w = wv[i];
                                        int64_t d = args.trunc ? args.gdiv.trunc_div(gv[i]) : args.gdiv.floor_div(gv[i]);
                                        if (args.decay) d += args.trunc ? args.ediv.trunc_div(w) : args.ediv.floor_div(w);
                                        const int64_t nw = w - d;
                                        ovf |= !fits_i32(nw);
                                        const int32_t s32 = (int32_t)nw;
                                        args.wt[e] = s32;
                                        mx = max(mx, abs_u32(s32));
                                        if (args.wp) {
                                            // limb planes of the new weight, entry (t, ci) of row co
                                            uint16_t* pp = args.wp + (int64_t)co * args.row_k + pcol;
                                            int32_t x = s32;
#pragma unroll
                                            for (int l = 0; l < 4; ++l) {
                                                int dg;
                                                if (l < 3) {
                                                    const int rr = x & 255;
                                                    dg = rr - ((rr >> 7) << 8);
                                                    x = (x >> 8) + (rr >> 7);
                                                } else {
                                                    dg = x;
                                                }
                                                pp[l * args.w_plane] = (uint16_t)(__float_as_uint((float)dg) >> 16);
                                            }
                                        }
                                    }
                                }
                            }
#pragma unroll
                            for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, off));
                            ovf = __any_sync(0xffffffffu, ovf);
                            if (lane == 0) {
                                if (mx) atomicMax(args.maxabs_w, mx);
                                if (ovf) atomicOr(args.status, ST_OVERFLOW);
                            }
                        }
                    }
                } else if (MODE == TC_FWD && args.fuse) {
                    // z* = floor(z / SF), NITRO-ReLU piece and value, optional
                    // 2x2 max-pool across lanes; int8 outputs straight from
                    // registers (the 2x2 windows of a tile lie inside one warp:
                    // x partner lane ^ 1, y partner lane ^ wb).
                    const int mq = udiv32(args.dv_ntx, T.mt), tb = udiv32(args.dv_nty, mq);
                    const int tx = T.mt - mq * args.ntx, ty = mq - tb * args.nty;
                    const int xx = r & ((1 << args.lg_wb) - 1);
                    const int yy = (r >> args.lg_wb) & ((1 << args.lg_hb) - 1);
                    const int bbx = r >> (args.lg_wb + args.lg_hb);
                    const int x = tx * args.wb + xx, y = ty * args.hb + yy, b = tb * args.bb + bbx;
                    const bool valid = x < args.W && y < args.H && b < args.B;
                    const int C = args.Cout;
                    const int64_t zlo = args.z_lo;
                    const uint64_t zrange = (uint64_t)(args.z_hi - args.z_lo);
                    const FloorDiv32 sf32 = args.sf32;
                    const int64_t pix = ((int64_t)b * args.H + y) * args.W + x;
                    const bool anchor = valid && !(x & 1) && !(y & 1) && x + 1 < args.W && y + 1 < args.H;
                    const int64_t opix = ((int64_t)b * args.oh + (y >> 1)) * args.ow + (x >> 1);
                    const int dys = args.wb;
                    // one group of 16 columns at a time (only its packed words live)
#pragma unroll
                    for (int k = 0; k < NH / 16; ++k) {
                        if (col0 + 16 * k >= C) break;   // uniform across the warp
                        uint32_t vpk[4], rpk[4];
#pragma unroll
                        for (int g4 = 0; g4 < 4; ++g4) {
                            uint32_t vp = 0, rp = 0;
#pragma unroll
                            for (int u = 0; u < 4; ++u) {
                                // z* = floor(z / SF) = floor((z >> 8) / 9Cin).  Inside
                                // [-127 SF, 128 SF) it fits 32 bits and indexes the
                                // NITRO-ReLU table; outside, the value is flat (table
                                // ends) and only the sign picks the piece.
                                const uint64_t z = acc[16 * k + 4 * g4 + u];
                                const bool inside = z - (uint64_t)zlo < zrange;
                                const bool neg = (int32_t)(z >> 32) < 0;
                                const int zq = sf32.floor_div((int32_t)((int64_t)z >> 8));
                                const int idx = inside ? zq + 127 : (neg ? 0 : 254);
                                const int reg = inside ? (neg ? 1 : 2) : (neg ? 0 : 3);
                                rp |= (uint32_t)reg << (8 * u);
                                vp |= (uint32_t)(uint8_t)relu_tab[idx] << (8 * u);
                            }
                            vpk[g4] = vp;
                            rpk[g4] = rp;
                        }
                        const int c16 = col0 + 16 * k;
                        if (valid) st16(args.region + pix * C + c16, rpk);
                        if (!args.pool) {
                            if (valid) {
                                const int64_t o = pix * C + c16;
                                st16(args.act + o, vpk);
                                if (args.out2) st16(args.out2 + o, vpk);
                                if (args.next_nhwc) st16_bf16(args.next_nhwc + o, vpk, bf16_tab);
                            }
                        } else {
                            uint32_t opk[4], apk[4];
#pragma unroll
                            for (int g4 = 0; g4 < 4; ++g4) {
                                const uint32_t v00 = vpk[g4];
                                const uint32_t v01 = __shfl_xor_sync(0xffffffffu, v00, 1);
                                const uint32_t v10 = __shfl_xor_sync(0xffffffffu, v00, dys);
                                const uint32_t v11 = __shfl_xor_sync(0xffffffffu, v00, dys ^ 1);
                                // four windows at once, a byte each: signed maxima, then
                                // the first position (order (0,0), (0,1), (1,0), (1,1))
                                // that holds the maximum
                                const uint32_t best = __vmaxs4(__vmaxs4(v00, v01), __vmaxs4(v10, v11));
                                const uint32_t e0 = __vcmpeq4(v00, best);
                                const uint32_t e1 = __vcmpeq4(v01, best);
                                const uint32_t e2 = __vcmpeq4(v10, best);
                                uint32_t ap = 0x03030303u;
                                ap = (ap & ~e2) | (0x02020202u & e2);
                                ap = (ap & ~e1) | (0x01010101u & e1);
                                ap &= ~e0;
                                opk[g4] = best;
                                apk[g4] = ap;
                            }
                            if (anchor) {
                                const int64_t o = opix * C + c16;
                                st16(args.act + o, opk);
                                if (args.out2) st16(args.out2 + o, opk);
                                st16(args.argmax + o, apk);
                                if (args.next_nhwc) st16_bf16(args.next_nhwc + o, opk, bf16_tab);
                            }
                        }
                    }
                } else if (MODE == TC_DGRAD && args.fuse) {
                    // gradient at the lower layer's (pooled) output -> int32 with
                    // the OVERFLOW rule -> max-pool backward (to the recorded
                    // window position) -> NITRO-ReLU backward -> lower delta.
                    const int mq = udiv32(args.dv_ntx, T.mt), tb = udiv32(args.dv_nty, mq);
                    const int tx = T.mt - mq * args.ntx, ty = mq - tb * args.nty;
                    const int xx = r & ((1 << args.lg_wb) - 1);
                    const int yy = (r >> args.lg_wb) & ((1 << args.lg_hb) - 1);
                    const int bbx = r >> (args.lg_wb + args.lg_hb);
                    const int x = tx * args.wb + xx, y = ty * args.hb + yy, b = tb * args.bb + bbx;
                    const bool valid = x < args.W && y < args.H && b < args.B;
                    const int Cl = args.Cin;
                    bool ovf = false;
                    uint32_t mx = 0;
                    if (valid) {
                        const int64_t opix = ((int64_t)b * args.H + y) * args.W + x;
                        const int npos = args.low_pool ? 4 : 1;
                        int64_t ppix[4];
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            ppix[k] = args.low_pool
                                ? ((int64_t)b * args.low_h + 2 * y + (k >> 1)) * args.low_w + 2 * x + (k & 1)
                                : opix;
                        // the int32 values first (storage rule), then the argmax and
                        // region words of all the thread's channels and window positions
                        // in one batch of 16-byte loads, then per 4 channels the floor
                        // quotient by alpha_inv, the routing and the stores
                        constexpr int NG16 = NH / 16;
                        int32_t gsv[NH];
#pragma unroll
                        for (int i = 0; i < NH; ++i) {
                            const int64_t gv = (int64_t)acc[i];
                            ovf |= col0 + i < Cl && !fits_i32(gv);
                            gsv[i] = (int32_t)gv;
                        }
                        // two groups of 16 channels per batch of code loads
#pragma unroll
                        for (int kp = 0; kp < NG16; kp += 2) {
                            if (col0 + 16 * kp >= Cl) break;   // uniform across the warp
                            uint4 amv[2], rgv[2][4];
#pragma unroll
                            for (int h = 0; h < 2; ++h) {
                                const int c16 = col0 + 16 * (kp + h);
                                const bool in = kp + h < NG16 && c16 < Cl;
                                amv[h] = (args.low_pool && in)
                                    ? *reinterpret_cast<const uint4*>(args.low_argmax + opix * Cl + c16)
                                    : make_uint4(0, 0, 0, 0);
#pragma unroll
                                for (int k = 0; k < 4; ++k)
                                    rgv[h][k] = (k < npos && in)
                                        ? *reinterpret_cast<const uint4*>(args.low_region + ppix[k] * Cl + c16)
                                        : make_uint4(0, 0, 0, 0);
                            }
#pragma unroll
                            for (int h = 0; h < 2; ++h) {
                                const int k16 = kp + h;
                                const int c16 = col0 + 16 * k16;
                                if (k16 >= NG16 || c16 >= Cl) break;
                                const uint32_t amw4[4] = {amv[h].x, amv[h].y, amv[h].z, amv[h].w};
#pragma unroll
                                for (int e4 = 0; e4 < 4; ++e4) {
                                    const int c0 = c16 + 4 * e4;
                                    int32_t gs[4], gq[4];   // gradient and floor(gradient / alpha_inv)
#pragma unroll
                                    for (int e = 0; e < 4; ++e) {
                                        gs[e] = gsv[16 * k16 + 4 * e4 + e];
                                        gq[e] = args.alpha32.floor_div(gs[e]);
                                    }
                                    const uint32_t amw = amw4[e4];
#pragma unroll
                                    for (int k = 0; k < 4; ++k) {
                                        if (k >= npos) break;
                                        const uint32_t rw[4] = {rgv[h][k].x, rgv[h][k].y, rgv[h][k].z,
                                                                rgv[h][k].w};
                                        const uint32_t rgw = rw[e4];
                                        int32_t dv[4];
#pragma unroll
                                        for (int e = 0; e < 4; ++e) {
                                            const int reg = (int)((rgw >> (8 * e)) & 255u);
                                            const int am = (int)((amw >> (8 * e)) & 255u);
                                            const int32_t v = am != k ? 0 : (reg == 1 ? gq[e] : (reg == 2 ? gs[e] : 0));
                                            dv[e] = v;
                                            mx = max(mx, abs_u32(v));
                                        }
                                        *reinterpret_cast<int4*>(args.low_delta + ppix[k] * Cl + c0) =
                                            make_int4(dv[0], dv[1], dv[2], dv[3]);
                                    }
                                }
                            }
                        }
                    }
#pragma unroll
                    for (int off = 16; off; off >>= 1) mx = max(mx, __shfl_xor_sync(0xffffffffu, mx, off));
                    ovf = __any_sync(0xffffffffu, ovf);
                    if (lane == 0) {
                        if (mx) atomicMax(args.low_maxabs, mx);
                        if (ovf) atomicOr(args.status, ST_OVERFLOW);
                    }
                } else {
                    const int mq = udiv32(args.dv_ntx, T.mt), tb = udiv32(args.dv_nty, mq);
                    const int tx = T.mt - mq * args.ntx, ty = mq - tb * args.nty;
                    const int xx = r & ((1 << args.lg_wb) - 1);
                    const int yy = (r >> args.lg_wb) & ((1 << args.lg_hb) - 1);
                    const int bbx = r >> (args.lg_wb + args.lg_hb);
                    const int x = tx * args.wb + xx, y = ty * args.hb + yy, b = tb * args.bb + bbx;
                    if (x < args.W && y < args.H && b < args.B) {
                        int64_t* o = args.out + (((int64_t)b * args.H + y) * args.W + x) * args.ncols + col0;
                        if (args.out_vec && col0 + NH <= args.ncols && (args.ncols & 1) == 0) {
#pragma unroll
                            for (int i = 0; i < NH; i += 2) {
                                longlong2 v;
                                v.x = (long long)acc[i];
                                v.y = (long long)acc[i + 1];
                                *reinterpret_cast<longlong2*>(o + i) = v;
                            }
                        } else {
#pragma unroll
                            for (int i = 0; i < NH; ++i)
                                if (col0 + i < args.ncols) o[i] = (int64_t)acc[i];
                        }
                    }
                }
            }
        }
    epi_done:;
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(C::TCOLS)
                     : "memory");
    }
}

// ------------------------------------------------------------------ timeout probe
// Exercises the failure path of the bounded waits without a fault: the CTA
// holds TMEM like the contraction kernel, warp 0 waits on an mbarrier that
// nothing ever completes with a short limit, gives up, raises TIMEOUT and the
// abort flag; warps 1 and 2 wait on another such barrier under the kernel's
// normal limit and leave when they see the flag.  TMEM is then freed and the
// kernel returns, so the context stays usable.
__global__ void __launch_bounds__(96, 1) k_tc_wait_probe(uint32_t* status, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bars[2];
    __shared__ uint32_t tmem_slot;
    __shared__ int abort_s;
    volatile int* abort_flag = &abort_s;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bars[0]), 1);
        mbar_init(smem_u32(&bars[1]), 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_u32(&tmem_slot)),
                     "r"(32)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_slot;
    if (lane == 0) {
        // phase 0 of a fresh barrier never completes: both waits must give up
        if (warp == 0) mbar_wait(smem_u32(&bars[0]), 0, abort_flag, status, limit_ns);
        else mbar_wait(smem_u32(&bars[1]), 0, abort_flag, status);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(32)
                     : "memory");
    }
}

// ------------------------------------------------------------------ limb packing
__device__ __forceinline__ uint16_t bf16_bits(int v) {
    return __bfloat16_as_ushort(__float2bfloat16_rn((float)v));   // exact for |v| <= 256
}

// int8 NHWC [P][C] -> bf16 NHWC [P][Cp] copy, zero in channels C..Cp-1
__global__ void k_pack_act_nhwc(const int8_t* __restrict__ x, int64_t P, int C, int Cp,
                                uint16_t* __restrict__ out) {
    pdl_wait();
    const int64_t n = P * Cp;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = i / Cp;
        const int c = (int)(i - p * Cp);
        out[i] = c < C ? bf16_bits(x[p * C + c]) : (uint16_t)0;
    }
}

// int8 NHWC x [B][H][W][Cin] (9 Cin <= 64) -> bf16 im2col rows [B][H][W][64]:
// entry k = t Cin + ci holds x at (y + ky - 1, x + kx - 1) for tap t = 3 ky + kx,
// zero outside the image and for k >= 9 Cin.  A CTA takes one image row at a
// time: the three input rows around it (with a zero pixel on either side) are
// staged in shared memory, then each thread writes 8 entries (16 bytes).
__global__ void __launch_bounds__(256) k_pack_im2col(const int8_t* __restrict__ x, int B, int H,
                                                     int W, int Cin,
                                                     uint16_t* __restrict__ out) {
    pdl_wait();
    extern __shared__ int8_t win[];            // [3][W + 2][Cin]
    __shared__ int tab[kBK];                   // window offset of entry k, or -1
    const int rowlen = (W + 2) * Cin;
    for (int k = threadIdx.x; k < kBK; k += blockDim.x) {
        int off = -1;
        if (k < 9 * Cin) {
            const int t = k / Cin, ci = k - t * Cin;
            off = (t / 3) * rowlen + (t % 3) * Cin + ci;
        }
        tab[k] = off;
    }
    for (int64_t row = blockIdx.x; row < (int64_t)B * H; row += gridDim.x) {
        const int y = (int)(row % H);
        const int64_t b = row / H;
        __syncthreads();                       // readers of the previous row are done
        for (int i = threadIdx.x; i < 3 * rowlen; i += blockDim.x) {
            const int r = i / rowlen, rem = i - r * rowlen;
            const int px = rem / Cin - 1, ci = rem - (rem / Cin) * Cin;
            const int iy = y + r - 1;
            win[i] = (iy >= 0 && iy < H && px >= 0 && px < W)
                         ? x[((b * H + iy) * W + px) * Cin + ci]
                         : (int8_t)0;
        }
        __syncthreads();
        uint4* orow = reinterpret_cast<uint4*>(out + row * W * kBK);
        for (int i = threadIdx.x; i < W * (kBK / 8); i += blockDim.x) {
            const int px = i / (kBK / 8), k0 = (i - px * (kBK / 8)) * 8;
            const int8_t* wp = win + px * Cin;
            uint32_t w[4];
#pragma unroll
            for (int j = 0; j < 8; j += 2) {
                const int o0 = tab[k0 + j], o1 = tab[k0 + j + 1];
                const uint32_t h0 = bf16_bits(o0 >= 0 ? wp[o0] : 0);
                const uint32_t h1 = bf16_bits(o1 >= 0 ? wp[o1] : 0);
                w[j / 2] = h0 | (h1 << 16);
            }
            orow[i] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

// shared memory of k_pack_im2col's row window
inline size_t im2col_smem(int W, int Cin) { return (size_t)3 * (W + 2) * Cin; }

// int8 NHWC [P][C] -> bf16 NHWC [P][C] for C % 8 == 0: eight channels per
// thread (one 8-byte load, one 16-byte store)
__global__ void k_pack_act_nhwc8(const int8_t* __restrict__ x, int64_t n8,
                                 uint16_t* __restrict__ out) {
    pdl_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
         i += (int64_t)gridDim.x * blockDim.x) {
        const uint2 v = reinterpret_cast<const uint2*>(x)[i];
        const uint32_t in[2] = {v.x, v.y};
        uint32_t w[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const uint32_t word = in[k >> 1] >> (16 * (k & 1));
            w[k] = (uint32_t)bf16_bits((int8_t)(word & 255u)) |
                   ((uint32_t)bf16_bits((int8_t)((word >> 8) & 255u)) << 16);
        }
        reinterpret_cast<uint4*>(out)[i] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// int32 delta NHWC (n values, n % 8 == 0) -> limb planes [L][n], eight values
// per thread and one 16-byte store per plane (L from *maxabs).  The
// input is read as 16-byte words when `d` is 16-byte aligned (vec != 0).
__global__ void __launch_bounds__(256) k_pack_delta_nhwc(const int32_t* __restrict__ d, int64_t n,
                                                         int vec, const uint32_t* maxabs,
                                                         uint16_t* __restrict__ out) {
    pdl_wait();
    const int L = limb_count(*maxabs);
    const int64_t n8 = n / 8;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
         i += (int64_t)gridDim.x * blockDim.x) {
        int32_t v[8];
        if (vec) {
            const int4 a0 = reinterpret_cast<const int4*>(d)[2 * i];
            const int4 a1 = reinterpret_cast<const int4*>(d)[2 * i + 1];
            v[0] = a0.x; v[1] = a0.y; v[2] = a0.z; v[3] = a0.w;
            v[4] = a1.x; v[5] = a1.y; v[6] = a1.z; v[7] = a1.w;
        } else {
#pragma unroll
            for (int k = 0; k < 8; ++k) v[k] = d[8 * i + k];
        }
        for (int l = 0; l < L; ++l) {
            uint32_t w[4];
#pragma unroll
            for (int k = 0; k < 8; k += 2) {
                uint32_t hb[2];
#pragma unroll
                for (int u = 0; u < 2; ++u) {
                    int dg;
                    if (l < L - 1) {
                        // v = 256 q + r: digit r or r - 256, remainder q or q + 1
                        const int r = v[k + u] & 255;
                        dg = r - ((r >> 7) << 8);
                        v[k + u] = (v[k + u] >> 8) + (r >> 7);
                    } else {
                        dg = v[k + u];
                    }
                    hb[u] = __float_as_uint((float)dg) >> 16;   // exact: |dg| <= 128
                }
                w[k / 2] = hb[0] | (hb[1] << 16);
            }
            reinterpret_cast<uint4*>(out + (int64_t)l * n)[i] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}


// W [Cout][9][Cin] -> w_planes [L][Cout][row_k] with entry (t, ci) at
// t tap_k + ci (padding left zero; row_k = 9 Ck, tap_k = Ck with Ck = Cin
// rounded up to 64, or row_k = 64, tap_k = Cin for im2col rows)
__global__ void k_pack_weights(const int32_t* __restrict__ W, int Cout, int Cin, int row_k,
                               int tap_k, const uint32_t* maxabs, uint16_t* __restrict__ wp) {
    pdl_wait();
    const int L = limb_count(*maxabs);
    const int64_t n = (int64_t)Cout * 9 * Cin;
    const int64_t nk = (int64_t)Cout * row_k;
    auto split = [L](int64_t x, uint16_t* dst, int64_t plane) {
        for (int l = 0; l < L; ++l) {
            int v;
            if (l < L - 1) {
                const int64_t dg = ((x + 128) & 255) - 128;
                v = (int)dg;
                x = (x - dg) >> 8;
            } else {
                v = (int)x;
            }
            dst[l * plane] = bf16_bits(v);
        }
    };
    if (wp) {
        for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
             i += (int64_t)gridDim.x * blockDim.x) {
            const int ci = (int)(i % Cin);
            const int t = (int)((i / Cin) % 9);
            const int co = (int)(i / (9LL * Cin));
            split(W[i], wp + (int64_t)co * row_k + t * tap_k + ci, nk);
        }
    }

}

// ------------------------------------------------------------------ host side
PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// bf16 tensor map, dims innermost first; strides in elements for dims 1..r-1.
bool make_map(CUtensorMap* m, const void* base, int rank, const uint64_t* dims,
              const uint64_t* strides_elems, const uint32_t* box) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t gdim[5], gstride[4];
    cuuint32_t bdim[5], estr[5];
    for (int i = 0; i < rank; ++i) {
        gdim[i] = dims[i];
        bdim[i] = box[i];
        estr[i] = 1;
    }
    for (int i = 0; i < rank - 1; ++i) gstride[i] = strides_elems[i] * 2;
    CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, (cuuint32_t)rank, const_cast<void*>(base),
                    gdim, gstride, bdim, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

int sm_count() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess ||
            cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
            n = 148;
    }
    return n;
}

inline int log2_exact(int v) {
    int l = 0;
    while ((1 << l) < v) ++l;
    return (1 << l) == v ? l : -1;
}

template <int MODE, int N, int PB>
cudaError_t launch_gemm(const CUtensorMap& a, const CUtensorMap& b, const TcArgs& args_in,
                        cudaStream_t s) {
    using C = TcCfg<N, PB>;
    TcArgs args = args_in;
    args.dv_tn = FloorDiv32::make((uint32_t)args.tiles_n);
    args.dv_tm = FloorDiv32::make((uint32_t)args.tiles_m);
    args.dv_ntx = FloorDiv32::make((uint32_t)args.ntx);
    args.dv_nty = FloorDiv32::make((uint32_t)args.nty);
    args.lg_wb = log2_exact(args.wb);
    args.lg_hb = log2_exact(args.hb);
    if (args.tiles_n < 1 || args.tiles_m < 1 || args.ntx < 1 || args.nty < 1 || args.lg_wb < 0 ||
        args.lg_hb < 0)
        return cudaErrorInvalidValue;
    static bool attr_set = false;
    if (!attr_set) {
        // the setmaxnreg split must fit the registers the CTA is launched with,
        // else setmaxnreg.inc would wait forever: never launch such a build
        cudaFuncAttributes fa{};
        cudaError_t e = cudaFuncGetAttributes(&fa, k_tc_gemm<MODE, N, PB>);
        if (e != cudaSuccess) return e;
        if (fa.maxThreadsPerBlock < kThreads ||
            128 * kRegsProducer + 32 * kEpiWarps * kRegsEpilogue > kThreads * fa.numRegs)
            return cudaErrorInvalidConfiguration;
        e = cudaFuncSetAttribute(k_tc_gemm<MODE, N, PB>,
                                 cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const int grid = args.total_tiles < sm_count() ? args.total_tiles : sm_count();
    launch_k(k_tc_gemm<MODE, N, PB>, grid, kThreads, C::SMEM, s, a, b, args);
    return cudaGetLastError();
}

// Tile width n and B limbs per stage (pb) from the (last seen) limb count of
// B: as many limbs per stage as the operand has, up to the TMEM budget
// (pb n <= 256).  Any choice is exact; it only changes speed.
int pick_pb(int n, int limbs_hint) {
    if (n == 128) return limbs_hint > 1 ? 2 : 1;
    return limbs_hint > 2 ? 4 : (limbs_hint == 2 ? 2 : 1);
}

// The B tensor map's box spans pb limb planes (one TMA load per stage and
// 64-channel block brings all of them), so pb must match the variant.
template <int MODE>
cudaError_t launch_gemm_pb(int n, int pb, const CUtensorMap& a, const CUtensorMap& b,
                           const TcArgs& args, cudaStream_t s) {
    if (n == 128)
        return pb == 2 ? launch_gemm<MODE, 128, 2>(a, b, args, s) : launch_gemm<MODE, 128, 1>(a, b, args, s);
    if (pb == 4) return launch_gemm<MODE, 64, 4>(a, b, args, s);
    return pb == 2 ? launch_gemm<MODE, 64, 2>(a, b, args, s) : launch_gemm<MODE, 64, 1>(a, b, args, s);
}

int pick_n(int cols) { return cols % 128 == 0 ? 128 : 64; }

void pixel_tiling(const LayerGeom& g, int batch, TcArgs& a) {
    if (g.w > 8) { a.wb = 16; a.hb = 8; a.bb = 1; }
    else if (g.w > 4 || g.h > 4) { a.wb = 8; a.hb = 8; a.bb = 2; }
    else { a.wb = 4; a.hb = 4; a.bb = 8; }     // 4 x 4 maps: eight whole images per tile
    a.ntx = (g.w + a.wb - 1) / a.wb;
    a.nty = (g.h + a.hb - 1) / a.hb;
    a.tiles_m = a.ntx * a.nty * ((batch + a.bb - 1) / a.bb);
}

inline int grid1d(int64_t n) {
    int64_t g = (n + 255) / 256;
    return (int)(g < 1 ? 1 : (g > 152 * 8 ? 152 * 8 : g));
}

template <typename T>
bool dalloc(std::vector<void*>& allocs, T** p, size_t count) {
    void* q = nullptr;
    if (cudaMalloc(&q, (count ? count : 1) * sizeof(T)) != cudaSuccess) return false;
    allocs.push_back(q);
    *p = static_cast<T*>(q);
    return true;
}

inline int round_up(int v, int m) { return (v + m - 1) / m * m; }

// K split of the weight gradient: at most one wave of CTAs (every CTA one work
// unit), each split at least one exact chunk.  Returns the split count.
int wgrad_splits(int tiles, int kb_total, int* kb_per_split) {
    int splits = sm_count() / tiles;
    const int max_splits = (kb_total + kChunkBlocks - 1) / kChunkBlocks;
    splits = splits < 1 ? 1 : (splits > max_splits ? max_splits : splits);
    *kb_per_split = (kb_total + splits - 1) / splits;
    return (kb_total + *kb_per_split - 1) / *kb_per_split;
}

}  // namespace

bool tc_wgrad_fusable(const TcLayer& t, const LayerGeom& g, int batch) {
    if (!t.wgrad || batch <= 0) return false;
    const bool lin = g.kind == NITRO_LINEAR;
    const int gh = lin ? 1 : g.h, gw = lin ? batch : g.w;
    const int wb = gw <= 8 ? 8 : (gw <= 16 ? 16 : (gw <= 32 ? 32 : 64)), hb = 64 / wb;
    const int taps = (t.im2col || lin) ? 1 : 9;
    const int tiles = (taps * t.cin_k + kBM - 1) / kBM * ((g.cout + pick_n(g.cout) - 1) / pick_n(g.cout));
    const int kb_total = (lin ? 1 : batch) * ((gw + wb - 1) / wb) * ((gh + hb - 1) / hb);
    int kbs = 0;
    return wgrad_splits(tiles, kb_total, &kbs) == 1;
}

bool tc_layer_init(TcLayer& t, const LayerGeom& g, int max_batch, bool has_dgrad,
                   const uint32_t* maxabs_w, const uint32_t* maxabs_d,
                   std::vector<void*>& allocs, std::vector<void*>& host_allocs) {
    t = TcLayer();
    t.maxabs_w = maxabs_w;
    t.maxabs_d = maxabs_d;
    if (g.kind != NITRO_CONV3X3 || max_batch < 1 || !encode_fn()) return true;
    // Narrow inputs (Cin < 32, e.g. image channels) stay on the CUDA-core
    // kernels: zero-padding them to a 64-wide K-block wastes most MMA work.
    // Inputs with 9 Cin <= 64 run as one 64-wide K-block of im2col rows.
    const bool pix_ok = g.h >= 8 && g.w >= 8;
    const bool pix4 = g.h == 4 && g.w == 4;       // forward only: 4 x 4 x 8-image tiles
    const bool wide = g.cin >= 32;
    t.im2col = pix_ok && 9 * g.cin <= kBK && im2col_smem(g.w, g.cin) <= 48 * 1024;
    t.fwd = (pix_ok && (wide || t.im2col)) || (pix4 && wide);
    t.wgrad = (wide || t.im2col) && g.cout % 8 == 0;
    // the input gradient reads the forward planes, which im2col layers lay out
    // without taps
    t.dgrad = has_dgrad && pix_ok && g.cout % 8 == 0 && !t.im2col;
    t.cin8 = t.im2col ? kBK : round_up(g.cin, 8);
    t.cin_k = round_up(g.cin, 64);
    const size_t hw = (size_t)g.h * g.w;
    const size_t nwk = (size_t)g.cout * (t.im2col ? kBK : 9 * t.cin_k);
    bool ok = true;
    if (ok && (t.fwd || t.wgrad)) ok = dalloc(allocs, &t.act_nhwc, (size_t)max_batch * hw * t.cin8);
    if (ok && (t.wgrad || t.dgrad))
        ok = dalloc(allocs, &t.d_nhwc, (size_t)kMaxLimbs * max_batch * hw * g.cout);
    if (ok && (t.fwd || t.dgrad)) ok = dalloc(allocs, &t.w_planes, (size_t)kMaxLimbs * nwk);
    if (ok) {
        void* h = nullptr;
        ok = cudaMallocHost(&h, 2 * sizeof(uint32_t)) == cudaSuccess;
        if (ok) {
            host_allocs.push_back(h);
            t.max_host = static_cast<uint32_t*>(h);
            t.max_host[0] = t.max_host[1] = 0;
        }
    }
    if (ok && t.w_planes) ok = cudaMemset(t.w_planes, 0, (size_t)kMaxLimbs * nwk * 2) == cudaSuccess;
    return ok;
}

bool tc_linear_init(TcLayer& t, const LayerGeom& g, int max_batch, uint16_t* act_bf16,
                    const uint32_t* maxabs_w, const uint32_t* maxabs_d,
                    std::vector<void*>& allocs, std::vector<void*>& host_allocs) {
    t = TcLayer();
    t.maxabs_w = maxabs_w;
    t.maxabs_d = maxabs_d;
    if (g.kind != NITRO_LINEAR || max_batch < 1 || !act_bf16 || !encode_fn()) return true;
    // TMA strides in multiples of 16 bytes; 8-wide output channel groups
    if (g.cin % 8 != 0 || g.cout % 8 != 0) return true;
    t.wgrad = true;
    t.cin8 = g.cin;
    t.cin_k = round_up(g.cin, 64);
    t.act_nhwc = act_bf16;       // the forward's bf16 copy of the layer input
    bool ok = dalloc(allocs, &t.d_nhwc, (size_t)kMaxLimbs * max_batch * g.cout);
    if (ok) {
        void* h = nullptr;
        ok = cudaMallocHost(&h, 2 * sizeof(uint32_t)) == cudaSuccess;
        if (ok) {
            host_allocs.push_back(h);
            t.max_host = static_cast<uint32_t*>(h);
            t.max_host[0] = t.max_host[1] = 0;
        }
    }
    return ok;
}

int tc_limb_hint(const TcLayer& t, int which) {
    if (!t.own_hints) {
        const uint32_t* h = which ? t.hint_d : t.hint_w;
        return h ? limb_count(*h) : 1;
    }
    return t.max_host ? limb_count(t.max_host[which]) : 1;
}

cudaError_t tc_weights_hint(TcLayer& t, cudaStream_t s) {
    if (!t.w_planes || !t.maxabs_w || !t.own_hints) return cudaSuccess;
    // host copy of max |W|, read later as a kernel-variant hint only
    return cudaMemcpyAsync(t.max_host, t.maxabs_w, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
}

void tc_weight_planes(const TcLayer& t, const LayerGeom& g, uint16_t** planes, int64_t* plane,
                      int* row_k, int* tap_k) {
    *planes = t.w_planes;
    *row_k = t.im2col ? kBK : 9 * t.cin_k;
    *tap_k = t.im2col ? g.cin : t.cin_k;
    *plane = (int64_t)g.cout * *row_k;
}

cudaError_t tc_refresh_weights(TcLayer& t, const LayerGeom& g, const int32_t* W,
                               const uint32_t* maxabs_w, cudaStream_t s) {
    if (!t.w_planes) return cudaSuccess;
    const int64_t n = (int64_t)g.cout * 9 * g.cin;
    {
        ProfScope ps(K_TC_PACK_W, s, 0.0, (double)n * 4 * 2);
        const int row_k = t.im2col ? kBK : 9 * t.cin_k, tap_k = t.im2col ? g.cin : t.cin_k;
        launch_k(k_pack_weights, grid1d(n), 256, 0, s, W, g.cout, g.cin, row_k, tap_k, maxabs_w,
                                                 t.w_planes);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !t.own_hints) return e;
    return cudaMemcpyAsync(t.max_host, maxabs_w, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
}

cudaError_t tc_pack_input(TcLayer& t, const LayerGeom& g, const int8_t* x, int batch,
                          bool nhwc_done, cudaStream_t s) {
    if (batch <= 0 || !t.act_nhwc || nhwc_done) return cudaSuccess;
    const int64_t P = (int64_t)batch * g.h * g.w;
    if (t.im2col) {
        ProfScope ps(K_TC_PACK_X, s, 0.0, (double)P * (g.cin + 2 * kBK));
        const int64_t rows = (int64_t)batch * g.h;
        const int grid = (int)(rows < 152 * 8 ? rows : 152 * 8);
        launch_k(k_pack_im2col, grid, 256, im2col_smem(g.w, g.cin), s, x, batch, g.h, g.w, g.cin,
                                                                 t.act_nhwc);
        return cudaGetLastError();
    }
    ProfScope ps(K_TC_PACK_X, s, 0.0, (double)P * (g.cin + 2 * t.cin8));
    if (g.cin == t.cin8 && g.cin % 8 == 0 && ((uintptr_t)x & 7) == 0) {
        launch_k(k_pack_act_nhwc8, grid1d(P * g.cin / 8), 256, 0, s, x, P * g.cin / 8, t.act_nhwc);
        return cudaGetLastError();
    }
    launch_k(k_pack_act_nhwc, grid1d(P * t.cin8), 256, 0, s, x, P, g.cin, t.cin8, t.act_nhwc);
    return cudaGetLastError();
}

cudaError_t tc_conv_forward(TcLayer& t, const LayerGeom& g, int batch, int64_t* z,
                            const TcFwdOut* fo, uint32_t* status, cudaStream_t s, bool* done,
                            bool* fused) {
    *done = false;
    *fused = false;
    if (!t.fwd || batch <= 0) return cudaSuccess;
    TcArgs a{};
    a.B = batch; a.H = g.h; a.W = g.w; a.Cin = g.cin; a.Cout = g.cout;
    a.Bp = round_up(batch, 8);
    a.cin_k = t.cin_k;
    a.taps = t.im2col ? 1 : 9;
    pixel_tiling(g, batch, a);
    const int n = pick_n(g.cout);
    a.tiles_n = (g.cout + n - 1) / n;
    a.total_tiles = a.tiles_m * a.tiles_n;
    a.kb_total = a.taps * (t.cin_k / kBK);
    a.kb_per_split = a.kb_total;
    a.ncols = g.cout;
    a.max_a = nullptr;
    a.max_b = t.maxabs_w;
    a.out = z;
    a.out_vec = ((uintptr_t)z & 15) == 0;
    a.status = status;
    a.atomic_out = 0;
    if (fo && g.cout % 16 == 0) {
        a.fuse = 1;
        const int64_t sf = 256LL * 9LL * g.cin;
        a.sf32 = FloorDiv32::make(9u * (uint32_t)g.cin);
        a.z_hi = 128 * sf;
        a.z_lo = -127 * sf;
        a.alpha = FloorDiv::make((uint64_t)fo->alpha_inv);
        a.mu = fo->mu;
        a.pool = g.pool;
        a.oh = g.oh;
        a.ow = g.ow;
        a.act = fo->act;
        a.out2 = fo->out2;
        a.region = fo->region;
        a.argmax = fo->argmax;
        a.next_nhwc = fo->next_nhwc;
    }
    CUtensorMap ma, mb;
    const uint64_t da[4] = {(uint64_t)t.cin8, (uint64_t)g.w, (uint64_t)g.h, (uint64_t)batch};
    const uint64_t sa[3] = {(uint64_t)t.cin8, (uint64_t)g.w * t.cin8, (uint64_t)g.h * g.w * t.cin8};
    const uint32_t ba[4] = {64, (uint32_t)a.wb, (uint32_t)a.hb, (uint32_t)a.bb};
    const uint64_t kw = (uint64_t)a.taps * t.cin_k;   // w_planes row length
    const int pb = pick_pb(n, tc_limb_hint(t, 0));
    const uint64_t db[3] = {kw, (uint64_t)g.cout, (uint64_t)kMaxLimbs};
    const uint64_t sb[2] = {kw, kw * g.cout};
    const uint32_t bb[3] = {64, (uint32_t)n, (uint32_t)pb};
    if (!make_map(&ma, t.act_nhwc, 4, da, sa, ba) || !make_map(&mb, t.w_planes, 3, db, sb, bb))
        return cudaErrorInvalidValue;
    const double ops = 2.0 * batch * g.h * g.w * g.cout * 9.0 * g.cin;
    ProfScope ps(K_TC_CONV_FWD, s, ops, 0.0);
    cudaError_t e = launch_gemm_pb<TC_FWD>(n, pb, ma, mb, a, s);
    if (e == cudaSuccess) {
        *done = true;
        *fused = a.fuse != 0;
    }
    return e;
}

cudaError_t tc_pack_delta(TcLayer& t, const LayerGeom& g, const int32_t* delta,
                          const uint32_t* maxabs_delta, int batch, cudaStream_t s,
                          bool planes_done) {
    if (batch <= 0 || (!t.wgrad && !t.dgrad)) return cudaSuccess;
    // limb planes of delta (NHWC, read by the wgrad and dgrad passes), unless
    // an earlier call split this delta already
    const int64_t n = (int64_t)batch * g.h * g.w * g.cout;   // cout % 8 == 0
    if (!planes_done) {
        ProfScope ps(K_TC_PACK_D, s, 0.0, (double)n * 4 * 2);
        launch_k(k_pack_delta_nhwc, grid1d(n / 8), 256, 0, s, delta, n, ((uintptr_t)delta & 15) == 0,
                                                       maxabs_delta, t.d_nhwc);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !t.own_hints) return e;
    return cudaMemcpyAsync(t.max_host + 1, maxabs_delta, sizeof(uint32_t), cudaMemcpyDeviceToHost, s);
}

cudaError_t tc_conv_wgrad(TcLayer& t, const LayerGeom& g, const int32_t* delta,
                          const uint32_t* maxabs_delta, int batch, int64_t* dW,
                          uint32_t* status, cudaStream_t s, bool* done, bool planes_done,
                          const TcSgd* sgd, bool* sgd_done) {
    *done = false;
    if (sgd_done) *sgd_done = false;
    if (batch <= 0 || (!t.wgrad && !t.dgrad)) return cudaSuccess;
    cudaError_t pe = tc_pack_delta(t, g, delta, maxabs_delta, batch, s, planes_done);
    if (pe != cudaSuccess) return pe;
    if (!t.wgrad) return cudaSuccess;
    // A linear layer is one image of height 1 and width `batch` with a single
    // centred tap: rows = input features, K = the samples.
    const bool lin = g.kind == NITRO_LINEAR;
    const int nimg = lin ? 1 : batch, gh = lin ? 1 : g.h, gw = lin ? batch : g.w;
    const int hw = gh * gw;
    TcArgs a{};
    a.B = nimg; a.H = gh; a.W = gw; a.Cin = g.cin; a.Cout = g.cout;
    a.Bp = round_up(nimg, 8);
    a.cin_k = t.cin_k;
    a.taps = (t.im2col || lin) ? 1 : 9;
    a.rows = lin ? g.cin : 9 * g.cin;
    a.cstride = lin ? (int64_t)g.cin : 9LL * g.cin;
    // K-blocks: 64-pixel boxes (wb x hb) of one image
    a.wb = gw <= 8 ? 8 : (gw <= 16 ? 16 : (gw <= 32 ? 32 : 64));
    a.hb = 64 / a.wb;
    a.bb = 1;
    a.ntx = (gw + a.wb - 1) / a.wb;
    a.nty = (gh + a.hb - 1) / a.hb;
    const int n = pick_n(g.cout);
    a.tiles_m = (a.taps * t.cin_k + kBM - 1) / kBM;
    a.tiles_n = (g.cout + n - 1) / n;
    a.kb_total = nimg * a.ntx * a.nty;
    int splits = wgrad_splits(a.tiles_m * a.tiles_n, a.kb_total, &a.kb_per_split);
    a.total_tiles = a.tiles_m * a.tiles_n * splits;
    a.ncols = g.cout;
    a.max_a = nullptr;
    a.max_b = maxabs_delta;
    a.out = dW;
    a.status = status;
    a.atomic_out = splits > 1;
    // The update is folded in only without a K split: the sums are then final
    // in the accumulators.  With a split, the warp that completes an output
    // slot would have to read its sums back and update after every other
    // split has arrived; that tail measured ~50 us per launch on the VGG-style
    // step against ~7 us for the block's separate IntegerSGD launch, so split
    // layers report *sgd_done = false and are updated by IntegerSGD.
    if (sgd && sgd_done) *sgd_done = !a.atomic_out;
    if (sgd && a.atomic_out) sgd = nullptr;
    if (sgd) {
        if (sgd->gamma_inv < 1 || sgd->eta_inv < 0) return cudaErrorInvalidValue;
        a.sgd = 1;
        a.wt = sgd->W;
        a.maxabs_w = sgd->maxabs_w;
        a.gdiv = FloorDiv::make((uint64_t)sgd->gamma_inv);
        a.decay = sgd->eta_inv > 0;
        a.ediv = FloorDiv::make(sgd->eta_inv > 0 ? (uint64_t)sgd->eta_inv : 1);
        a.trunc = sgd->trunc;
        a.wp = sgd->planes;
        a.w_plane = sgd->plane;
        a.row_k = sgd->row_k;
        a.tap_k = sgd->tap_k;
    }
    CUtensorMap ma, mb;
    const uint64_t da[4] = {(uint64_t)t.cin8, (uint64_t)gw, (uint64_t)gh, (uint64_t)nimg};
    const uint64_t sa[3] = {(uint64_t)t.cin8, (uint64_t)gw * t.cin8, (uint64_t)hw * t.cin8};
    const uint32_t ba[4] = {64, (uint32_t)a.wb, (uint32_t)a.hb, 1};
    const uint64_t db[5] = {(uint64_t)g.cout, (uint64_t)gw, (uint64_t)gh, (uint64_t)nimg,
                            (uint64_t)kMaxLimbs};
    const uint64_t sb[4] = {(uint64_t)g.cout, (uint64_t)gw * g.cout, (uint64_t)hw * g.cout,
                            (uint64_t)nimg * hw * g.cout};
    const int pb = pick_pb(n, tc_limb_hint(t, 1));
    const uint32_t bb[5] = {64, (uint32_t)a.wb, (uint32_t)a.hb, 1, (uint32_t)pb};
    if (!make_map(&ma, t.act_nhwc, 4, da, sa, ba) || !make_map(&mb, t.d_nhwc, 5, db, sb, bb))
        return cudaErrorInvalidValue;
    if (a.atomic_out) {
        cudaError_t e = cudaMemsetAsync(dW, 0, sizeof(int64_t) * (size_t)a.cstride * g.cout, s);
        if (e != cudaSuccess) return e;
    }
    const double ops = 2.0 * nimg * hw * g.cout * (double)a.cstride;
    ProfScope ps(lin ? K_TC_LIN_WGRAD : K_TC_CONV_WGRAD, s, ops, 0.0);
    cudaError_t e = launch_gemm_pb<TC_WGRAD>(n, pb, ma, mb, a, s);
    if (e == cudaSuccess) *done = true;
    return e;
}

cudaError_t tc_conv_dgrad(TcLayer& t, const LayerGeom& g, int batch, int64_t* g64,
                          const TcDgradOut* fo, uint32_t* status, cudaStream_t s, bool* done,
                          bool* fused) {
    *done = false;
    *fused = false;
    if (!t.dgrad || batch <= 0) return cudaSuccess;
    TcArgs a{};
    a.B = batch; a.H = g.h; a.W = g.w; a.Cin = g.cin; a.Cout = g.cout;
    a.Bp = round_up(batch, 8);
    a.cin_k = t.cin_k;
    a.taps = 9;
    pixel_tiling(g, batch, a);
    const int n = pick_n(g.cin);
    a.tiles_n = (g.cin + n - 1) / n;
    a.total_tiles = a.tiles_m * a.tiles_n;
    a.kb_total = 9 * ((g.cout + kBK - 1) / kBK);
    a.kb_per_split = a.kb_total;
    a.ncols = g.cin;
    a.max_a = t.maxabs_d;
    a.max_b = t.maxabs_w;
    a.out = g64;
    a.out_vec = ((uintptr_t)g64 & 15) == 0;
    a.status = status;
    a.atomic_out = 0;
    if (fo && g.cin % 16 == 0) {
        a.fuse = 1;
        a.alpha32 = FloorDiv32::make((uint32_t)fo->alpha_inv);
        a.bound_a = fo->maxabs_delta;
        a.bound_b = fo->maxabs_w;
        a.low_h = fo->low_h;
        a.low_w = fo->low_w;
        a.low_pool = fo->low_pool;
        a.low_region = fo->low_region;
        a.low_argmax = fo->low_argmax;
        a.low_delta = fo->low_delta;
        a.low_maxabs = fo->low_maxabs;
        if (fo->low_pool && ((fo->low_h & 1) || (fo->low_w & 1))) {   // rows the pool dropped
            cudaError_t e = cudaMemsetAsync(fo->low_delta, 0,
                                            sizeof(int32_t) * (size_t)batch * fo->low_h * fo->low_w * g.cin, s);
            if (e != cudaSuccess) return e;
        }
    }
    CUtensorMap ma, mb;
    const uint64_t da[5] = {(uint64_t)g.cout, (uint64_t)g.w, (uint64_t)g.h, (uint64_t)batch,
                            (uint64_t)kMaxLimbs};
    // limb planes are batch-sized at this call's batch
    const uint64_t plane = (uint64_t)batch * g.h * g.w * g.cout;
    const uint64_t sa[4] = {(uint64_t)g.cout, (uint64_t)g.w * g.cout, (uint64_t)g.h * g.w * g.cout,
                            plane};
    const uint32_t ba[5] = {64, (uint32_t)a.wb, (uint32_t)a.hb, (uint32_t)a.bb, 1};
    // forward planes [L][Cout][9][Cin64], read MN-major: boxes of 64 ci x 64 co
    const uint64_t db[4] = {(uint64_t)t.cin_k, 9, (uint64_t)g.cout, (uint64_t)kMaxLimbs};
    const uint64_t sb[3] = {(uint64_t)t.cin_k, (uint64_t)9 * t.cin_k, (uint64_t)9 * t.cin_k * g.cout};
    const int pb = pick_pb(n, tc_limb_hint(t, 0));
    const uint32_t bb[4] = {64, 1, 64, (uint32_t)pb};
    if (!make_map(&ma, t.d_nhwc, 5, da, sa, ba) || !make_map(&mb, t.w_planes, 4, db, sb, bb))
        return cudaErrorInvalidValue;
    const double ops = 2.0 * batch * g.h * g.w * g.cin * 9.0 * g.cout;
    ProfScope ps(K_TC_CONV_DGRAD, s, ops, 0.0);
    cudaError_t e = launch_gemm_pb<TC_DGRAD>(n, pb, ma, mb, a, s);
    if (e == cudaSuccess) {
        *done = true;
        *fused = a.fuse != 0;
    }
    return e;
}

cudaError_t tc_timeout_probe(uint32_t* status, uint64_t limit_ns, cudaStream_t s) {
    ProfScope ps(K_TC_PROBE, s, 0.0, 0.0);
    k_tc_wait_probe<<<1, 96, 0, s>>>(status, limit_ns);
    return cudaGetLastError();
}

// ------------------------------------------------------------------ plain GEMM
namespace {
__global__ void k_maxabs(const int32_t* __restrict__ x, int64_t n, uint32_t* out) {
    pdl_wait();
    uint32_t m = 0;
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        m = max(m, abs_u32(x[i]));
#pragma unroll
    for (int off = 16; off; off >>= 1) m = max(m, __shfl_xor_sync(0xffffffffu, m, off));
    if ((threadIdx.x & 31) == 0 && m) atomicMax(out, m);
}
}  // namespace

cudaError_t tc_maxabs(const int32_t* x, int64_t n, uint32_t* out, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(out, 0, sizeof(uint32_t), s);
    if (e != cudaSuccess || n <= 0) return e;
    ProfScope ps(K_TC_PACK, s, 0.0, (double)n * 4);
    launch_k(k_maxabs, grid1d(n), 256, 0, s, x, n, out);
    return cudaGetLastError();
}

cudaError_t tc_pack_int8(const int8_t* x, int64_t rows, int cols, uint16_t* out, cudaStream_t s) {
    if (rows <= 0) return cudaSuccess;
    ProfScope ps(K_TC_PACK, s, 0.0, (double)rows * cols * 3);
    launch_k(k_pack_act_nhwc, grid1d(rows * cols), 256, 0, s, x, rows, cols, cols, out);
    return cudaGetLastError();
}

cudaError_t tc_pack_limbs(const int32_t* x, int64_t n, const uint32_t* maxabs, uint16_t* planes,
                          cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    ProfScope ps(K_TC_PACK, s, 0.0, (double)n * 4 * 2);
    launch_k(k_pack_delta_nhwc, grid1d(n / 8), 256, 0, s, x, n, ((uintptr_t)x & 15) == 0, maxabs, planes);
    return cudaGetLastError();
}

cudaError_t tc_gemm_run(const uint16_t* a_bf16, const uint16_t* b_planes, int M, int N, int K,
                        const uint32_t* max_b, int64_t* out, uint32_t* status, cudaStream_t s) {
    if (M <= 0 || N <= 0) return cudaSuccess;
    TcArgs a{};
    a.B = M;
    a.ncols = N;
    a.ntx = a.nty = 1;
    a.wb = a.hb = a.bb = 1;
    const int n = pick_n(N);
    a.tiles_m = (M + kBM - 1) / kBM;
    a.tiles_n = (N + n - 1) / n;
    a.kb_total = (K + kBK - 1) / kBK;
    // few output tiles (a batch of 64 against a linear layer): split K so that
    // about one wave of CTAs runs, at least four K-blocks per split, partial
    // sums added with 64-bit atomics into a zeroed C
    const int tiles = a.tiles_m * a.tiles_n;
    int splits = sm_count() / tiles;
    const int max_splits = (a.kb_total + 3) / 4;
    splits = splits < 1 ? 1 : (splits > max_splits ? max_splits : splits);
    a.kb_per_split = (a.kb_total + splits - 1) / splits;
    splits = (a.kb_total + a.kb_per_split - 1) / a.kb_per_split;
    a.total_tiles = tiles * splits;
    a.atomic_out = splits > 1;
    a.max_a = nullptr;
    a.max_b = max_b;
    a.out = out;
    a.status = status;
    if (a.atomic_out) {
        cudaError_t e = cudaMemsetAsync(out, 0, sizeof(int64_t) * (size_t)M * N, s);
        if (e != cudaSuccess) return e;
    }
    CUtensorMap ma, mb;
    const uint64_t da[2] = {(uint64_t)K, (uint64_t)M};
    const uint64_t sa[1] = {(uint64_t)K};
    const uint32_t ba[2] = {64, 128};
    const uint64_t db[3] = {(uint64_t)K, (uint64_t)N, (uint64_t)kMaxLimbs};
    const uint64_t sb[2] = {(uint64_t)K, (uint64_t)K * N};
    const uint32_t bb[3] = {64, (uint32_t)n, 1};
    if (!make_map(&ma, a_bf16, 2, da, sa, ba) || !make_map(&mb, b_planes, 3, db, sb, bb))
        return cudaErrorInvalidValue;
    ProfScope ps(K_TC_GEMM, s, 2.0 * M * N * (double)K, 0.0);
    return launch_gemm_pb<TC_GEMM>(n, 1, ma, mb, a, s);
}

}  // namespace nitro
