// Integer data pre-processing (App. A) on the GPU.
//
// Over the n 8-bit values x of a dataset:
//   mu    = floor(sum x / n)                       k_prep_reduce<0>: byte sum
//   omega = floor(sum |x - mu| / n)                k_prep_reduce<1>: sum of
//           absolute differences to mu; its last CTA derives omega and the map
//   x_hat = clamp(floor((x - mu) 51 / omega), -127, 127), omega = 0 read as 1
//                                                  k_prep_apply: map lookup
//
// The input is 8-bit, so both sums take four bytes per instruction (__vsadu4
// adds the absolute differences of the four byte lanes; against zero it is the
// plain byte sum), and x_hat, a function of one byte, is a lookup in a
// 256-entry table held in shared memory.  Every pass streams the data with
// 16-byte loads.  The second pass walks the data backwards, so it first meets
// the part the first pass left in L2; the apply pass walks forwards again.
#include <new>

#include "nitro.h"
#include "nitro_internal.cuh"
#include "prof.cuh"

using namespace nitro;

namespace {

constexpr int kPrepThreads = 256;      // also the size of the map: one entry per thread
constexpr unsigned kAll = 0xffffffffu;

struct PrepState {
    unsigned long long sum;      // sum of x
    unsigned long long sad;      // sum of |x - mu|
    unsigned long long ticket;   // CTAs done with the second pass
    long long mu, omega;
    int8_t map[256];             // x_hat of every byte value
};

__device__ __forceinline__ unsigned long long block_sum(unsigned long long v) {
    __shared__ unsigned long long part[kPrepThreads / 32];
#pragma unroll
    for (int off = 16; off; off >>= 1) v += __shfl_xor_sync(kAll, v, off);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = v;
    __syncthreads();
    unsigned long long t = 0;
    if (threadIdx.x == 0)
        for (int w = 0; w < kPrepThreads / 32; ++w) t += part[w];
    return t;   // valid in thread 0
}

// PASS 0: st->sum += sum x.  PASS 1: st->sad += sum |x - mu| with mu from the
// finished first pass; the last CTA to finish writes mu, omega and the map.
template <int PASS>
__global__ void __launch_bounds__(kPrepThreads) k_prep_reduce(const uint8_t* __restrict__ x,
                                                              int64_t n, PrepState* st) {
    uint32_t mu = 0;
    if (PASS == 1) mu = (uint32_t)(__ldcg(&st->sum) / (unsigned long long)n);   // <= 255
    const uint32_t mu4 = mu * 0x01010101u;
    // bytes before the first 16-byte boundary, the 16-byte body, the tail
    const int64_t head = min(n, (int64_t)((16 - ((uintptr_t)x & 15)) & 15));
    const int64_t nv = (n - head) >> 4;
    const int64_t tail0 = head + (nv << 4);
    const uint4* xv = reinterpret_cast<const uint4*>(x + head);
    const int64_t tid = (int64_t)blockIdx.x * kPrepThreads + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * kPrepThreads;
    unsigned long long acc = 0;
    for (int64_t i = tid; i < nv; i += stride) {
        const uint4 v = __ldg(xv + (PASS == 1 ? nv - 1 - i : i));
        acc += (uint32_t)(__vsadu4(v.x, mu4) + __vsadu4(v.y, mu4)) +
               (uint32_t)(__vsadu4(v.z, mu4) + __vsadu4(v.w, mu4));
    }
    const int64_t ns = head + (n - tail0);   // at most 30 scalar bytes
    if (tid < ns) {
        const int64_t j = tid < head ? tid : tail0 + (tid - head);
        const int dv = (int)x[j] - (int)mu;
        acc += (unsigned long long)(dv < 0 ? -dv : dv);
    }
    const unsigned long long t = block_sum(acc);
    __shared__ bool last;
    if (threadIdx.x == 0) {
        atomicAdd(PASS == 0 ? &st->sum : &st->sad, t);
        if (PASS == 1) {
            __threadfence();
            last = atomicAdd(&st->ticket, 1ull) == (unsigned long long)gridDim.x - 1;
        }
    }
    if (PASS == 0) return;
    __syncthreads();
    if (!last) return;
    __threadfence();
    const long long omega = (long long)(__ldcg(&st->sad) / (unsigned long long)n);
    const long long div = omega > 0 ? omega : 1;
    const long long num = ((long long)threadIdx.x - (long long)mu) * 51;
    long long q = num / div;
    if (num % div != 0 && num < 0) --q;   // floor
    st->map[threadIdx.x] = (int8_t)(q < -127 ? -127 : (q > 127 ? 127 : q));
    if (threadIdx.x == 0) {
        st->mu = (long long)mu;
        st->omega = omega;
    }
}

__device__ __forceinline__ uint32_t map4(uint32_t w, const uint8_t* m) {
    return (uint32_t)m[w & 255u] | ((uint32_t)m[(w >> 8) & 255u] << 8) |
           ((uint32_t)m[(w >> 16) & 255u] << 16) | ((uint32_t)m[w >> 24] << 24);
}

// out[i] = map[x[i]].  16-byte vectors when x and out sit at the same offset
// from a 16-byte boundary; bytes otherwise.  out may equal x (each element is
// read, then written, by one thread).
__global__ void __launch_bounds__(kPrepThreads) k_prep_apply(const uint8_t* x, int64_t n,
                                                             const PrepState* __restrict__ st,
                                                             int8_t* out) {
    __shared__ uint8_t m[256];
    m[threadIdx.x] = (uint8_t)st->map[threadIdx.x];
    __syncthreads();
    const bool vec = (((uintptr_t)x ^ (uintptr_t)out) & 15) == 0;
    const int64_t head = vec ? min(n, (int64_t)((16 - ((uintptr_t)x & 15)) & 15)) : n;
    const int64_t nv = (n - head) >> 4;
    const int64_t tail0 = head + (nv << 4);
    const int64_t tid = (int64_t)blockIdx.x * kPrepThreads + threadIdx.x;
    const int64_t stride = (int64_t)gridDim.x * kPrepThreads;
    const uint4* xv = reinterpret_cast<const uint4*>(x + head);
    uint4* ov = reinterpret_cast<uint4*>(out + head);
    for (int64_t i = tid; i < nv; i += stride) {
        const uint4 v = xv[i];
        ov[i] = make_uint4(map4(v.x, m), map4(v.y, m), map4(v.z, m), map4(v.w, m));
    }
    for (int64_t j = tid; j < head; j += stride) out[j] = (int8_t)m[x[j]];
    for (int64_t j = tail0 + tid; j < n; j += stride) out[j] = (int8_t)m[x[j]];
}

int grid_for_bytes(int64_t n, int sms) {
    const int64_t want = ((n >> 4) + kPrepThreads - 1) / kPrepThreads;
    const int64_t cap = (int64_t)sms * 8;
    return (int)(want < 1 ? 1 : (want > cap ? cap : want));
}

constexpr int64_t kPrepMaxN = (int64_t)1 << 48;   // 255 n stays far inside uint64

}  // namespace

struct nitro_prep {
    PrepState* st = nullptr;
    int sms = 0;
    bool fitted = false;
};

extern "C" {

nitro_status nitro_prep_create(nitro_prep** out) {
    if (!out) return NITRO_ERR_ARG;
    *out = nullptr;
    nitro_prep* p = new (std::nothrow) nitro_prep();
    if (!p) return NITRO_ERR_CUDA;
    int dev = 0;
    bool ok = cudaGetDevice(&dev) == cudaSuccess &&
              cudaDeviceGetAttribute(&p->sms, cudaDevAttrMultiProcessorCount, dev) == cudaSuccess &&
              cudaMalloc(&p->st, sizeof(PrepState)) == cudaSuccess &&
              cudaMemset(p->st, 0, sizeof(PrepState)) == cudaSuccess;
    if (!ok) {
        if (p->st) cudaFree(p->st);
        delete p;
        return NITRO_ERR_CUDA;
    }
    *out = p;
    return NITRO_OK;
}

nitro_status nitro_prep_fit(nitro_prep* p, const uint8_t* x, int64_t n, void* stream) {
    if (!p || !x || n < 1 || n > kPrepMaxN) return NITRO_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaMemsetAsync(p->st, 0, 3 * sizeof(unsigned long long), s) != cudaSuccess)
        return NITRO_ERR_CUDA;
    const int grid = grid_for_bytes(n, p->sms);
    {
        ProfScope ps(K_PREP_SUM, s, 0.0, (double)n);
        k_prep_reduce<0><<<grid, kPrepThreads, 0, s>>>(x, n, p->st);
    }
    {
        ProfScope ps(K_PREP_MAD, s, 0.0, (double)n);
        k_prep_reduce<1><<<grid, kPrepThreads, 0, s>>>(x, n, p->st);
    }
    if (cudaGetLastError() != cudaSuccess) return NITRO_ERR_CUDA;
    p->fitted = true;
    return NITRO_OK;
}

nitro_status nitro_prep_apply(nitro_prep* p, const uint8_t* x, int64_t n, int8_t* out,
                              void* stream) {
    if (!p || !p->fitted || n < 0 || n > kPrepMaxN) return NITRO_ERR_ARG;
    if (n == 0) return NITRO_OK;
    if (!x || !out) return NITRO_ERR_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    {
        ProfScope ps(K_PREP_APPLY, s, 0.0, 2.0 * (double)n);
        k_prep_apply<<<grid_for_bytes(n, p->sms), kPrepThreads, 0, s>>>(x, n, p->st, out);
    }
    return cudaGetLastError() == cudaSuccess ? NITRO_OK : NITRO_ERR_CUDA;
}

nitro_status nitro_prep_stats(nitro_prep* p, int64_t* mu, int64_t* omega) {
    if (!p || !p->fitted || !mu || !omega) return NITRO_ERR_ARG;
    long long v[2];
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpy(v, &p->st->mu, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess)
        return NITRO_ERR_CUDA;
    *mu = v[0];
    *omega = v[1];
    return NITRO_OK;
}

void nitro_prep_destroy(nitro_prep* p) {
    if (!p) return;
    cudaFree(p->st);
    delete p;
}

}  // extern "C"
