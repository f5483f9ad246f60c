// Launch counter and per-kernel CUDA-event timing (see prof.cuh) plus the
// diagnostic ABI calls that read them; the launch policy switch (programmatic
// dependent launch, NITRO_PDL=0 turns it off).
#include <atomic>
#include <cstdlib>
#include <mutex>
#include <vector>

#include "nitro.h"
#include "prof.cuh"

namespace nitro {
namespace {

constexpr int kMaxRecords = 1 << 16;

struct Record {
    int id;
    double ops, bytes;
    cudaEvent_t a, b;
};

std::atomic<uint64_t> g_launches{0};
std::atomic<int> g_enabled{0};
std::mutex g_mu;
std::vector<Record> g_records;      // recorded since the last reset
std::vector<cudaEvent_t> g_pool;    // events free for reuse

cudaEvent_t take_event() {
    if (!g_pool.empty()) {
        cudaEvent_t e = g_pool.back();
        g_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

const char* const kNames[K_COUNT] = {
    "simt_conv_fwd", "simt_conv_dgrad", "simt_conv_wgrad", "simt_linear_fwd",
    "simt_linear_dgrad", "simt_linear_wgrad", "fwd_epilogue", "learn_partial",
    "learn_dw", "grad_to_delta", "integersgd", "learn_finish_loss", "tc_conv_fwd",
    "tc_conv_wgrad", "tc_conv_dgrad", "tc_pack_limbs", "tc_finish", "tc_gemm", "lr_backward",
    "tc_pack_weights", "tc_pack_input", "tc_pack_delta", "prep_sum", "prep_mad",
    "prep_apply", "lr_pool", "lrpool_to_delta", "tc_timeout_probe", "tc_linear_wgrad"};

}  // namespace

const char* kernel_name(int id) { return (id >= 0 && id < K_COUNT) ? kNames[id] : "?"; }

bool pdl_enabled() {
    static const bool on = [] {
        const char* e = std::getenv("NITRO_PDL");
        return !(e && e[0] == '0');
    }();
    return on;
}

ProfScope::ProfScope(int id, cudaStream_t s, double ops, double bytes) : slot_(-1), s_(s) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (!g_enabled.load(std::memory_order_relaxed)) return;
    std::lock_guard<std::mutex> lk(g_mu);
    if ((int)g_records.size() >= kMaxRecords) return;
    Record r{id, ops, bytes, take_event(), take_event()};
    if (!r.a || !r.b) return;
    if (cudaEventRecord(r.a, s) != cudaSuccess) return;
    slot_ = (int)g_records.size();
    g_records.push_back(r);
}

ProfScope::~ProfScope() {
    if (slot_ < 0) return;
    std::lock_guard<std::mutex> lk(g_mu);
    cudaEventRecord(g_records[slot_].b, s_);
}

}  // namespace nitro

using namespace nitro;

extern "C" {

uint64_t nitro_kernel_launches(void) { return g_launches.load(); }

void nitro_profile_enable(int on) { g_enabled.store(on ? 1 : 0); }

void nitro_profile_reset(void) {
    std::lock_guard<std::mutex> lk(g_mu);
    for (Record& r : g_records) {
        g_pool.push_back(r.a);
        g_pool.push_back(r.b);
    }
    g_records.clear();
}

int nitro_profile_kernel_count(void) { return K_COUNT; }

const char* nitro_profile_kernel_name(int id) { return kernel_name(id); }

nitro_status nitro_profile_read(int id, uint64_t* launches, double* ms, double* ops,
                                double* bytes) {
    if (id < 0 || id >= K_COUNT || !launches || !ms || !ops || !bytes) return NITRO_ERR_ARG;
    std::lock_guard<std::mutex> lk(g_mu);
    *launches = 0;
    *ms = *ops = *bytes = 0.0;
    for (Record& r : g_records) {
        if (r.id != id) continue;
        if (cudaEventSynchronize(r.b) != cudaSuccess) return NITRO_ERR_CUDA;
        float t = 0.f;
        if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) return NITRO_ERR_CUDA;
        *launches += 1;
        *ms += t;
        *ops += r.ops;
        *bytes += r.bytes;
    }
    return NITRO_OK;
}

int nitro_profile_record_count(void) {
    std::lock_guard<std::mutex> lk(g_mu);
    return (int)g_records.size();
}

nitro_status nitro_profile_record(int i, int* kernel, double* ms, double* ops, double* bytes) {
    if (!kernel || !ms || !ops || !bytes) return NITRO_ERR_ARG;
    std::lock_guard<std::mutex> lk(g_mu);
    if (i < 0 || i >= (int)g_records.size()) return NITRO_ERR_ARG;
    Record& r = g_records[i];
    if (cudaEventSynchronize(r.b) != cudaSuccess) return NITRO_ERR_CUDA;
    float t = 0.f;
    if (cudaEventElapsedTime(&t, r.a, r.b) != cudaSuccess) return NITRO_ERR_CUDA;
    *kernel = r.id;
    *ms = t;
    *ops = r.ops;
    *bytes = r.bytes;
    return NITRO_OK;
}

}  // extern "C"
