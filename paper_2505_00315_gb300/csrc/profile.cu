// Measurement support for libmosa (not part of the layer's arithmetic): a
// count of the kernels the library has launched, and optional CUDA-event
// timing of individual stages on the stream they run on.
#include <atomic>
#include <mutex>
#include <vector>

#include "../../include/mosa.h"
#include "profile.h"

namespace mosa {
namespace {

std::atomic<unsigned long long> g_launches{0};
std::atomic<uint32_t> g_mask{0};
std::atomic<bool> g_timeline{false};
std::mutex g_mu;

struct Pending {
    int stage;
    cudaEvent_t start, stop;
    bool recycle;  // false for events owned by a captured graph
};
thread_local CaptureRecord *t_capture = nullptr;
static_assert(kNumStages <= 16, "kernel-span slots in the workspace");
thread_local unsigned long long *t_span_base = nullptr;
thread_local unsigned long long *t_active_span = nullptr;
std::vector<Pending> g_pending;
std::vector<cudaEvent_t> g_free;
double g_ms[kNumStages] = {};
int32_t g_count[kNumStages] = {};

const char *kNames[kNumStages] = {"router", "select", "qkv", "attn_fwd", "out",
                                  "out_bwd", "attn_bwd", "in_bwd", "w_bwd", "dwo",
                                  "fwd_unit", "bwd_unit"};

cudaEvent_t take_event() {
    if (!g_free.empty()) {
        cudaEvent_t e = g_free.back();
        g_free.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

// start = all ones (atomicMin target), end = 0 (atomicMax target)
__global__ void reset_spans_kernel(unsigned long long *slots, uint32_t stages) {
    const int i = threadIdx.x;
    if (i < 16 && ((stages >> i) & 1u)) {
        slots[2 * i] = ~0ull;
        slots[2 * i + 1] = 0ull;
    }
}

}  // namespace

bool timeline_on() { return g_timeline.load(std::memory_order_relaxed); }

cudaError_t begin_timeline_call(uint32_t stages, cudaStream_t s) {
    if (!timeline_on() || t_span_base == nullptr) return cudaSuccess;
    reset_spans_kernel<<<1, 32, 0, s>>>(t_span_base, stages);
    note_launches(1);
    return cudaGetLastError();
}

void note_launches(int n) {
    if (t_capture != nullptr) {
        t_capture->launches += (unsigned long long)n;
        return;
    }
    g_launches.fetch_add((unsigned long long)n, std::memory_order_relaxed);
}

void capture_into(CaptureRecord *rec) { t_capture = rec; }

uint32_t profile_mask() {
    return g_mask.load(std::memory_order_relaxed) | (timeline_on() ? 0x80000000u : 0u);
}

void replayed(const CaptureRecord &rec) {
    g_launches.fetch_add(rec.launches, std::memory_order_relaxed);
    if (rec.pairs.empty()) return;
    std::lock_guard<std::mutex> lk(g_mu);
    for (const CaptureRecord::Pair &q : rec.pairs) g_pending.push_back({q.stage, q.start, q.stop, false});
}

void set_span_base(unsigned long long *base) { t_span_base = base; }
unsigned long long *active_span() { return t_active_span; }

StageScope::StageScope(int stage, cudaStream_t s) : stage_(stage), stream_(s) {
    prev_span_ = t_active_span;
    if (!(g_mask.load(std::memory_order_relaxed) & (1u << stage))) {
        // timeline mode: the call cleared this stage's slot at its start
        if (timeline_on() && t_span_base != nullptr) t_active_span = t_span_base + 2 * stage;
        return;
    }
    if (t_span_base != nullptr) {
        // reset this stage's span slot (start = max, end = 0) ahead of its kernels
        unsigned long long *slot = t_span_base + 2 * stage;
        if (cudaMemsetAsync(slot, 0xFF, sizeof(unsigned long long), s) == cudaSuccess &&
            cudaMemsetAsync(slot + 1, 0, sizeof(unsigned long long), s) == cudaSuccess)
            t_active_span = slot;
    }
    if (t_capture != nullptr) {
        // recorded into the graph: these events live as long as the graph
        // External records become event nodes of the graph (a plain record
        // during capture would only mark a dependency inside the capture).
        if (cudaEventCreate(&start_) == cudaSuccess && cudaEventCreate(&stop_) == cudaSuccess &&
            cudaEventRecordWithFlags(start_, s, cudaEventRecordExternal) == cudaSuccess)
            active_ = true;
        return;
    }
    std::lock_guard<std::mutex> lk(g_mu);
    start_ = take_event();
    stop_ = take_event();
    if (start_ && stop_ && cudaEventRecord(start_, s) == cudaSuccess) {
        active_ = true;
    }
}

StageScope::~StageScope() {
    t_active_span = prev_span_;
    if (!active_) return;
    if (t_capture != nullptr) {
        if (cudaEventRecordWithFlags(stop_, stream_, cudaEventRecordExternal) == cudaSuccess)
            t_capture->pairs.push_back({stage_, start_, stop_});
        return;
    }
    std::lock_guard<std::mutex> lk(g_mu);
    if (cudaEventRecord(stop_, stream_) == cudaSuccess)
        g_pending.push_back({stage_, start_, stop_, true});
}

}  // namespace mosa

using namespace mosa;

extern "C" {

unsigned long long mosa_kernel_launches(void) { return g_launches.load(); }

mosa_status mosa_profile_stages(uint32_t stage_mask) {
    g_mask.store(stage_mask & ((1u << kNumStages) - 1u));
    return MOSA_OK;
}

mosa_status mosa_profile_timeline(int32_t on) {
    if (on != 0 && on != 1) return MOSA_ERR_INVALID_ARG;
    g_timeline.store(on != 0);
    return MOSA_OK;
}

int32_t mosa_profile_read(double *total_ms, int32_t *count, int32_t max_stages) {
    std::lock_guard<std::mutex> lk(g_mu);
    for (const Pending &p : g_pending) {
        float ms = 0.f;
        if (cudaEventSynchronize(p.stop) == cudaSuccess &&
            cudaEventElapsedTime(&ms, p.start, p.stop) == cudaSuccess) {
            g_ms[p.stage] += ms;
            g_count[p.stage] += 1;
        }
        if (p.recycle) {
            g_free.push_back(p.start);
            g_free.push_back(p.stop);
        }
    }
    g_pending.clear();
    const int n = max_stages < kNumStages ? max_stages : kNumStages;
    for (int i = 0; i < n; ++i) {
        if (total_ms) total_ms[i] = g_ms[i];
        if (count) count[i] = g_count[i];
    }
    for (int i = 0; i < kNumStages; ++i) {
        g_ms[i] = 0.0;
        g_count[i] = 0;
    }
    return kNumStages;
}

const char *mosa_stage_name(int32_t stage) {
    return (stage >= 0 && stage < kNumStages) ? kNames[stage] : "unknown";
}

}  // extern "C"
