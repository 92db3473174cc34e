// Internal hooks of the measurement support in profile.cu.
#pragma once

#include <cuda_runtime.h>

#include <vector>

namespace mosa {

enum Stage : int {
    kStageRouter = 0, kStageSelect, kStageQkv, kStageAttnFwd, kStageOut,
    kStageOutBwd, kStageAttnBwd, kStageInBwd, kStageWBwd, kStageDwo,
    kStageFwdUnit,  // F3 + F4 + F5 fused (k <= 128)
    kStageBwdUnit,  // B1 (G, row terms) + B2 fused (k <= 128)
    kNumStages
};

// Adds n to the library's kernel-launch counter (or, while this thread is
// capturing a graph, to the capture's own count).
void note_launches(int n);

// Stage-timing event pairs and kernel count recorded while a graph is being
// captured; they belong to the graph and are re-armed on every replay.
struct CaptureRecord {
    struct Pair {
        int stage;
        cudaEvent_t start, stop;
    };
    std::vector<Pair> pairs;
    unsigned long long launches = 0;
};
// Routes StageScope and note_launches of this thread into `rec` (nullptr ends).
void capture_into(CaptureRecord *rec);
// Accounts one replay of a captured graph: its kernels and its timing pairs.
void replayed(const CaptureRecord &rec);
// Stage-timing mask currently in force.
uint32_t profile_mask();

// Timeline mode (mosa_profile_timeline): every stage records its kernel span
// without CUDA events or per-stage slot resets; each layer call clears its
// stages' slots once, at its start, with begin_timeline_call.
bool timeline_on();
// Clears the span slots of the stages in `stages` (bit mask) on stream s when
// timeline mode is on (launches one small kernel); otherwise does nothing.
cudaError_t begin_timeline_call(uint32_t stages, cudaStream_t s);

// Kernel spans: the layer call names its workspace's span slots ([stage][2]);
// while a timed stage is open, active_span() is its slot (else nullptr) and
// the launchers pass it to their kernels.
void set_span_base(unsigned long long *base);
unsigned long long *active_span();

// Records a CUDA event pair around one stage when that stage's timing is on.
class StageScope {
  public:
    StageScope(int stage, cudaStream_t s);
    ~StageScope();
    StageScope(const StageScope &) = delete;
    StageScope &operator=(const StageScope &) = delete;

  private:
    int stage_;
    cudaStream_t stream_;
    cudaEvent_t start_ = nullptr, stop_ = nullptr;
    bool active_ = false;
    unsigned long long *prev_span_ = nullptr;
};

}  // namespace mosa
