// Internal hooks of the measurement support in profile.cu.
#pragma once

#include <cuda_runtime.h>

namespace mosa {

enum Stage : int {
    kStageRouter = 0, kStageSelect, kStageQkv, kStageAttnFwd, kStageOut,
    kStageOutBwd, kStageAttnBwd, kStageInBwd, kStageWBwd, kStageRows, kNumStages
};

// Adds n to the library's kernel-launch counter.
void note_launches(int n);

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
};

}  // namespace mosa
