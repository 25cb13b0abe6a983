// Optional per-launch-site CUDA-event timing (instrumentation for the benchmark; off by default).
#pragma once

#include <cuda_runtime.h>

namespace jab {

bool timing_on();
// Records a start event on construction and a stop event on destruction when timing is on.
class TimedSite {
 public:
  TimedSite(const char* name, cudaStream_t st, int kernels = 1);
  ~TimedSite();
  TimedSite(const TimedSite&) = delete;
  TimedSite& operator=(const TimedSite&) = delete;

 private:
  const char* name_;
  cudaStream_t st_;
  int kernels_;
  cudaEvent_t a_ = nullptr, b_ = nullptr;
};

}  // namespace jab
