// Per-launch-site device timing with CUDA events (see jab_timing_* in include/jab.h).
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "../../include/jab.h"
#include "timing.h"

namespace jab {
namespace {

struct Pending {
  const char* name;
  cudaEvent_t a, b;
  int kernels;
};
struct Total {
  double ms = 0.0;
  int64_t ranges = 0, kernels = 0;
};

std::mutex mu;
bool on = false;
std::vector<Pending> pending;
std::vector<cudaEvent_t> pool;
std::vector<std::string> order;
std::map<std::string, Total> totals;

cudaEvent_t take_event() {
  if (!pool.empty()) {
    cudaEvent_t e = pool.back();
    pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

}  // namespace

bool timing_on() {
  std::lock_guard<std::mutex> lk(mu);
  return on;
}

TimedSite::TimedSite(const char* name, cudaStream_t st, int kernels)
    : name_(name), st_(st), kernels_(kernels) {
  std::lock_guard<std::mutex> lk(mu);
  if (!on) return;
  a_ = take_event();
  b_ = take_event();
  if (a_) cudaEventRecord(a_, st_);
}

TimedSite::~TimedSite() {
  if (!a_ || !b_) return;
  cudaEventRecord(b_, st_);
  std::lock_guard<std::mutex> lk(mu);
  pending.push_back({name_, a_, b_, kernels_});
}

}  // namespace jab

using namespace jab;

extern "C" {

jab_status jab_timing_enable(int32_t enable) {
  std::lock_guard<std::mutex> lk(mu);
  on = enable != 0;
  return JAB_OK;
}

jab_status jab_timing_collect(void) {
  std::lock_guard<std::mutex> lk(mu);
  jab_status st = JAB_OK;
  for (const Pending& p : pending) {
    float ms = 0.f;
    if (cudaEventSynchronize(p.b) != cudaSuccess || cudaEventElapsedTime(&ms, p.a, p.b) != cudaSuccess)
      st = JAB_ERR_CUDA;
    const std::string key(p.name);
    if (!totals.count(key)) order.push_back(key);
    Total& t = totals[key];
    t.ms += ms;
    t.ranges += 1;
    t.kernels += p.kernels;
    pool.push_back(p.a);
    pool.push_back(p.b);
  }
  pending.clear();
  return st;
}

int32_t jab_timing_count(void) {
  std::lock_guard<std::mutex> lk(mu);
  return (int32_t)order.size();
}

jab_status jab_timing_get(int32_t i, const char** name, double* total_ms, int64_t* ranges,
                          int64_t* kernels) {
  std::lock_guard<std::mutex> lk(mu);
  if (i < 0 || i >= (int32_t)order.size()) return JAB_ERR_INVALID_ARG;
  const Total& t = totals[order[i]];
  if (name) *name = order[i].c_str();
  if (total_ms) *total_ms = t.ms;
  if (ranges) *ranges = t.ranges;
  if (kernels) *kernels = t.kernels;
  return JAB_OK;
}

jab_status jab_timing_reset(void) {
  std::lock_guard<std::mutex> lk(mu);
  totals.clear();
  order.clear();
  return JAB_OK;
}

}  // extern "C"
