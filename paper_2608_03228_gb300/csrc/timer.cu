// Profiling aids of the C ABI (the paper has no counterpart): a count of the
// kernels this library launches, and CUDA-event timing of selected kernel
// kinds on the stream of the call that launches them.
#include <atomic>
#include <mutex>
#include <utility>
#include <vector>

#include "common.cuh"
#include "kernels.h"

namespace saki {
namespace {

std::atomic<long long> g_launches{0};

struct TimerState {
  bool armed = false;
  int device = -1;
  std::vector<std::pair<cudaEvent_t, cudaEvent_t>> events;   // reused across arm/stop cycles
  size_t used = 0;
};
std::mutex g_mu;
TimerState g_timer[kTimedKinds];

}  // namespace

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

KernelTimer::KernelTimer(int kind, cudaStream_t s) : kind_(0), s_(s), stop_(nullptr) {
  if (kind <= 0 || kind >= kTimedKinds) return;
  std::lock_guard<std::mutex> lock(g_mu);
  TimerState& t = g_timer[kind];
  if (!t.armed) return;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return;
  if (t.device < 0) t.device = dev;
  if (dev != t.device) return;   // events belong to the device of the first timed launch
  if (t.used == t.events.size()) {
    cudaEvent_t a = nullptr, b = nullptr;
    if (cudaEventCreate(&a) != cudaSuccess) return;
    if (cudaEventCreate(&b) != cudaSuccess) {
      cudaEventDestroy(a);
      return;
    }
    t.events.emplace_back(a, b);
  }
  const auto& ev = t.events[t.used];
  if (cudaEventRecord(ev.first, s) != cudaSuccess) return;
  ++t.used;
  kind_ = kind;
  stop_ = ev.second;
}

KernelTimer::~KernelTimer() {
  if (kind_) cudaEventRecord(stop_, s_);
}

}  // namespace saki

extern "C" {

SAKI_API int64_t saki_launch_count(void) { return saki::g_launches.load(std::memory_order_relaxed); }

SAKI_API saki_status saki_kernel_timer_start(int32_t kind) {
  if (kind <= 0 || kind >= saki::kTimedKinds) return SAKI_ERR_INVALID_ARGUMENT;
  std::lock_guard<std::mutex> lock(saki::g_mu);
  saki::TimerState& t = saki::g_timer[kind];
  t.armed = true;
  t.used = 0;
  return SAKI_OK;
}

SAKI_API saki_status saki_kernel_timer_stop(int32_t kind, double* total_ms, int64_t* launches) {
  if (kind <= 0 || kind >= saki::kTimedKinds || !total_ms || !launches) return SAKI_ERR_INVALID_ARGUMENT;
  std::lock_guard<std::mutex> lock(saki::g_mu);
  saki::TimerState& t = saki::g_timer[kind];
  double sum = 0.0;
  saki_status st = SAKI_OK;
  for (size_t i = 0; i < t.used; ++i) {
    float ms = 0.f;
    if (cudaEventSynchronize(t.events[i].second) != cudaSuccess ||
        cudaEventElapsedTime(&ms, t.events[i].first, t.events[i].second) != cudaSuccess) {
      st = SAKI_ERR_CUDA;
      break;
    }
    sum += ms;
  }
  *total_ms = sum;
  *launches = (int64_t)t.used;
  t.armed = false;
  t.used = 0;
  return st;
}

}  // extern "C"
