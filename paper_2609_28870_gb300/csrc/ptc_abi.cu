// C-ABI entry points that belong to no stage, and the launch timer.
#include <atomic>
#include <cstring>
#include <map>
#include <mutex>
#include <string>
#include <vector>

#include "ptc_internal.h"

namespace ptc {
namespace {
struct Pending {
  const char* name;
  cudaEvent_t a, b;
};
struct Timer {
  std::mutex mu;
  bool on = false;
  std::vector<cudaEvent_t> pool;
  std::vector<Pending> pending;
  const char* open_name = nullptr;
  cudaEvent_t open_a = nullptr;
  std::map<std::string, std::pair<uint64_t, double>> totals;
};
Timer& timer() {
  static Timer t;
  return t;
}
std::atomic<uint64_t> g_launches{0};
cudaEvent_t take_event(Timer& t) {
  if (!t.pool.empty()) {
    cudaEvent_t e = t.pool.back();
    t.pool.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}
}  // namespace

void timer_launch_begin(const char* name, cudaStream_t s) {
  g_launches.fetch_add(1, std::memory_order_relaxed);
  Timer& t = timer();
  std::lock_guard<std::mutex> g(t.mu);
  if (!t.on) return;
  t.open_name = name;
  t.open_a = take_event(t);
  if (t.open_a) cudaEventRecord(t.open_a, s);
}

void timer_launch_end(cudaStream_t s) {
  Timer& t = timer();
  std::lock_guard<std::mutex> g(t.mu);
  if (!t.on || !t.open_a) return;
  cudaEvent_t b = take_event(t);
  if (!b) return;
  cudaEventRecord(b, s);
  t.pending.push_back(Pending{t.open_name, t.open_a, b});
  t.open_a = nullptr;
}

void timer_resolve() {
  Timer& t = timer();
  std::lock_guard<std::mutex> g(t.mu);
  for (const Pending& p : t.pending) {
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) {
      auto& e = t.totals[p.name];
      e.first += 1;
      e.second += ms;
    }
    t.pool.push_back(p.a);
    t.pool.push_back(p.b);
  }
  t.pending.clear();
}

}  // namespace ptc

extern "C" void ptc_timer_enable(int on) {
  ptc::Timer& t = ptc::timer();
  std::lock_guard<std::mutex> g(t.mu);
  t.on = on != 0;
}

extern "C" void ptc_timer_reset(void) {
  ptc::Timer& t = ptc::timer();
  std::lock_guard<std::mutex> g(t.mu);
  t.totals.clear();
}

extern "C" uint32_t ptc_timer_read(ptc_kernel_time* out, uint32_t cap) {
  ptc::Timer& t = ptc::timer();
  std::lock_guard<std::mutex> g(t.mu);
  uint32_t i = 0;
  for (const auto& kv : t.totals) {
    if (out && i < cap) {
      std::memset(out[i].name, 0, sizeof(out[i].name));
      std::strncpy(out[i].name, kv.first.c_str(), sizeof(out[i].name) - 1);
      out[i].launches = kv.second.first;
      out[i].total_ms = kv.second.second;
    }
    ++i;
  }
  return i;
}

extern "C" uint64_t ptc_launch_count(void) { return ptc::g_launches.load(); }

extern "C" const char* ptc_strerror(ptc_status s) {
  switch (s) {
    case PTC_OK: return "ok";
    case PTC_ERR_INVALID_ARG: return "invalid argument or malformed device input";
    case PTC_ERR_UNSORTED: return "request timestamps are not non-decreasing";
    case PTC_ERR_OVERFLOW: return "size or cost overflow (N or D >= 2^32-1, or a cost constant >= 2^64)";
    case PTC_ERR_WORKSPACE: return "workspace missing, misaligned or too small";
    case PTC_ERR_CUDA: return "CUDA runtime error";
    case PTC_ERR_TIMEOUT: return "a bounded device-side wait gave up";
    case PTC_ERR_HASH_COLLISION: return "two different prefixes share one block id";
    case PTC_ERR_NOT_IMPLEMENTED: return "not implemented";
  }
  return "unknown status";
}

extern "C" const char* ptc_version(void) { return "ptc 0.1.0 (sm_103a)"; }
