// Measurement hook: the rate at which this GPU settles random read-modify-
// write probes of 16-byte slots in a DRAM-sized table.  That is the ceiling of
// the id table's insert (stage a2), whose every probe of a key not matched by
// the prior-request hint reads a random slot and claims it with a 128-bit CAS;
// the plain HBM copy bandwidth does not bound it.  Instrumentation for the
// roofline figures only; no stage of the path calls it.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kProbeThreads = 256;

__device__ __forceinline__ uint64_t probe_slot(uint64_t seed, uint64_t i, uint64_t mask) {
  return splitmix64_at(seed, i) & mask;
}

// Thread g settles probes g, g + stride, ... < n: a relaxed 16-byte load of a
// random slot, then, if the slot is empty (all ones), a 128-bit CAS that
// claims it.  All slots must start empty.
__global__ void __launch_bounds__(kProbeThreads) k_probe_rmw(ulonglong2* table, uint64_t mask, uint64_t n,
                                                              uint64_t seed, unsigned long long* sink) {
  grid_dep_sync();
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  uint64_t acc = 0;
  for (uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    ulonglong2* p = table + probe_slot(seed, i, mask);
    ulonglong2 v;
    asm volatile("ld.relaxed.gpu.global.v2.u64 {%0, %1}, [%2];" : "=l"(v.x), "=l"(v.y) : "l"(p) : "memory");
    if (v.x == ~0ULL && v.y == ~0ULL) {
      ulonglong2 old;
      asm volatile(
          "{\n\t.reg .b128 c, w, d;\n\t"
          "mov.b128 c, {%2, %3};\n\t"
          "mov.b128 w, {%4, %5};\n\t"
          "atom.global.cas.b128 d, [%6], c, w;\n\t"
          "mov.b128 {%0, %1}, d;\n\t}"
          : "=l"(old.x), "=l"(old.y)
          : "l"(~0ULL), "l"(~0ULL), "l"(i), "l"(seed), "l"(p)
          : "memory");
      acc ^= old.x;
    }
  }
  if (acc == 0x9E3779B97F4A7C15ULL) atomicAdd(sink, 1ULL);  // keeps the loads; practically never true
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" ptc_status ptc_probe_random_rmw(void* table, uint64_t slots, uint64_t probes, uint64_t seed, void* sink,
                                           void* stream) {
  if (table == nullptr || sink == nullptr || slots == 0 || (slots & (slots - 1)) != 0 ||
      (reinterpret_cast<uintptr_t>(table) & 15) != 0 || (reinterpret_cast<uintptr_t>(sink) & 7) != 0)
    return PTC_ERR_INVALID_ARG;
  if (probes == 0) return PTC_OK;
  const uint64_t want = (probes + kProbeThreads - 1) / kProbeThreads;
  const uint32_t cap = (uint32_t)(8 * num_sms());
  const uint32_t grid = want < cap ? (uint32_t)want : cap;
  cudaStream_t s = (cudaStream_t)stream;
  PTC_KERNEL("k_probe_rmw", s, k_probe_rmw, grid, kProbeThreads, 0, reinterpret_cast<ulonglong2*>(table), slots - 1,
             probes, seed, reinterpret_cast<unsigned long long*>(sink));
  return cudaPeekAtLastError() == cudaSuccess ? PTC_OK : PTC_ERR_CUDA;
}
