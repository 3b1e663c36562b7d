// C-ABI entry points that belong to no stage, the launch timer, the host
// staging buffers and the fill / copy kernels every stage uses.
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

namespace {
thread_local bool t_no_host_alloc = false;
}
NoHostAlloc::NoHostAlloc() : prev(t_no_host_alloc) { t_no_host_alloc = true; }
NoHostAlloc::~NoHostAlloc() { t_no_host_alloc = prev; }

namespace {
thread_local HostStage* t_pinned = nullptr;
thread_local HostStage t_fallback;
}  // namespace

// The calling thread's staging block: page-locked and mapped, allocated on
// the thread's first call (ptc_release_host_staging frees it), or ordinary
// thread-local memory when page-locked memory cannot be had.
HostStage* host_stage() {
  HostStage*& pinned = t_pinned;
  HostStage& fallback = t_fallback;
  if (!pinned) {
    fallback.dev = nullptr;
    if (t_no_host_alloc) return &fallback;
    void* p = nullptr;
    if (cudaHostAlloc(&p, sizeof(HostStage), cudaHostAllocPortable | cudaHostAllocMapped) == cudaSuccess) {
      pinned = static_cast<HostStage*>(p);
      void* d = nullptr;
      pinned->dev = cudaHostGetDevicePointer(&d, p, 0) == cudaSuccess ? static_cast<HostStage*>(d) : nullptr;
      (void)cudaGetLastError();
    } else {
      (void)cudaGetLastError();
      pinned = &fallback;
    }
  }
  return pinned;
}

namespace {
__global__ void k_fill(uint32_t* __restrict__ p, uint32_t v, uint64_t words) {
  grid_dep_sync();
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const uint64_t quads = (((uintptr_t)p & 15) == 0) ? words / 4 : 0;
  uint4* p4 = reinterpret_cast<uint4*>(p);
  for (uint64_t q = i; q < quads; q += stride) p4[q] = make_uint4(v, v, v, v);
  for (uint64_t w = quads * 4 + i; w < words; w += stride) p[w] = v;
}

struct FillMany {
  uint32_t* p[kFillRanges];
  uint64_t words[kFillRanges];
  uint32_t v[kFillRanges];
};

__global__ void k_fill_many(FillMany a) {
  grid_dep_sync();
  const uint32_t r = blockIdx.y;
  uint32_t* p = a.p[r];
  const uint32_t v = a.v[r];
  const uint64_t words = a.words[r];
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  const uint64_t i = (uint64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const uint64_t quads = (((uintptr_t)p & 15) == 0) ? words / 4 : 0;
  uint4* p4 = reinterpret_cast<uint4*>(p);
  for (uint64_t q = i; q < quads; q += stride) p4[q] = make_uint4(v, v, v, v);
  for (uint64_t w = quads * 4 + i; w < words; w += stride) p[w] = v;
}

__global__ void k_copy_words(const uint32_t* __restrict__ src, uint32_t* dst, uint32_t words) {
  grid_dep_sync();
  const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x, nth = gridDim.x * blockDim.x;
  const uint32_t quads = (((uintptr_t)src | (uintptr_t)dst) & 15) == 0 ? words / 4 : 0;
  for (uint32_t q = tid; q < quads; q += nth)
    reinterpret_cast<uint4*>(dst)[q] = reinterpret_cast<const uint4*>(src)[q];
  for (uint32_t i = quads * 4 + tid; i < words; i += nth) dst[i] = src[i];
}

// Earlier calls' error words (deferred, see defer_status) join this call's.
__global__ void k_carry_err(const uint32_t* err, uint32_t n, DevStatus* st) {
  grid_dep_sync();
  if (threadIdx.x < n && err[threadIdx.x]) atomicOr(&st->err, err[threadIdx.x]);
}

__global__ void k_copy_err(const DevStatus* st, uint32_t* slot, uint64_t* value_slot, uint32_t value_index,
                           uint32_t value_count) {
  grid_dep_sync();
  *slot = st->err;
  if (value_slot)
    for (uint32_t i = 0; i < value_count; ++i) value_slot[i] = st->value[value_index + i];
}
}  // namespace

ptc_status fill_async(void* p, uint32_t pattern, size_t bytes, cudaStream_t s) {
  if (bytes == 0) return PTC_OK;
  if ((bytes & 3) || ((uintptr_t)p & 3)) {
    if (cudaMemsetAsync(p, (int)(pattern & 0xFF), bytes, s) != cudaSuccess) return PTC_ERR_CUDA;
    return PTC_OK;
  }
  const uint64_t words = bytes / 4;
  const uint64_t want = (words / 4 + 255) / 256;
  const uint32_t cap = (uint32_t)(4 * num_sms());
  const uint32_t grid = want < cap ? (uint32_t)(want ? want : 1) : cap;
  PTC_KERNEL("k_fill", s, k_fill, grid, 256, 0, static_cast<uint32_t*>(p), pattern, words);
  return PTC_OK;
}

ptc_status fill_many_async(const FillRange* r, int n, cudaStream_t s) {
  FillMany a{};
  uint32_t m = 0;
  uint64_t most = 0;
  for (int i = 0; i < n; ++i) {
    if (r[i].bytes == 0) continue;
    if ((r[i].bytes & 3) || ((uintptr_t)r[i].p & 3) || m == (uint32_t)kFillRanges) {
      if (fill_async(r[i].p, r[i].pattern, r[i].bytes, s) != PTC_OK) return PTC_ERR_CUDA;
      continue;
    }
    a.p[m] = static_cast<uint32_t*>(r[i].p);
    a.words[m] = r[i].bytes / 4;
    a.v[m] = r[i].pattern;
    most = a.words[m] > most ? a.words[m] : most;
    ++m;
  }
  if (m == 0) return PTC_OK;
  const uint64_t want = (most / 4 + 255) / 256;
  const uint32_t cap = (uint32_t)(4 * num_sms());
  const uint32_t gx = want < cap ? (uint32_t)(want ? want : 1) : cap;
  PTC_KERNEL("k_fill_many", s, k_fill_many, dim3(gx, m), 256, 0, a);
  return PTC_OK;
}

ptc_status copy_to_host_async(void* host_dst, const void* dev_src, size_t bytes, cudaStream_t s) {
  HostStage* hs = host_stage();
  const char* lo = reinterpret_cast<const char*>(hs);
  const char* d = static_cast<const char*>(host_dst);
  const bool staged = hs->dev != nullptr && d >= lo && d + bytes <= lo + sizeof(HostStage);
  if (staged && (bytes & 3) == 0 && ((uintptr_t)dev_src & 3) == 0 && ((uintptr_t)d & 3) == 0) {
    uint32_t* dst = reinterpret_cast<uint32_t*>(reinterpret_cast<char*>(hs->dev) + (d - lo));
    const uint32_t words = (uint32_t)(bytes / 4);
    const uint32_t grid = words <= 1024 ? 1u : (words / 1024 < 16 ? words / 1024 : 16u);
    PTC_KERNEL("k_copy_words", s, k_copy_words, grid, 256, 0, static_cast<const uint32_t*>(dev_src), dst, words);
    return PTC_OK;
  }
  if (cudaMemcpyAsync(host_dst, dev_src, bytes, cudaMemcpyDeviceToHost, s) != cudaSuccess) return PTC_ERR_CUDA;
  return PTC_OK;
}

namespace {
constexpr int kRkThreads = 256;
constexpr int kRkPer = kRankTile / kRkThreads;  // consecutive words per thread
static_assert(kRkPer * kRkThreads == (int)kRankTile, "rank tile");

__device__ __forceinline__ bool rank_last_cta(uint32_t* done) {
  __shared__ uint32_t s_last;
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(done, 1u) == gridDim.x - 1;
  __syncthreads();
  if (s_last) __threadfence();
  return s_last;
}

__global__ void __launch_bounds__(kRkThreads) k_rank_count(const uint32_t* __restrict__ bits, uint32_t nwords,
                                                          uint32_t ntiles, uint32_t* tcnt, uint32_t* tpre,
                                                          uint32_t* done, uint64_t* total) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kRkThreads / 32];
  const uint32_t w0 = blockIdx.x * kRankTile + threadIdx.x;
  uint32_t c = 0;
#pragma unroll
  for (int k = 0; k < kRkPer; ++k)
    if (w0 + k * kRkThreads < nwords) c += __popc(bits[w0 + k * kRkThreads]);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(kFull, c, o);
  if ((threadIdx.x & 31) == 0) s_w[threadIdx.x >> 5] = c;
  __syncthreads();
  if (threadIdx.x == 0) {
    uint32_t t = 0;
    for (int i = 0; i < kRkThreads / 32; ++i) t += s_w[i];
    tcnt[blockIdx.x] = t;
  }
  if (!rank_last_cta(done)) return;
  const uint32_t all = cta_tiles_prefix(tcnt, tpre, ntiles);
  if (total && threadIdx.x == 0) *total = all;
}

__global__ void __launch_bounds__(kRkThreads) k_rank_words(const uint32_t* __restrict__ bits, uint32_t nwords,
                                                          const uint32_t* __restrict__ tpre, uint32_t* __restrict__ pre) {
  grid_dep_sync();
  __shared__ uint32_t s_w[kRkThreads / 32];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint32_t w0 = blockIdx.x * kRankTile + threadIdx.x * kRkPer;
  uint32_t c[kRkPer], sum = 0;
#pragma unroll
  for (int k = 0; k < kRkPer; ++k) {
    c[k] = w0 + k < nwords ? __popc(bits[w0 + k]) : 0u;
    sum += c[k];
  }
  uint32_t incl = sum;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(kFull, incl, o);
    if (lane >= (uint32_t)o) incl += y;
  }
  if (lane == 31) s_w[w] = incl;
  __syncthreads();
  uint32_t run = tpre[blockIdx.x] + incl - sum;
  for (int i = 0; i < (int)w; ++i) run += s_w[i];
#pragma unroll
  for (int k = 0; k < kRkPer; ++k) {
    if (w0 + k < nwords) pre[w0 + k] = run;
    run += c[k];
  }
}
}  // namespace

ptc_status bitmap_ranks(const uint32_t* bits, uint32_t nwords, uint32_t* pre, uint32_t* tcnt, uint32_t* tpre,
                        uint32_t* done, uint64_t* total, cudaStream_t s) {
  if (nwords == 0) return PTC_OK;
  const uint32_t T = rank_tiles(nwords);
  PTC_KERNEL("k_rank_count", s, k_rank_count, T, kRkThreads, 0, bits, nwords, T, tcnt, tpre, done, total);
  PTC_KERNEL("k_rank_words", s, k_rank_words, T, kRkThreads, 0, bits, nwords, tpre, pre);
  return PTC_OK;
}

ptc_status carry_errors(const uint32_t* err, uint32_t n, DevStatus* st, cudaStream_t s) {
  if (n == 0) return PTC_OK;
  if (n > 32) return PTC_ERR_INVALID_ARG;
  PTC_KERNEL("k_carry_err", s, k_carry_err, 1, 32, 0, err, n, st);
  return PTC_OK;
}

ptc_status defer_status(const DevStatus* dev, uint32_t* slot, cudaStream_t stream, uint64_t* value_slot,
                        uint32_t value_index, uint32_t value_count) {
  if (cudaGetLastError() != cudaSuccess) return PTC_ERR_CUDA;
  if (value_index + value_count > 8) return PTC_ERR_INVALID_ARG;
  PTC_KERNEL("k_copy_err", stream, k_copy_err, 1, 1, 0, dev, slot, value_slot, value_index, value_count);
  return PTC_OK;
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
    case PTC_ERR_BOUNDS: return "checked build: an index read from data fell outside its array";
  }
  return "unknown status";
}

#ifdef PTC_CHECKED
extern "C" const char* ptc_version(void) { return "ptc 0.1.0 (sm_103a, checked)"; }
#else
extern "C" const char* ptc_version(void) { return "ptc 0.1.0 (sm_103a)"; }
#endif

namespace {
std::atomic<uint32_t> g_wait_polls{0};
}  // namespace

uint32_t ptc::test_wait_polls() { return g_wait_polls.load(std::memory_order_relaxed); }

void ptc::release_host_stage() {
  if (t_pinned && t_pinned != &t_fallback) {
    (void)cudaFreeHost(t_pinned);
    (void)cudaGetLastError();
  }
  t_pinned = nullptr;
}

extern "C" void ptc_release_host_staging(void) { ptc::release_host_stage(); }

extern "C" void ptc_test_wait_polls(uint32_t polls) { g_wait_polls.store(polls, std::memory_order_relaxed); }
