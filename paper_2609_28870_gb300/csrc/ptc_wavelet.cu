// Stage c: LRU stack distance of every access (paper App. B, stack distance
// between reuses), as a 2-D dominance count on a wavelet matrix.
//
// For access i with previous use p = prev[i]:
//   SD_i - 1 = #distinct blocks in (p, i) = #{ j in (p, i) : prev[j] < p or prev[j] = none }
// because every block touched in (p, i) has exactly one access in that window
// whose previous use lies before p (its first access inside the window), and
// p's own block is not touched in (p, i).  With v_j = prev[j] + 1 (none -> 0)
// this is "count v_j < p + 1 for j in [p+1, i)": a range-rank query.
//
// Wavelet matrix (Claude, Navarro, Ordonez 2015) over v[0..N): L levels for
// values < 2^L.  Level l keeps one bit per position — bit (L-1-l) of the value
// at that position in level l's order — and level l+1's order is the stable
// partition of level l's order by that bit (zeros first, Z_l of them).
//
// Layout of one level: blocks of 224 positions in 32 bytes,
//   word 0 = zeros before the block, words 1..7 = 224 bits (LSB first)
// so a rank is one 32-byte sector.
//   k_wm_zeros   Z_l for every level in one pass over prev
//   k_wm_level   one level: ballot bits -> rank blocks; stable partition by
//                bit with tile zero counts through decoupled look-back
//   k_wm_query   per access, L rank steps (early exit on an empty range)
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kLvThreads = 1024;
constexpr int kLvWarps = kLvThreads / 32;
constexpr int kBlkBits = 224;                     // positions per rank block
constexpr int kLvTile = kLvWarps * kBlkBits;      // 7168 positions per tile
constexpr int kQThreads = 256;

__device__ __forceinline__ uint32_t value_at(const uint32_t* __restrict__ prev, uint64_t j) {
  const uint32_t p = prev[j];
  return p == kNone ? 0u : p + 1u;
}

__global__ void __launch_bounds__(256) k_wm_zeros(const uint32_t* __restrict__ prev, uint64_t n, uint32_t L,
                                                  unsigned long long* __restrict__ ones, DevStatus* st) {
  __shared__ unsigned long long s_ones[33];
  if (threadIdx.x < 33) s_ones[threadIdx.x] = 0;
  __syncthreads();
  const uint32_t lane = threadIdx.x & 31;
  uint64_t acc = 0;  // lane l accumulates the ones of level l
  bool bad = false;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t base = (uint64_t)blockIdx.x * blockDim.x; base < n; base += stride) {
    const uint64_t j = base + threadIdx.x;
    uint32_t v = 0;
    if (j < n) {
      const uint32_t p = prev[j];
      if (p != kNone && p >= j) bad = true;
      v = p == kNone ? 0u : p + 1u;
    }
    for (uint32_t l = 0; l < L; ++l) {
      const uint32_t m = __ballot_sync(kFull, (v >> (L - 1 - l)) & 1u);
      if (lane == (l & 31)) acc += __popc(m);
    }
  }
  if (bad) raise_err(st, kErrInvalid);
  // L <= 33: level 32 (if any) was accumulated by lane 0 together with level 0
  // only when L == 33, which needs n >= 2^32 and is rejected on the host.
  if (lane < L) atomicAdd(&s_ones[lane], (unsigned long long)acc);
  __syncthreads();
  if (threadIdx.x < L && s_ones[threadIdx.x]) atomicAdd(&ones[threadIdx.x], s_ones[threadIdx.x]);
}

struct LevelArgs {
  const uint32_t* prev;   // level 0 input (values derived on the fly)
  const uint32_t* vin;    // levels >= 1
  uint32_t* vout;         // null on the last level
  uint32_t* mat;          // this level's rank blocks
  uint64_t n;
  uint32_t shift;         // bit tested at this level
  const unsigned long long* ones;  // ones per level; Z_l = n - ones[l]
  uint32_t level;
  uint64_t* lb;
  DevStatus* st;
};

__global__ void __launch_bounds__(kLvThreads) k_wm_level(LevelArgs a) {
  __shared__ uint32_t s_wz[kLvWarps];
  __shared__ uint64_t s_base;
  const uint32_t epoch = a.level + 1;
  const uint32_t tile = next_tile(a.st, (int)epoch);
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const uint64_t blk = (uint64_t)tile * kLvWarps + w;
  const uint64_t base = blk * kBlkBits;
  uint32_t v[7], word[7], vmask[7];
  uint32_t zeros = 0;
#pragma unroll
  for (int k = 0; k < 7; ++k) {
    const uint64_t j = base + (uint64_t)k * 32 + lane;
    const bool valid = j < a.n;
    v[k] = valid ? (a.level == 0 ? value_at(a.prev, j) : a.vin[j]) : 0u;
    word[k] = __ballot_sync(kFull, valid && ((v[k] >> a.shift) & 1u));
    vmask[k] = __ballot_sync(kFull, valid);
    zeros += __popc(vmask[k] & ~word[k]);
  }
  if (lane == 0) s_wz[w] = zeros;
  __syncthreads();
  if (w == 0) {
    const uint32_t z = s_wz[lane];
    uint32_t x = z;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(kFull, x, o);
      if (lane >= (uint32_t)o) x += y;
    }
    s_wz[lane] = x - z;  // exclusive over warps
    const uint64_t tile_zeros = __shfl_sync(kFull, x, 31);
    const uint64_t prefix = lookback_sum(a.lb, tile, tile_zeros, epoch, a.st);
    if (lane == 0) s_base = prefix;
  }
  __syncthreads();
  const uint64_t zb = s_base + s_wz[w];  // zeros before this rank block
  if (base <= a.n && lane < 8) {
    uint32_t out = (uint32_t)zb;
#pragma unroll
    for (int k = 0; k < 7; ++k)
      if (lane == (uint32_t)k + 1) out = word[k];
    a.mat[blk * 8 + lane] = out;
  }
  if (a.vout != nullptr) {
    const uint64_t Z = a.n - a.ones[a.level];
    uint64_t zrun = zb;
    const uint32_t lt = lanemask_lt();
#pragma unroll
    for (int k = 0; k < 7; ++k) {
      const uint64_t j = base + (uint64_t)k * 32 + lane;
      const uint32_t zmask = vmask[k] & ~word[k];
      if (j < a.n) {
        const uint64_t zb_elem = zrun + __popc(zmask & lt);
        const bool one = (word[k] >> lane) & 1u;
        const uint64_t dst = one ? Z + (j - zb_elem) : zb_elem;
        if (dst < a.n) a.vout[dst] = v[k];  // always true unless a bounded wait gave up
      }
      zrun += __popc(zmask);
    }
  }
}

__device__ __forceinline__ uint32_t rank0(const uint32_t* __restrict__ lvl, uint32_t pos) {
  const uint32_t b = pos / kBlkBits;
  const uint32_t off = pos - b * kBlkBits;
  const uint4* p = reinterpret_cast<const uint4*>(lvl + (uint64_t)b * 8);
  const uint4 lo = __ldg(p), hi = __ldg(p + 1);
  const uint32_t wi = off >> 5;
  const uint32_t m = (1u << (off & 31)) - 1u;
  const uint32_t w[7] = {lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
  uint32_t ones = 0;
#pragma unroll
  for (int k = 0; k < 7; ++k) {
    const uint32_t x = (uint32_t)k < wi ? w[k] : ((uint32_t)k == wi ? (w[k] & m) : 0u);
    ones += __popc(x);
  }
  return lo.x + off - ones;
}

__global__ void __launch_bounds__(kQThreads) k_wm_query(const uint32_t* __restrict__ prev, uint64_t n, uint32_t L,
                                                        const uint32_t* __restrict__ mat, uint64_t level_words,
                                                        const unsigned long long* __restrict__ ones,
                                                        uint32_t* __restrict__ dist, DevStatus* st) {
  __shared__ uint32_t s_z[33];
  if (threadIdx.x < L) s_z[threadIdx.x] = (uint32_t)(n - ones[threadIdx.x]);
  __syncthreads();
  const uint64_t i = (uint64_t)blockIdx.x * kQThreads + threadIdx.x;
  if (i >= n) return;
  const uint32_t p = prev[i];
  if (p == kNone) {
    dist[i] = kNone;
    return;
  }
  if ((uint64_t)p >= i) {
    raise_err(st, kErrInvalid);
    dist[i] = kNone;
    return;
  }
  const uint32_t x = p + 1;
  uint32_t s = p + 1, e = (uint32_t)i, cnt = 0;
  const uint32_t nmax = (uint32_t)n;
  for (uint32_t l = 0; l < L && s < e; ++l) {
    if (e > nmax) e = nmax;  // positions stay in [0, n] on a well-formed matrix
    if (s > e) s = e;
    const uint32_t* lvl = mat + (uint64_t)l * level_words;
    const uint32_t zs = rank0(lvl, s), ze = rank0(lvl, e);
    if ((x >> (L - 1 - l)) & 1u) {
      cnt += ze - zs;
      s = s_z[l] + (s - zs);
      e = s_z[l] + (e - ze);
    } else {
      s = zs;
      e = ze;
    }
  }
  dist[i] = 1 + cnt;
}

uint32_t value_bits(uint64_t n) {  // values lie in [0, n]
  uint32_t L = 1;
  while (L < 33 && (1ULL << L) <= n) ++L;
  return L;
}

struct WmLayout {
  DevStatus* st;
  unsigned long long* ones;
  uint64_t* lb;
  uint32_t* va;
  uint32_t* vb;
  uint32_t* mat;
  uint64_t level_words;
  uint32_t L;
  size_t zero_bytes;
  size_t total;
};

WmLayout wm_layout(void* ws, uint64_t n) {
  WmLayout L;
  Carver cv(ws);
  L.L = value_bits(n);
  const uint64_t nblk = n / kBlkBits + 2;
  L.level_words = nblk * 8;
  L.st = cv.take<DevStatus>(1);
  L.ones = cv.take<unsigned long long>(40);
  L.lb = cv.take<uint64_t>(ceil_div_u32(n + 1, kLvTile) + 1);
  L.zero_bytes = cv.off;
  L.va = cv.take<uint32_t>(n ? n : 1);
  L.vb = cv.take<uint32_t>(n ? n : 1);
  L.mat = cv.take<uint32_t>(L.level_words * L.L);
  L.total = cv.bytes();
  return L;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_stack_distance_workspace_bytes(uint64_t n) { return wm_layout(nullptr, n).total; }

extern "C" ptc_status ptc_stack_distance(const uint32_t* prev, uint64_t n, uint32_t* dist_out, void* ws,
                                         size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (n == 0) return PTC_OK;
  if (!prev || !dist_out) return PTC_ERR_INVALID_ARG;
  if (!ws_ok(ws, ws_bytes, wm_layout(nullptr, n).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const WmLayout W = wm_layout(ws, n);
  if (begin_call(ws, W.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  PTC_LAUNCH("k_wm_zeros", s, k_wm_zeros<<<1216, 256, 0, s>>>(prev, n, W.L, W.ones, W.st));
  const uint32_t tiles = ceil_div_u32(n + 1, kLvTile);
  const uint32_t* vin = nullptr;
  uint32_t* vout = W.va;
  for (uint32_t l = 0; l < W.L; ++l) {
    LevelArgs a;
    a.prev = prev;
    a.vin = vin;
    a.vout = (l + 1 < W.L) ? vout : nullptr;
    a.mat = W.mat + (uint64_t)l * W.level_words;
    a.n = n;
    a.shift = W.L - 1 - l;
    a.ones = W.ones;
    a.level = l;
    a.lb = W.lb;
    a.st = W.st;
    PTC_LAUNCH("k_wm_level", s, k_wm_level<<<tiles, kLvThreads, 0, s>>>(a));
    vin = vout;
    vout = (vout == W.va) ? W.vb : W.va;
  }
  PTC_LAUNCH("k_wm_query", s, k_wm_query<<<ceil_div_u32(n, kQThreads), kQThreads, 0, s>>>(prev, n, W.L, W.mat, W.level_words, W.ones, dist_out,
                                                               W.st));
  DevStatus h;
  return end_call(W.st, s, &h);
}
