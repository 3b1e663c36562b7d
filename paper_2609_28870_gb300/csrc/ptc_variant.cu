// ptc_stack_distance_variant — stack distances under the semantics variants
// (Sec. 3.1: the paper's simulator keeps a whole request resident and makes
// room for it before the prefill; engines differ in the order they touch a
// request's blocks).
//
// Touch order.  Leaf-first touches the blocks of request r (accesses
// off[r] .. off[r+1]-1, root-first) in reverse, so access i sits at position
//   pi(i) = off[r] + off[r+1] - 1 - i
// of the touch stream.  Every block appears at most once per request, so the
// previous touch of the block at pi(i) is pi(prev[i]): prev in touch order is
// the permuted prev, and no new sort is needed.
//
// Residency.  Per block, a block is looked up when touched: the window of the
// stack distance ends at the access itself, and the distance is the one
// ptc_stack_distance computes on the touch stream.  Per request, every block
// is looked up at the request's arrival: the window ends at the request's
// first position e = off[r], and the distance is 1 + the distinct blocks
// touched in (p, e) — the block's depth in the LRU stack at arrival.  The
// per-block window (p, i) splits at e, and a block touched in [e, i) is new to
// the window iff its own previous touch lies before p, so
//   dist_request(i) = dist_block(i) - #{ j in [e, i) : prev[j] < p or none }.
// The count runs over the request's own accesses only.  They fall into runs
// (prev growing by one, or first accesses), cut at request starts; inside a
// run prev[j] = q + (j - start), so a run contributes min(max(p - q, 0), len)
// (all of it if cold), and the access's own run contributes its offset.  A
// trace with few runs (at most a third of the accesses) takes this route;
// otherwise the matrix over every access answers the windows ending at e
// directly (ptc_wavelet.cu).
//
//   k_var_tiles   one thread per request: offset checks, and the request
//                 holding each tile's first access
//   k_var_reqof   the request of every access (root-first, per request: the
//                 window end off[r] directly)
//   k_var_perm    leaf-first: prev and the window ends in touch order
//   k_var_heads   per request: run heads of the touch stream (a bitmap)
//   k_var_rec     per request: each run's start and first prev value
//   k_var_fix     per request: the count above, off the per-block distance
//   k_var_unperm  leaf-first: the distances back in depth order
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kVT = 256;
constexpr int kVPer = 8;
constexpr uint32_t kVTile = kVT * kVPer;

__global__ void __launch_bounds__(kVT) k_var_tiles(const uint64_t* __restrict__ off, uint32_t n_req, uint64_t n,
                                                   uint32_t tiles, uint32_t* __restrict__ tile_req, DevStatus* st) {
  grid_dep_sync();
  const uint32_t r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= n_req) return;
  const uint64_t lo = off[r], hi = off[r + 1];
  if (hi < lo || hi > n || (r == 0 && lo != 0) || (r + 1 == n_req && hi != n)) {
    raise_err(st, kErrInvalid);
    return;
  }
  for (uint64_t t = (lo + kVTile - 1) / kVTile; t * kVTile < hi; ++t) tile_req[t] = r;
  if (r + 1 == n_req) tile_req[tiles] = r;
}

struct VarArgs {
  const uint64_t* off;
  const uint32_t* prev;
  uint32_t n;
  uint32_t n_req;
  const uint32_t* tile_req;
  uint32_t* req_of;  // leaf-first only
  uint32_t* prevp;   // prev in touch order (leaf-first)
  uint32_t* wend;    // window end of every access in touch order (per request)
  const uint32_t* distp;
  uint32_t* dist;
  int leaf;
  int request;
  DevStatus* st;
};

__global__ void __launch_bounds__(kVT) k_var_reqof(const __grid_constant__ VarArgs a) {
  grid_dep_sync();
  const uint32_t t = blockIdx.x;
  uint32_t r0 = __ldg(a.tile_req + t), r1 = __ldg(a.tile_req + t + 1);
  r0 = r0 < a.n_req ? r0 : a.n_req - 1;
  r1 = r1 < a.n_req ? (r1 > r0 ? r1 : r0) : a.n_req - 1;
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = (uint64_t)t * kVTile + k * kVT + threadIdx.x;
    if (i < a.n) {
      const uint32_t r = req_search(a.off, r0, r1, i);
      if (a.leaf) a.req_of[i] = r;
      else a.wend[i] = (uint32_t)__ldg(a.off + r);
    }
  }
}

// Loads are issued for four positions at a time before any is used.
__global__ void __launch_bounds__(kVT) k_var_perm(const __grid_constant__ VarArgs a) {
  grid_dep_sync();
  constexpr int kH = 4;
  bool bad = false;
#pragma unroll 1
  for (int half = 0; half < kVPer / kH; ++half) {
    const uint64_t base = (uint64_t)blockIdx.x * kVTile + half * kH * kVT + threadIdx.x;
    // offsets are below n < 2^32, so 32 bits hold them
    uint32_t r[kH], p[kH], rp[kH], lo[kH], hi[kH], plo[kH], phi[kH];
#pragma unroll
    for (int k = 0; k < kH; ++k) {
      const uint64_t i = base + k * kVT;
      r[k] = i < a.n ? a.req_of[i] : 0u;
      p[k] = i < a.n ? __ldg(a.prev + i) : kNone;
    }
#pragma unroll
    for (int k = 0; k < kH; ++k) {
      const uint64_t i = base + k * kVT;
      lo[k] = (uint32_t)__ldg(a.off + r[k]);
      hi[k] = (uint32_t)__ldg(a.off + r[k] + 1);
      rp[k] = (p[k] != kNone && p[k] < i) ? a.req_of[p[k]] : 0u;
    }
#pragma unroll
    for (int k = 0; k < kH; ++k) {
      plo[k] = (uint32_t)__ldg(a.off + rp[k]);
      phi[k] = (uint32_t)__ldg(a.off + rp[k] + 1);
    }
#pragma unroll
    for (int k = 0; k < kH; ++k) {
      const uint64_t i = base + k * kVT;
      if (i >= a.n) continue;
      // pi(i), and pi(prev); malformed offsets or prev that put them outside
      // the trace are reported (k_var_tiles has checked the offsets too)
      if (!(lo[k] <= i && i < hi[k] && hi[k] <= a.n)) {
        bad = true;
        continue;
      }
      const uint32_t ip = (uint32_t)((uint64_t)lo[k] + hi[k] - 1 - i);
      uint32_t pp = kNone;
      if (p[k] != kNone) {
        if (p[k] < i && plo[k] <= p[k] && p[k] < phi[k] && phi[k] <= a.n)
          pp = (uint32_t)((uint64_t)plo[k] + phi[k] - 1 - p[k]);
        else
          bad = true;
      }
      a.prevp[ip] = pp;
      if (a.request) a.wend[ip] = lo[k];
    }
  }
  if (bad) raise_err(a.st, kErrInvalid);
}

struct RunArgs {
  const uint32_t* prev;  // in touch order
  const uint32_t* wend;  // request start of every touch position
  uint32_t n;
  uint32_t* bits;        // run heads, one bit per position
  const uint32_t* pre;   // heads before each word
  const unsigned long long* total;
  uint32_t* rec_start;   // R + 1 entries (rec_start[R] = n)
  uint32_t* rec_q;       // first prev value of each run (kNone: a run of first accesses)
  uint32_t* dist;        // per-block distances in touch order, corrected in place
};

// A position starts a run if it starts its request, or its prev is not the
// previous position's prev plus one (first accesses run together).  A warp
// covers 32 consecutive positions, one bitmap word.
__global__ void __launch_bounds__(kVT) k_var_heads(const __grid_constant__ RunArgs a) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint64_t base = (uint64_t)blockIdx.x * kVTile + threadIdx.x;
  uint32_t p[kVPer], w[kVPer], before[kVPer];
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = base + k * kVT;
    p[k] = i < a.n ? __ldg(a.prev + i) : kNone;
    w[k] = i < a.n ? __ldg(a.wend + i) : 0u;
    before[k] = (lane == 0 && i > 0 && i <= a.n) ? __ldg(a.prev + i - 1) : kNone;
  }
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = base + k * kVT;
    uint32_t pb = __shfl_up_sync(kFull, p[k], 1);
    if (lane == 0) pb = before[k];
    const bool head = i < a.n && (i == 0 || w[k] == i || (p[k] == kNone) != (pb == kNone) ||
                                  (p[k] != kNone && p[k] != pb + 1u));
    const uint32_t word = __ballot_sync(kFull, head);
    if (lane == 0 && i < a.n) a.bits[i >> 5] = word;
  }
}

__device__ __forceinline__ uint32_t heads_through(const RunArgs& a, uint32_t i) {  // heads at positions <= i
  const uint32_t w = i >> 5, m = (i & 31) == 31 ? kFull : ((2u << (i & 31)) - 1u);
  return __ldg(a.pre + w) + __popc(__ldg(a.bits + w) & m);
}

__global__ void __launch_bounds__(kVT) k_var_rec(const __grid_constant__ RunArgs a) {
  grid_dep_sync();
  const uint64_t base = (uint64_t)blockIdx.x * kVTile + threadIdx.x;
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = base + k * kVT;
    if (i < a.n && ((__ldg(a.bits + (i >> 5)) >> (i & 31)) & 1u)) {
      const uint32_t t = heads_through(a, (uint32_t)i) - 1;
      a.rec_start[t] = (uint32_t)i;
      a.rec_q[t] = __ldg(a.prev + i);
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) a.rec_start[*a.total] = a.n;
}

__global__ void __launch_bounds__(kVT) k_var_fix(const __grid_constant__ RunArgs a) {
  grid_dep_sync();
  constexpr int kH = 4;  // positions whose loads are in flight together
#pragma unroll 1
  for (int half = 0; half < kVPer / kH; ++half) {
    const uint64_t base = (uint64_t)blockIdx.x * kVTile + half * kH * kVT + threadIdx.x;
    uint32_t p[kH], e[kH], t[kH], st[kH];
#pragma unroll
    for (int k = 0; k < kH; ++k) {
      const uint64_t i = base + k * kVT;
      p[k] = i < a.n ? __ldg(a.prev + i) : kNone;
      e[k] = i < a.n ? __ldg(a.wend + i) : 0u;
      t[k] = p[k] != kNone ? heads_through(a, (uint32_t)i) - 1 : 0u;
    }
#pragma unroll
    for (int k = 0; k < kH; ++k) st[k] = p[k] != kNone ? a.rec_start[t[k]] : 0u;
#pragma unroll
    for (int k = 0; k < kH; ++k) {
      const uint64_t i = base + k * kVT;
      if (p[k] == kNone) continue;
      uint32_t cnt = (uint32_t)i - st[k];  // earlier positions of its own run
      uint32_t end = st[k];
      for (uint32_t u = t[k]; u-- > 0;) {  // earlier runs of its request
        const uint32_t s0 = a.rec_start[u];
        if (s0 < e[k]) break;
        const uint32_t len = end - s0, q = a.rec_q[u];
        cnt += q == kNone ? len : (p[k] > q ? (p[k] - q < len ? p[k] - q : len) : 0u);
        end = s0;
      }
      a.dist[i] -= cnt;
    }
  }
}

__global__ void __launch_bounds__(kVT) k_var_unperm(const __grid_constant__ VarArgs a) {
  grid_dep_sync();
  const uint64_t base = (uint64_t)blockIdx.x * kVTile + threadIdx.x;
  uint32_t r[kVPer], ip[kVPer], d[kVPer];
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = base + k * kVT;
    r[k] = i < a.n ? a.req_of[i] : 0u;
  }
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = base + k * kVT;
    const uint64_t lo = __ldg(a.off + r[k]), hi = __ldg(a.off + r[k] + 1);
    ip[k] = (i < a.n && lo <= i && i < hi && hi <= a.n) ? (uint32_t)(lo + hi - 1 - i) : kNone;
  }
#pragma unroll
  for (int k = 0; k < kVPer; ++k) d[k] = ip[k] != kNone ? a.distp[ip[k]] : kNone;
#pragma unroll
  for (int k = 0; k < kVPer; ++k) {
    const uint64_t i = base + k * kVT;
    if (i < a.n) a.dist[i] = d[k];
  }
}

struct VarLayout {
  DevStatus* st;
  uint32_t* done;             // bitmap_ranks' counter
  unsigned long long* heads;  // number of runs
  size_t zero_bytes;
  uint32_t* tile_req;
  uint32_t* req_of;
  uint32_t* prevp;
  uint32_t* wend;
  uint32_t* distp;
  uint32_t *bits, *pre, *tcnt, *tpre, *rec_start, *rec_q;
  uint32_t nwords;
  void* sd;  // workspace of the stack-distance stage
  size_t sd_bytes;
  size_t total;
};

VarLayout var_layout(void* ws, uint64_t n, int leaf, int request) {
  VarLayout L;
  Carver cv(ws);
  L.st = cv.take<DevStatus>(1);
  L.done = cv.take<uint32_t>(1);
  L.heads = cv.take<unsigned long long>(1);
  L.zero_bytes = cv.off;
  L.tile_req = cv.take<uint32_t>((n + kVTile - 1) / kVTile + 1);
  L.req_of = leaf ? cv.take<uint32_t>(n) : nullptr;
  L.prevp = leaf ? cv.take<uint32_t>(n) : nullptr;
  L.distp = leaf ? cv.take<uint32_t>(n) : nullptr;
  L.wend = request ? cv.take<uint32_t>(n) : nullptr;
  L.nwords = (uint32_t)((n + 31) / 32);
  const uint32_t rt = rank_tiles(L.nwords) + 1;
  L.bits = request ? cv.take<uint32_t>(L.nwords + 1) : nullptr;
  L.pre = request ? cv.take<uint32_t>(L.nwords + 1) : nullptr;
  L.tcnt = request ? cv.take<uint32_t>(rt) : nullptr;
  L.tpre = request ? cv.take<uint32_t>(rt) : nullptr;
  L.rec_start = request ? cv.take<uint32_t>(n + 1) : nullptr;
  L.rec_q = request ? cv.take<uint32_t>(n) : nullptr;
  const size_t a = ptc_stack_distance_workspace_bytes(n), b = stack_distance_points_bytes(n);
  L.sd_bytes = a > b ? a : b;
  L.sd = cv.take<char>(L.sd_bytes);
  L.total = cv.bytes();
  return L;
}

bool variant_ok(int order, int residency) {
  return (order == PTC_TOUCH_ROOT_FIRST || order == PTC_TOUCH_LEAF_FIRST) &&
         (residency == PTC_RESIDENCY_BLOCK || residency == PTC_RESIDENCY_REQUEST);
}

}  // namespace
}  // namespace ptc

using namespace ptc;

extern "C" size_t ptc_stack_distance_variant_workspace_bytes(uint64_t n, uint32_t n_req, int touch_order,
                                                             int residency) {
  (void)n_req;
  if (touch_order == PTC_TOUCH_ROOT_FIRST && residency == PTC_RESIDENCY_BLOCK)
    return ptc_stack_distance_workspace_bytes(n);
  return var_layout(nullptr, n, touch_order == PTC_TOUCH_LEAF_FIRST, residency == PTC_RESIDENCY_REQUEST).total;
}

extern "C" ptc_status ptc_stack_distance_variant_ex(const uint32_t* prev, uint64_t n, const uint64_t* req_blk_off,
                                                    uint32_t n_req, int touch_order, int residency, uint32_t* dist_out,
                                                    int method, void* ws, size_t ws_bytes, void* stream) {
  if (n >= (uint64_t)kNone) return PTC_ERR_OVERFLOW;
  if (!variant_ok(touch_order, residency)) return PTC_ERR_INVALID_ARG;
  if (method != PTC_SD_AUTO && method != PTC_SD_POINTS && method != PTC_SD_RUNS) return PTC_ERR_INVALID_ARG;
  if (n == 0) return PTC_OK;
  if (!prev || !dist_out || !req_blk_off || n_req == 0) return PTC_ERR_INVALID_ARG;
  if (touch_order == PTC_TOUCH_ROOT_FIRST && residency == PTC_RESIDENCY_BLOCK)
    return ptc_stack_distance(prev, n, dist_out, ws, ws_bytes, stream);
  const int leaf = touch_order == PTC_TOUCH_LEAF_FIRST, request = residency == PTC_RESIDENCY_REQUEST;
  if (!ws_ok(ws, ws_bytes, var_layout(nullptr, n, leaf, request).total)) return PTC_ERR_WORKSPACE;
  cudaStream_t s = (cudaStream_t)stream;
  const VarLayout L = var_layout(ws, n, leaf, request);
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t tiles = ceil_div_u32(n, kVTile);
  PTC_KERNEL("k_var_tiles", s, k_var_tiles, ceil_div_u32(n_req, kVT), kVT, 0, req_blk_off, n_req, n, tiles,
             L.tile_req, L.st);
  VarArgs a{req_blk_off, prev, (uint32_t)n, n_req, L.tile_req, L.req_of, L.prevp, L.wend, L.distp, dist_out,
            leaf, request, L.st};
  PTC_KERNEL("k_var_reqof", s, k_var_reqof, tiles, kVT, 0, a);
  if (leaf) PTC_KERNEL("k_var_perm", s, k_var_perm, tiles, kVT, 0, a);
  const uint32_t* tprev = leaf ? L.prevp : prev;  // the touch stream
  uint32_t* tdist = leaf ? L.distp : dist_out;
  ptc_status rc_sd = PTC_OK;
  bool few_runs = true;
  if (request) {
    // runs of the touch stream, cut at request starts
    const RunArgs ra{tprev, L.wend, (uint32_t)n, L.bits, L.pre, L.heads, L.rec_start, L.rec_q, tdist};
    PTC_KERNEL("k_var_heads", s, k_var_heads, tiles, kVT, 0, ra);
    if (bitmap_ranks(L.bits, L.nwords, L.pre, L.tcnt, L.tpre, L.done, reinterpret_cast<uint64_t*>(L.heads), s) !=
        PTC_OK)
      return PTC_ERR_CUDA;
    uint64_t* hv = &host_stage()->out[0];
    if (copy_to_host_async(hv, L.heads, sizeof(uint64_t), s) != PTC_OK) return PTC_ERR_CUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return PTC_ERR_CUDA;
    few_runs = method == PTC_SD_RUNS || (method == PTC_SD_AUTO && *hv <= n / 3);
    if (few_runs) {
      PTC_KERNEL("k_var_rec", s, k_var_rec, tiles, kVT, 0, ra);
      rc_sd = ptc_stack_distance(tprev, n, tdist, L.sd, L.sd_bytes, s);
      PTC_KERNEL("k_var_fix", s, k_var_fix, tiles, kVT, 0, ra);
    } else {
      rc_sd = stack_distance_points(tprev, n, tdist, L.sd, L.sd_bytes, s, L.wend);
    }
  } else {
    rc_sd = ptc_stack_distance(tprev, n, tdist, L.sd, L.sd_bytes, s);
  }
  if (leaf) PTC_KERNEL("k_var_unperm", s, k_var_unperm, tiles, kVT, 0, a);
  DevStatus h;
  const ptc_status rc = end_call(L.st, s, &h);
  return rc != PTC_OK ? rc : rc_sd;
}

extern "C" ptc_status ptc_stack_distance_variant(const uint32_t* prev, uint64_t n, const uint64_t* req_blk_off,
                                                 uint32_t n_req, int touch_order, int residency, uint32_t* dist_out,
                                                 void* ws, size_t ws_bytes, void* stream) {
  return ptc_stack_distance_variant_ex(prev, n, req_blk_off, n_req, touch_order, residency, dist_out, PTC_SD_AUTO, ws,
                                       ws_bytes, stream);
}
