// Stage a1: chained block keys (paper Sec. 2.2 block identity).
//
// Block k of a request covers tokens [Bk, Bk+B).  Its key is a polynomial of
// the whole prefix over GF(2^61 - 1) at two seeded bases u (one per key word):
//     S_k = sum_{t < B(k+1)} (tok_t + 1) u^(t+1)
// Every coefficient is at least 1, so two different prefixes, of equal or of
// different length, differ as polynomials (Karp-Rabin; a pair collides with
// probability at most length / 2^61 per base).  Written per block:
//     h_j = sum_{i<B} (tok_{Bj+i} + 1) u^(i+1)                 (block-local)
//     S_k = sum_{j<=k} h_j u^(Bj)
// so the chain across a request is a plain segmented sum of g_j = h_j u^(Bj):
// one scan, no sequential chain, and the sum itself is the key.
//
// Kernels
//   k_block_offsets  per-request block counts -> exclusive scan (look-back),
//                    validates offsets and timestamp order, max blocks/request
//   k_pow_tables     u^(B e) for e < 2^32 as two 65,536-entry levels
//                    (filled up to the longest request)
//   k_hash16         B = 16, aligned tokens: the tile's request offsets in
//                    shared memory, one block per thread
//   k_hash_tile      B any multiple of 16, aligned tokens: one block per
//                    thread, its 16-token chunks hashed one after another
//                    with two-limb products, 256-block tiles whatever B
//   k_hash_local     any other B or tokens not 16-byte aligned: tokens
//                    staged through padded shared memory with 16-byte
//                    loads; each thread hashes 16 tokens (one "sub-chunk")
//                    with 3 x 21-bit limbs of u^1..u^16 held as constant
//                    kernel parameters; sub-chunks of one block combine by
//                    shuffles; the segmented sum runs across the CTA.  Keys
//                    after the tile's first request start are final; the tile
//                    records its aggregate.  No tile depends on another.
//   k_hash_chain     each tile's carry from its predecessors' aggregates
//                    (all already written, so nothing waits), added to the
//                    keys of the tile's leading blocks.
#include "ptc_internal.h"

namespace ptc {
namespace {

constexpr int kOffThreads = 256;  // one request per thread: the grid spreads over many SMs
constexpr int kOffPer = 1;
constexpr int kOffTile = kOffThreads * kOffPer;

constexpr int kHashThreads = 256;
constexpr int kWinTokens = 8192 + 256;
constexpr int kWinWords = kWinTokens + kWinTokens / 16;

constexpr int kEpochOffsets = 1;
constexpr int kEpochWide = 2;  // st->tile_ctr slot counting the tiles of k_hash16_wide

// ---------------------------------------------------------------- block scans
// Exclusive sum over a CTA of kOffThreads threads; returns the CTA total in *total.
__device__ __forceinline__ uint64_t cta_exclusive_sum(uint64_t v, uint64_t* total) {
  __shared__ uint64_t s_w[kOffThreads / 32];
  const uint32_t lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  uint64_t x = v;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    uint64_t y = __shfl_up_sync(kFull, x, d);
    if (lane >= (uint32_t)d) x += y;
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    uint64_t t = lane < kOffThreads / 32 ? s_w[lane] : 0;
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      uint64_t y = __shfl_up_sync(kFull, t, d);
      if (lane >= (uint32_t)d) t += y;
    }
    if (lane < kOffThreads / 32) s_w[lane] = t;  // inclusive over warps
  }
  __syncthreads();
  uint64_t warp_excl = w ? s_w[w - 1] : 0;
  *total = s_w[kOffThreads / 32 - 1];
  return warp_excl + x - v;
}

__global__ void __launch_bounds__(kOffThreads) k_block_offsets(const uint64_t* __restrict__ tok_off,
                                                               const int64_t* __restrict__ ts, uint32_t R,
                                                               uint64_t n_tok, uint32_t B, uint32_t tb,
                                                               uint64_t* __restrict__ blk_off,
                                                               uint32_t* __restrict__ tile_req, uint64_t tile_cap,
                                                               uint64_t* lb, DevStatus* st) {
  grid_dep_sync();
  const uint32_t tile = next_tile(st, kEpochOffsets);
  const uint64_t r0 = (uint64_t)tile * kOffTile + (uint64_t)threadIdx.x * kOffPer;
  uint64_t cnt[kOffPer];
  uint64_t local = 0, kmax = 0;
  uint32_t err = 0;
#pragma unroll
  for (int j = 0; j < kOffPer; ++j) {
    uint64_t r = r0 + j;
    cnt[j] = 0;
    if (r < R) {
      uint64_t a = tok_off[r], b = tok_off[r + 1];
      if (b < a || b > n_tok) {
        err |= kErrInvalid;
      } else {
        cnt[j] = (b - a) / B;
      }
      if (ts != nullptr && r + 1 < R && ts[r + 1] < ts[r]) err |= kErrUnsorted;
      local += cnt[j];
      kmax = cnt[j] > kmax ? cnt[j] : kmax;
    }
  }
  if (err) raise_err(st, err);
  {  // the longest request: one atomic per warp
    uint64_t m = kmax;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const uint64_t y = __shfl_xor_sync(kFull, m, o);
      m = y > m ? y : m;
    }
    if ((threadIdx.x & 31) == 0 && m) atomicMax((unsigned long long*)&st->value[1], (unsigned long long)m);
  }
  uint64_t total;
  uint64_t excl = cta_exclusive_sum(local, &total);
  const uint64_t base = lookback_sum_cta(lb, tile, total, kEpochOffsets, st);
  uint64_t run = base + excl;
#pragma unroll
  for (int j = 0; j < kOffPer; ++j) {
    uint64_t r = r0 + j;
    if (r < R) {
      blk_off[r] = run;
      // hash tiles whose first block lies in this request
      if (cnt[j]) {
        const uint64_t last = (run + cnt[j] - 1) / tb;
        for (uint64_t t = (run + tb - 1) / tb; t <= last && t < tile_cap; ++t) tile_req[t] = (uint32_t)r;
      }
    }
    run += cnt[j];
    if (r + 1 == R) {
      blk_off[R] = run;
      st->value[0] = run;
      if (run >= (uint64_t)kNone) raise_err(st, kErrOverflow);
    }
  }
}

// ---------------------------------------------------------------- powers
// tables[(b*2 + w) * 65536 + e] for base b in {0,1} and
//   w = 0: u_b^(B e)          w = 1: u_b^(B 65536 e)
constexpr int kPowChunk = 8;  // powers per thread: short dependent chains

struct PowBases {
  uint64_t base[4];
};

// Only the entries some block can use are filled: exponents e = k reach at
// most the longest request's block count minus one (st->value[1]).
// Blocks the key kernels may touch: N as the offsets kernel left it, or none
// if its look-back gave up (then the offsets are not a prefix sum and must
// not steer any read; the call reports PTC_ERR_TIMEOUT).
__device__ __forceinline__ uint64_t blocks_live(const DevStatus* st, uint64_t keys_cap) {
  if (ld_relaxed_u32(&st->err) & kErrTimeout) return 0;
  const uint64_t N = st->value[0];
  return N < keys_cap ? N : keys_cap;
}

__global__ void k_pow_tables(PowBases pb, uint64_t* __restrict__ tables, const DevStatus* st) {
  grid_dep_sync();
  const uint32_t gid = blockIdx.x * blockDim.x + threadIdx.x;  // 4 tables x 8192 chunks of kPowChunk
  const uint32_t t = gid >> 13, chunk = gid & 8191;
  if (t >= 4) return;
  const uint64_t kmax = st->value[1];
  const uint64_t need = (t & 1) ? (kmax >> 16) : (kmax < 65535 ? kmax : 65535);
  const uint64_t base = pb.base[t];
  const uint64_t e0 = (uint64_t)chunk * kPowChunk;
  if (e0 > need) return;
  uint64_t v = p61_pow(base, e0);
  uint64_t* out = tables + (uint64_t)t * 65536 + e0;
  for (int i = 0; i < kPowChunk; ++i) {
    out[i] = v;
    v = p61_mul(v, base);
  }
}

__device__ __forceinline__ uint64_t pow_at(const uint64_t* __restrict__ lo, const uint64_t* __restrict__ hi,
                                           uint64_t e) {
  uint64_t v = __ldg(&lo[e & 0xFFFF]);
  const uint64_t h = e >> 16;
  if (h) v = p61_mul(v, __ldg(&hi[h & 0xFFFF]));
  return v;
}

// ---------------------------------------------------------------- hash
struct HashConsts {
  uint32_t limb[2][3][16];   // 21-bit limbs of u_b^(j + 1)
  uint32_t limb2[2][2][16];  // the same split 31 + 30 bits (tokens below 2^27)
  uint64_t csum[2][17];      // sum_{j < n} u_b^(j + 1): the "+ 1" of n tokens
  uint64_t sub_mul[2][32];   // u_b^(16 q)
};

struct HashCarry {
  uint64_t v0, v1, f;
};

struct SegSumOp {
  __device__ HashCarry operator()(const HashCarry& a, const HashCarry& b) const {
    HashCarry r;
    r.f = a.f | b.f;
    r.v0 = b.f ? b.v0 : p61_add(a.v0, b.v0);
    r.v1 = b.f ? b.v1 : p61_add(a.v1, b.v1);
    return r;
  }
};

struct HashArgs {
  const uint32_t* tokens;
  uint64_t n_tok;
  const uint64_t* tok_off;
  const uint64_t* blk_off;
  uint32_t R;
  uint32_t B;
  ulonglong2* keys;
  uint64_t keys_cap;
  const uint64_t* tables;
  const uint32_t* tile_req;
  HashCarry* tile_agg;   // per tile: (request starts inside?, sum of g after the last start)
  uint32_t* tile_lead;   // per tile: blocks before its first request start (keys left normalised)
  DevStatus* st;
  int aligned;
  uint32_t* wide_list;  // k_hash16: tiles left to k_hash16_wide (their count in st->tile_ctr[kEpochWide])
};

__device__ __forceinline__ uint32_t pad16(uint32_t i) { return i + (i >> 4); }

// 32 x 32 -> 64-bit multiply-add; written in C so the compiler can take the
// constant operand straight from the parameter bank.
__device__ __forceinline__ uint64_t mad_wide(uint32_t a, uint32_t b, uint64_t c) {
  return (uint64_t)a * (uint64_t)b + c;
}

// Sum over the 16 words t[m .. m+15] of t * u^(j + 1) for both bases, as
// 21-bit limb accumulators (M is the word offset of the first token).
template <int M, int NW>
__device__ __forceinline__ void hash16(const uint32_t (&wd)[NW], const HashConsts& c, uint64_t (&acc)[6]) {
  static_assert(M + 16 <= NW, "chunk words out of range");
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint32_t t = wd[j + M];
    acc[0] = mad_wide(t, c.limb[0][0][j], acc[0]);
    acc[1] = mad_wide(t, c.limb[0][1][j], acc[1]);
    acc[2] = mad_wide(t, c.limb[0][2][j], acc[2]);
    acc[3] = mad_wide(t, c.limb[1][0][j], acc[3]);
    acc[4] = mad_wide(t, c.limb[1][1][j], acc[4]);
    acc[5] = mad_wide(t, c.limb[1][2][j], acc[5]);
  }
}

// The same sum with two limbs (31 + 30 bits), exact when every token is
// below 2^27: 16 products of at most 2^58 stay below 2^62.
template <int M, int NW>
__device__ __forceinline__ void hash16_2(const uint32_t (&wd)[NW], const HashConsts& c, uint64_t (&acc)[4]) {
  static_assert(M + 16 <= NW, "chunk words out of range");
#pragma unroll
  for (int j = 0; j < 16; ++j) {
    const uint32_t t = wd[j + M];
    acc[0] = mad_wide(t, c.limb2[0][0][j], acc[0]);
    acc[1] = mad_wide(t, c.limb2[0][1][j], acc[1]);
    acc[2] = mad_wide(t, c.limb2[1][0][j], acc[2]);
    acc[3] = mad_wide(t, c.limb2[1][1][j], acc[3]);
  }
}

// Congruent to (a0 + a1 2^31) mod p and below 2^61 + 3, for a0, a1 < 2^62.
__device__ __forceinline__ uint64_t limbs2_lazy(uint64_t a0, uint64_t a1) {
  const uint64_t x = (a0 & kP61) + (a0 >> 61) + ((a1 & ((1ULL << 30) - 1)) << 31) + (a1 >> 30);  // < 2^62 + 2^33
  return (x & kP61) + (x >> 61);
}

// a b mod p, reduced only below 2^61 + 5, for a < 2^63 and b < p: the
// product is below 2^124, so hi << 3 < 2^63 and the first sum stays below
// 2^63 + 2^61 + 8.
__device__ __forceinline__ uint64_t p61_mul_lazy(uint64_t a, uint64_t b) {
  const uint64_t lo = a * b, hi = __umul64hi(a, b);
  const uint64_t r = (lo & kP61) + (lo >> 61) + (hi << 3);
  return (r & kP61) + (r >> 61);
}

// (a0 + a1 2^21 + a2 2^42) mod p for a0, a1, a2 < 2^62 - 2^57 (sums of <= 32 products < 2^53)
__device__ __forceinline__ uint64_t limbs_to_p61(uint64_t a0, uint64_t a1, uint64_t a2) {
  uint64_t x = a0 + ((a1 & ((1ULL << 40) - 1)) << 21) + (a1 >> 40) + ((a2 & ((1ULL << 19) - 1)) << 42) + (a2 >> 19);
  return p61_fold(x);
}

__device__ __forceinline__ uint32_t find_request(const uint64_t* __restrict__ blk_off, uint32_t lo, uint32_t hi,
                                                 uint64_t b) {
  // largest r in [lo, hi] with blk_off[r] <= b (blk_off[lo] <= b holds)
  while (lo < hi) {
    uint32_t mid = (lo + hi + 1) >> 1;
    if (__ldg(&blk_off[mid]) <= b)
      lo = mid;
    else
      hi = mid - 1;
  }
  return lo;
}

// Shared second half of the local hash kernels: combine the sub-chunks of each
// block, normalise, segmented sum over the tile, write keys and the tile's
// aggregate.  Every thread of the CTA calls it.
template <int G>
__device__ __forceinline__ void hash_finish(const HashArgs& a, uint32_t tile, uint64_t b0, uint64_t b_end, uint64_t h0,
                                            uint64_t h1, uint32_t k, uint32_t lb, uint32_t s) {
  constexpr uint32_t TB = kHashThreads / G;
  __shared__ uint64_t s_h0[kHashThreads / G], s_h1[kHashThreads / G];
  __shared__ uint32_t s_k[kHashThreads / G];
  __shared__ HashCarry s_w[kHashThreads / 32];
  __shared__ uint32_t s_first_head;
  if (G > 1) {
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) {
      h0 = p61_add(h0, __shfl_xor_sync(kFull, h0, o));
      h1 = p61_add(h1, __shfl_xor_sync(kFull, h1, o));
    }
  }
  if (G > 1) {  // one value per block: the sub-chunk holding it hands it over
    if (s == 0) {
      s_h0[lb] = h0;
      s_h1[lb] = h1;
      s_k[lb] = k;
    }
    __syncthreads();
  }

  // ---- phase 2: normalise, segmented sum over requests, denormalise
  const uint32_t t = threadIdx.x;
  const bool valid = t < TB && b0 + t < b_end;
  const uint64_t* T = a.tables;
  HashCarry x{0, 0, 0};
  uint32_t kk = 0;
  if (valid) {
    kk = G > 1 ? s_k[t] : k;
    x.v0 = p61_mul(G > 1 ? s_h0[t] : h0, pow_at(T + 0 * 65536, T + 1 * 65536, kk));
    x.v1 = p61_mul(G > 1 ? s_h1[t] : h1, pow_at(T + 2 * 65536, T + 3 * 65536, kk));
    x.f = kk == 0;
  }
  SegSumOp op;
  const uint32_t lane = t & 31, w = t >> 5;
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    HashCarry y;
    y.v0 = __shfl_up_sync(kFull, x.v0, d);
    y.v1 = __shfl_up_sync(kFull, x.v1, d);
    y.f = __shfl_up_sync(kFull, x.f, d);
    if (lane >= (uint32_t)d) x = op(y, x);
  }
  if (lane == 31) s_w[w] = x;
  __syncthreads();
  if (w == 0) {
    HashCarry z = lane < kHashThreads / 32 ? s_w[lane] : HashCarry{0, 0, 0};
#pragma unroll
    for (int d = 1; d < 32; d <<= 1) {
      HashCarry y;
      y.v0 = __shfl_up_sync(kFull, z.v0, d);
      y.v1 = __shfl_up_sync(kFull, z.v1, d);
      y.f = __shfl_up_sync(kFull, z.f, d);
      if (lane >= (uint32_t)d) z = op(y, z);
    }
    if (lane < kHashThreads / 32) s_w[lane] = z;  // inclusive over warps
  }
  __syncthreads();
  if (w > 0) x = op(s_w[w - 1], x);
  // Blocks at or after the tile's first request start are final here; the
  // leading blocks still lack the carry from earlier tiles (k_hash_chain).
  if (t == 0) s_first_head = TB;
  __syncthreads();
  if (valid && kk == 0) atomicMin(&s_first_head, t);
  __syncthreads();
  if (valid) a.keys[b0 + t] = make_ulonglong2(x.v0, x.v1);
  if (t == 0) {
    a.tile_agg[tile] = s_w[kHashThreads / 32 - 1];
    const uint32_t nb = (uint32_t)(b_end - b0);
    a.tile_lead[tile] = s_first_head < nb ? s_first_head : nb;
  }
}

template <int G, bool FULL>
__global__ void __launch_bounds__(kHashThreads) k_hash_local(HashArgs a, const __grid_constant__ HashConsts c) {
  grid_dep_sync();
  __shared__ uint32_t s_tok[kWinWords];
  __shared__ uint64_t s_bnd[4];
  constexpr uint32_t TB = kHashThreads / G;

  const uint32_t tile = blockIdx.x;
  const uint64_t N = blocks_live(a.st, a.keys_cap);
  const uint64_t b0 = (uint64_t)tile * TB;
  if (b0 >= N) return;
  const uint64_t b_end = b0 + TB < N ? b0 + TB : N;
  const uint32_t B = a.B;

  if (threadIdx.x == 0) {
    const uint64_t ntiles = (N + TB - 1) / TB;
    const uint32_t r0 = a.tile_req[tile];
    const uint32_t rh = tile + 1 < ntiles ? a.tile_req[tile + 1] : a.R - 1;
    s_bnd[0] = r0;
    s_bnd[1] = find_request(a.blk_off, r0, rh, b_end - 1);
  }
  __syncthreads();
  const uint32_t r_first = (uint32_t)s_bnd[0], r_last = (uint32_t)s_bnd[1];
  const uint64_t t_begin = a.tok_off[r_first] + (uint64_t)B * (b0 - a.blk_off[r_first]);
  const uint64_t t_end = a.tok_off[r_last] + (uint64_t)B * (b_end - a.blk_off[r_last]);
  const uint64_t w0 = a.aligned ? (t_begin & ~3ULL) : t_begin;
  uint64_t w_end = t_end < w0 + kWinTokens ? t_end : w0 + kWinTokens;
  if (w_end > a.n_tok) w_end = a.n_tok;
  __syncthreads();

  // ---- stage the token window
  if (a.aligned) {
    const uint32_t nq = (uint32_t)((w_end - w0 + 3) >> 2);
    for (uint32_t i = threadIdx.x; i < nq; i += kHashThreads) {
      const uint64_t x = w0 + 4ULL * i;
      uint4 v;
      if (x + 3 < a.n_tok) {
        v = __ldcs(reinterpret_cast<const uint4*>(a.tokens + x));
      } else {
        v.x = x < a.n_tok ? a.tokens[x] : 0u;
        v.y = x + 1 < a.n_tok ? a.tokens[x + 1] : 0u;
        v.z = x + 2 < a.n_tok ? a.tokens[x + 2] : 0u;
        v.w = 0u;
      }
      const uint32_t o = pad16(4 * i);
      s_tok[o] = v.x;
      s_tok[o + 1] = v.y;
      s_tok[o + 2] = v.z;
      s_tok[o + 3] = v.w;
    }
  } else {
    const uint32_t n = (uint32_t)(w_end - w0);
    for (uint32_t i = threadIdx.x; i < n; i += kHashThreads) s_tok[pad16(i)] = a.tokens[w0 + i];
  }
  __syncthreads();

  // ---- phase 1: 16-token sub-chunks
  const uint32_t lb = threadIdx.x / G, s = threadIdx.x % G;
  const uint64_t b = b0 + lb;
  uint64_t h0 = 0, h1 = 0;
  uint32_t k = 0;
  if (b < b_end) {
    const uint32_t r = find_request(a.blk_off, r_first, r_last, b);
    k = (uint32_t)(b - a.blk_off[r]);
    const uint32_t first = 16 * s;  // block offset of this chunk's token 0
    const uint32_t nval = first < B ? (B - first < 16 ? B - first : 16) : 0u;  // tokens of the block in the chunk
    const uint64_t bstart = a.tok_off[r] + (uint64_t)B * k;
    uint64_t a00 = 0, a01 = 0, a02 = 0, a10 = 0, a11 = 0, a12 = 0;
    const uint64_t x0 = bstart + first;
    const bool in_win = FULL && x0 >= w0 && x0 + 16 <= w_end;
    if (in_win) {
      const uint32_t rel = (uint32_t)(x0 - w0);
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        const uint64_t t = s_tok[pad16(rel + j)];
        a00 += t * c.limb[0][0][j];
        a01 += t * c.limb[0][1][j];
        a02 += t * c.limb[0][2][j];
        a10 += t * c.limb[1][0][j];
        a11 += t * c.limb[1][1][j];
        a12 += t * c.limb[1][2][j];
      }
    } else {
#pragma unroll
      for (int j = 0; j < 16; ++j) {
        if (FULL || (uint32_t)j < nval) {
          const uint64_t x = x0 + (uint64_t)j;
          uint64_t t;
          if (x >= w0 && x < w_end)
            t = s_tok[pad16((uint32_t)(x - w0))];
          else
            t = x < a.n_tok ? a.tokens[x] : 0u;
          a00 += t * c.limb[0][0][j];
          a01 += t * c.limb[0][1][j];
          a02 += t * c.limb[0][2][j];
          a10 += t * c.limb[1][0][j];
          a11 += t * c.limb[1][1][j];
          a12 += t * c.limb[1][2][j];
        }
      }
    }
    h0 = p61_add(limbs_to_p61(a00, a01, a02), c.csum[0][FULL ? 16 : nval]);
    h1 = p61_add(limbs_to_p61(a10, a11, a12), c.csum[1][FULL ? 16 : nval]);
    if (G > 1 && s > 0) {
      h0 = p61_mul(h0, c.sub_mul[0][s]);
      h1 = p61_mul(h1, c.sub_mul[1][s]);
    }
  }
  hash_finish<G>(a, tile, b0, b_end, h0, h1, k, lb, s);
}

// B = 16 with 16-byte-aligned tokens: one block per thread, kHashThreads =
// 256 blocks per tile (as k_hash_local with G = 1), eight CTAs per SM (32
// registers; a few values spill to L1, which measured faster than six CTAs
// at 40 registers), so that a CTA waiting at one of its barriers leaves seven
// others to issue.  The requests that meet the tile are
// tile_req[tile] .. tile_req[tile + 1]; their block and token offsets are
// loaded into shared memory once, so a thread finds its request without a
// dependent chain of global loads, and its token loads and power-table loads
// all go out together.  Tiles meeting more than kH16Req requests search the
// global offsets instead.
constexpr int kH16Req = 256;

// One tile of k_hash16.  WIDE = false: two-limb products, exact while every
// token is below 2^27 (any vocabulary in use); a tile that holds a larger
// token is left to k_hash16_wide (its index goes to wide_list) and returns
// before it writes anything.  WIDE = true: three-limb products, exact for
// every 32-bit token.  Keeping the three-limb code out of the common kernel
// keeps that kernel's registers free of it (with it the kernel spilled more
// and took 0.7 ms longer on the mixed 10B-token trace).
template <bool WIDE>
__device__ __forceinline__ void hash16_tile(const HashArgs& a, const HashConsts& c, uint32_t tile, uint64_t N) {
  __shared__ uint64_t s_boff[kH16Req + 1];
  __shared__ uint64_t s_toff[kH16Req + 1];
  __shared__ uint32_t s_big;  // some block of the tile needs three limbs
  constexpr uint32_t TB = kHashThreads;
  const uint64_t b0 = (uint64_t)tile * TB;
  if (b0 >= N) return;
  const uint64_t b_end = b0 + TB < N ? b0 + TB : N;
  const uint64_t ntiles = (N + TB - 1) / TB;
  const uint32_t r_first = a.tile_req[tile];
  const uint32_t r_last = tile + 1 < ntiles ? a.tile_req[tile + 1] : a.R - 1;  // the last request meeting the tile
  const uint32_t nreq = r_last - r_first + 1;
  const bool cached = nreq <= kH16Req;
  if (cached) {
    for (uint32_t i = threadIdx.x; i <= nreq; i += kHashThreads) {
      s_boff[i] = a.blk_off[r_first + i];
      s_toff[i] = a.tok_off[r_first + i];
    }
  }
  if (threadIdx.x == 0) s_big = 0;
  __syncthreads();
  const uint32_t t = threadIdx.x;
  const uint64_t b = b0 + t;
  uint64_t h0 = 0, h1 = 0;
  uint32_t k = 0;
  uint64_t wd_x = 0;  // token offset of this thread's block
  uint64_t rstart = 0;  // first block of its request
  if (b < b_end) {
    uint64_t x;
    if (cached) {  // largest i with s_boff[i] <= b
      uint32_t lo = 0, hi = nreq - 1;
      while (lo < hi) {
        const uint32_t mid = (lo + hi + 1) >> 1;
        if (s_boff[mid] <= b)
          lo = mid;
        else
          hi = mid - 1;
      }
      rstart = s_boff[lo];
      k = (uint32_t)(b - rstart);
      x = s_toff[lo] + 16ULL * k;
    } else {
      const uint32_t r = find_request(a.blk_off, r_first, r_last, b);
      rstart = a.blk_off[r];
      k = (uint32_t)(b - rstart);
      x = a.tok_off[r] + 16ULL * k;
    }
    wd_x = x;
  }
  // Each lane reads the four aligned 16-byte words that start its 16 tokens;
  // a block that does not start on a 16-byte boundary also needs the first
  // one to three words of the next 16, which the next lane holds when its
  // block follows on directly (the usual case inside a request).
  const uint32_t m = (uint32_t)(wd_x & 3);
  const uint64_t x4 = wd_x - m;
  uint32_t wd[20];
  const bool live = b < b_end;
  const bool whole = live && x4 + 16 <= a.n_tok;
  {
    const uint4* q4 = reinterpret_cast<const uint4*>(a.tokens + x4);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (whole) v = __ldcs(q4 + q);
      wd[4 * q] = v.x;
      wd[4 * q + 1] = v.y;
      wd[4 * q + 2] = v.z;
      wd[4 * q + 3] = v.w;
    }
    if (live && !whole) {
#pragma unroll
      for (int q = 0; q < 16; ++q) wd[q] = x4 + q < a.n_tok ? a.tokens[x4 + q] : 0u;
    }
  }
  const uint64_t x_next = __shfl_down_sync(kFull, wd_x, 1);
  const uint32_t n0 = __shfl_down_sync(kFull, wd[0], 1), n1 = __shfl_down_sync(kFull, wd[1], 1),
                 n2 = __shfl_down_sync(kFull, wd[2], 1);
  const bool follows = (threadIdx.x & 31) != 31 && x_next == wd_x + 16 && whole;
  wd[16] = n0;
  wd[17] = n1;
  wd[18] = n2;
  wd[19] = 0;
  if (live && m && !follows) {
    const uint64_t y = x4 + 16;
    if (y + 4 <= a.n_tok) {
      const uint4 v = __ldcs(reinterpret_cast<const uint4*>(a.tokens + y));
      wd[16] = v.x;
      wd[17] = v.y;
      wd[18] = v.z;
    } else {
      wd[16] = y < a.n_tok ? a.tokens[y] : 0u;
      wd[17] = y + 1 < a.n_tok ? a.tokens[y + 1] : 0u;
      wd[18] = y + 2 < a.n_tok ? a.tokens[y + 2] : 0u;
    }
  }
  if (live) {
    if (!WIDE) {  // a token (or a word around the block: that only widens the test) reaching 2^27
      uint32_t any = 0;
#pragma unroll
      for (int j = 0; j < 19; ++j) any |= wd[j];
      if (any >> 27) s_big = 1;
      uint64_t acc[4] = {0, 0, 0, 0};
      switch (m) {
        case 0: hash16_2<0>(wd, c, acc); break;
        case 1: hash16_2<1>(wd, c, acc); break;
        case 2: hash16_2<2>(wd, c, acc); break;
        default: hash16_2<3>(wd, c, acc); break;
      }
      // lazily reduced (below 2^62 + 3); p61_mul_lazy takes it as it is
      h0 = limbs2_lazy(acc[0], acc[1]) + c.csum[0][16];
      h1 = limbs2_lazy(acc[2], acc[3]) + c.csum[1][16];
    } else {  // three limbs
      uint64_t acc[6] = {0, 0, 0, 0, 0, 0};
      switch (m) {
        case 0: hash16<0>(wd, c, acc); break;
        case 1: hash16<1>(wd, c, acc); break;
        case 2: hash16<2>(wd, c, acc); break;
        default: hash16<3>(wd, c, acc); break;
      }
      h0 = p61_add(limbs_to_p61(acc[0], acc[1], acc[2]), c.csum[0][16]);
      h1 = p61_add(limbs_to_p61(acc[3], acc[4], acc[5]), c.csum[1][16]);
    }
  }
  // g = h u^(16 k), then a plain prefix sum over the tile; a block whose
  // request starts inside the tile at index s subtracts the prefix before s.
  const uint64_t* T = a.tables;
  uint64_t v0 = 0, v1 = 0;  // below 2^61 + 5
  if (live) {
    v0 = p61_mul_lazy(h0, pow_at(T + 0 * 65536, T + 1 * 65536, k));
    v1 = p61_mul_lazy(h1, pow_at(T + 2 * 65536, T + 3 * 65536, k));
  }
  __shared__ uint64_t s_p0[kHashThreads], s_p1[kHashThreads];
  __shared__ uint64_t s_w0[kHashThreads / 32], s_w1[kHashThreads / 32];
  const uint32_t lane = t & 31, w = t >> 5;
  // warp scan with lazy reduction: from values below 2^61 + 5, two plain
  // steps stay below 2^63 + 20; a fold (x & p) + (x >> 61) brings such a sum
  // back below 2^61 + 4, so folding after d = 2 and d = 8 keeps every sum
  // below 2^64 and leaves the result below 2^62 + 8
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t y0 = __shfl_up_sync(kFull, v0, d), y1 = __shfl_up_sync(kFull, v1, d);
    if (lane >= (uint32_t)d) {
      v0 += y0;
      v1 += y1;
    }
    if (d == 2 || d == 8) {
      v0 = (v0 & kP61) + (v0 >> 61);
      v1 = (v1 & kP61) + (v1 >> 61);
    }
  }
  if (lane == 31) {
    s_w0[w] = v0;
    s_w1[w] = v1;
  }
  __syncthreads();
  if (!WIDE && s_big) {  // the tile goes to k_hash16_wide, which writes all of it
    if (t == 0) a.wide_list[atomicAdd(&a.st->tile_ctr[kEpochWide], 1u)] = tile;
    return;
  }
  if (w == 0) {  // exclusive prefix of the warp totals
    uint64_t z0 = lane < kHashThreads / 32 ? s_w0[lane] : 0, z1 = lane < kHashThreads / 32 ? s_w1[lane] : 0;
    const uint64_t x0 = z0, x1 = z1;
#pragma unroll
    for (int d = 1; d < kHashThreads / 32; d <<= 1) {
      const uint64_t y0 = __shfl_up_sync(kFull, z0, d), y1 = __shfl_up_sync(kFull, z1, d);
      if (lane >= (uint32_t)d) {
        z0 += y0;
        z1 += y1;
      }
      z0 = (z0 & kP61) + (z0 >> 61);
      z1 = (z1 & kP61) + (z1 >> 61);
    }
    if (lane < kHashThreads / 32) {
      s_w0[lane] = p61_fold(z0 + (kP61 << 2) - x0);  // z < 2^61 + 4, x < 2^62 + 8: stays in (0, 2^64)
      s_w1[lane] = p61_fold(z1 + (kP61 << 2) - x1);
    }
  }
  __syncthreads();
  v0 = p61_fold(v0 + s_w0[w]);
  v1 = p61_fold(v1 + s_w1[w]);
  // A request starting after b0 inside the tile subtracts the prefix before
  // its start; when none does (a long request spans the tile), the prefixes
  // are not exchanged.
  const bool inner = !cached || (nreq >= 2 && s_boff[1] < b_end);
  if (inner) {
    s_p0[t] = v0;
    s_p1[t] = v1;
    __syncthreads();
  }
  if (live) {
    const bool own_start = rstart >= b0;  // the request starts in this tile
    if (inner && own_start && rstart > b0) {
      const uint32_t sl = (uint32_t)(rstart - b0) - 1;
      v0 = p61_add(v0, kP61 - s_p0[sl]);
      v1 = p61_add(v1, kP61 - s_p1[sl]);
    }
    a.keys[b] = make_ulonglong2(v0, v1);
  }
  // the tile's aggregate for k_hash_chain: the last block's sum since its
  // request's start, and whether that start is in the tile; and the leading
  // blocks (before the tile's first request start)
  if (b + 1 == b_end) {
    HashCarry agg;
    agg.f = rstart >= b0;
    agg.v0 = v0;
    agg.v1 = v1;
    a.tile_agg[tile] = agg;
  }
  if (t == 0) {
    uint32_t lead = (uint32_t)(b_end - b0);
    if (cached) {
      for (uint32_t i = 0; i < nreq; ++i)
        if (s_boff[i] >= b0 && s_boff[i] < b_end && s_boff[i + 1] > s_boff[i]) {
          lead = (uint32_t)(s_boff[i] - b0);
          break;
        }
    } else {
      for (uint32_t r = r_first; r <= r_last; ++r) {
        const uint64_t st0 = a.blk_off[r];
        if (st0 >= b0 && st0 < b_end && a.blk_off[r + 1] > st0) {
          lead = (uint32_t)(st0 - b0);
          break;
        }
      }
    }
    a.tile_lead[tile] = lead;
  }
}

__global__ void __launch_bounds__(kHashThreads, 8) k_hash16(HashArgs a, const __grid_constant__ HashConsts c) {
  grid_dep_sync();
  hash16_tile<false>(a, c, blockIdx.x, blocks_live(a.st, a.keys_cap));
}

// The tiles k_hash16 left (a token at or above 2^27), a persistent grid over
// the list it wrote.
__global__ void __launch_bounds__(kHashThreads) k_hash16_wide(HashArgs a, const __grid_constant__ HashConsts c) {
  grid_dep_sync();
  const uint64_t N = blocks_live(a.st, a.keys_cap);
  const uint32_t n_wide = ld_relaxed_u32(&a.st->tile_ctr[kEpochWide]);
  for (uint32_t j = blockIdx.x; j < n_wide; j += gridDim.x) {
    const uint32_t tile = a.wide_list[j];
    if (in_bounds(a.st, tile, (N + kHashThreads - 1) / kHashThreads)) hash16_tile<true>(a, c, tile, N);
    __syncthreads();  // the next tile reuses the shared arrays
  }
}

// B a multiple of 16 (g = B / 16 chunks of 16 tokens) with 16-byte-aligned
// tokens: P consecutive blocks per thread (one here; two would suit B = 16,
// which k_hash16 takes), tiles of kHashThreads = 256 blocks whatever B,
// kHashThreads / P threads per CTA, 64 registers.
// The requests that meet the tile are tile_req[tile] .. tile_req[tile + 1];
// their block and token offsets are loaded into shared memory once, so a
// thread finds its request without a dependent chain of global loads.  A
// thread hashes its P g chunks one after another in one loop (four or five
// 16-byte loads each), so the code of the chunk product exists once and the
// registers of one chunk are live at a time: h_b = sum over chunks s of
// h_(b,s) u^(16 s).  The prefix sum then runs over one value per thread.
// Tiles meeting more than kH16Req requests search the global offsets.
// The 20 words x4 .. x4 + 19 of a 16-token chunk whose first token is word
// m of them (the fifth 16-byte load only when m > 0).
__device__ __forceinline__ void load_chunk(const HashArgs& a, uint64_t x4, uint32_t m, uint32_t (&wd)[20]) {
  if (x4 + 20 <= a.n_tok) {
    const uint4* q4 = reinterpret_cast<const uint4*>(a.tokens + x4);
#pragma unroll
    for (int q = 0; q < 5; ++q) {
      uint4 v = make_uint4(0, 0, 0, 0);
      if (q < 4 || m != 0) v = __ldcs(q4 + q);
      wd[4 * q] = v.x;
      wd[4 * q + 1] = v.y;
      wd[4 * q + 2] = v.z;
      wd[4 * q + 3] = v.w;
    }
  } else {  // within 20 words of the end of the token array
#pragma unroll
    for (int q = 0; q < 20; ++q) wd[q] = x4 + q < a.n_tok ? a.tokens[x4 + q] : 0u;
  }
}

// h of the 16 tokens wd[M .. M+15] for both bases, every token below 2^27:
// below 2^62 + 2.
template <int M>
__device__ __forceinline__ void chunk_narrow(const uint32_t (&wd)[20], const HashConsts& c, uint64_t& e0, uint64_t& e1) {
  uint64_t acc[4] = {0, 0, 0, 0};
  hash16_2<M>(wd, c, acc);
  e0 = limbs2_lazy(acc[0], acc[1]) + c.csum[0][16];
  e1 = limbs2_lazy(acc[2], acc[3]) + c.csum[1][16];
}

// The same for any 32-bit tokens (three limbs), fully reduced.
template <int M>
__device__ __forceinline__ void chunk_wide(const uint32_t (&wd)[20], const HashConsts& c, uint64_t& e0, uint64_t& e1) {
  uint64_t acc[6] = {0, 0, 0, 0, 0, 0};
  hash16<M>(wd, c, acc);
  e0 = p61_add(limbs_to_p61(acc[0], acc[1], acc[2]), c.csum[0][16]);
  e1 = p61_add(limbs_to_p61(acc[3], acc[4], acc[5]), c.csum[1][16]);
}

// Chunk s of a block into its h: h_s u^(16 s) added to the chunks before,
// kept below 2^62 + 2 by one fold (the first chunk is taken as it is).
__device__ __forceinline__ void chunk_add(const HashConsts& c, uint32_t s, uint64_t e0, uint64_t e1, uint64_t& h0,
                                          uint64_t& h1) {
  if (s == 0) {
    h0 = e0;
    h1 = e1;
    return;
  }
  h0 += p61_mul_lazy(e0, c.sub_mul[0][s]);
  h1 += p61_mul_lazy(e1, c.sub_mul[1][s]);
  h0 = (h0 & kP61) + (h0 >> 61);
  h1 = (h1 & kP61) + (h1 >> 61);
}

// B a multiple of 16 (g = B / 16 chunks of 16 tokens) with 16-byte-aligned
// tokens, B > 16: one block per thread, tiles of kHashThreads = 256 blocks
// whatever B, four CTAs per SM (64 registers).  The requests that meet the
// tile are tile_req[tile] .. tile_req[tile + 1]; their block and token
// offsets are loaded into shared memory once, so a thread finds its request
// without a dependent chain of global loads.  A thread hashes its block's g
// chunks one after another in one loop (four or five 16-byte loads each), so
// the code of the chunk product exists once and the registers of one chunk
// are live at a time: h = sum over chunks s of h_s u^(16 s).  Tiles meeting
// more than kTileReq requests search the global offsets.
constexpr int kTileReq = 256;

__global__ void __launch_bounds__(kHashThreads, 4) k_hash_tile(HashArgs a, const __grid_constant__ HashConsts c) {
  constexpr uint32_t TB = kHashThreads;
  grid_dep_sync();
  __shared__ uint64_t s_boff[kTileReq + 1];
  __shared__ uint64_t s_toff[kTileReq + 1];
  __shared__ uint64_t s_p0[TB], s_p1[TB];
  __shared__ uint64_t s_w0[TB / 32], s_w1[TB / 32];
  const uint32_t tile = blockIdx.x;
  const uint64_t N = blocks_live(a.st, a.keys_cap);
  const uint64_t b0 = (uint64_t)tile * TB;
  if (b0 >= N) return;
  const uint64_t b_end = b0 + TB < N ? b0 + TB : N;
  const uint64_t ntiles = (N + TB - 1) / TB;
  const uint32_t r_first = a.tile_req[tile];
  const uint32_t r_last = tile + 1 < ntiles ? a.tile_req[tile + 1] : a.R - 1;  // the last request meeting the tile
  const uint32_t nreq = r_last - r_first + 1;
  const bool cached = nreq <= kTileReq;
  if (cached) {
    for (uint32_t i = threadIdx.x; i <= nreq; i += TB) {
      s_boff[i] = a.blk_off[r_first + i];
      s_toff[i] = a.tok_off[r_first + i];
    }
  }
  __syncthreads();
  const uint32_t t = threadIdx.x, lane = t & 31, w = t >> 5;
  const uint32_t g = a.B / 16;
  const uint64_t b = b0 + t;
  const bool live = b < b_end;
  // the block's request starts at block rs, the block's tokens at xb
  uint64_t rs = 0, xb = 0;
  if (live) {
    if (cached) {  // largest i with s_boff[i] <= b
      uint32_t lo = 0, hi = nreq - 1;
      while (lo < hi) {
        const uint32_t mid = (lo + hi + 1) >> 1;
        if (s_boff[mid] <= b)
          lo = mid;
        else
          hi = mid - 1;
      }
      rs = s_boff[lo];
      xb = s_toff[lo] + (uint64_t)a.B * (b - rs);
    } else {
      const uint32_t r = find_request(a.blk_off, r_first, r_last, b);
      rs = a.blk_off[r];
      xb = a.tok_off[r] + (uint64_t)a.B * (b - rs);
    }
  }
  // h of the block, below 2^62 + 2.  The loop takes every chunk with
  // two-limb products; a block with a token of 2^27 or more is redone with
  // three limbs in a second loop (never taken over a real vocabulary), so
  // the two paths' registers are not live together.  (Loop bounds rather than
  // an enclosing branch, and the first loop running to its end: this shape
  // spills the fewest registers at 64.)
  uint64_t h0 = 0, h1 = 0;
  bool wide = false;
  const uint32_t gl = live ? g : 0u;
  {
#pragma unroll 1
    for (uint32_t s = 0; s < gl; ++s) {
      const uint64_t x = xb + 16ULL * s;
      const uint32_t m = (uint32_t)(x & 3);
      uint32_t wd[20];
      load_chunk(a, x - m, m, wd);
      uint32_t any = 0;  // words outside the chunk only widen the test
#pragma unroll
      for (int q = 0; q < 20; ++q) any |= wd[q];
      if (any >> 27) {
        wide = true;
        continue;
      }
      uint64_t e0, e1;
      switch (m) {
        case 0: chunk_narrow<0>(wd, c, e0, e1); break;
        case 1: chunk_narrow<1>(wd, c, e0, e1); break;
        case 2: chunk_narrow<2>(wd, c, e0, e1); break;
        default: chunk_narrow<3>(wd, c, e0, e1); break;
      }
      chunk_add(c, s, e0, e1, h0, h1);
    }
  }
  if (wide) {
#pragma unroll 1
    for (uint32_t s = 0; s < g; ++s) {
      const uint64_t x = xb + 16ULL * s;
      const uint32_t m = (uint32_t)(x & 3);
      uint32_t wd[20];
      load_chunk(a, x - m, m, wd);
      uint64_t e0, e1;
      switch (m) {
        case 0: chunk_wide<0>(wd, c, e0, e1); break;
        case 1: chunk_wide<1>(wd, c, e0, e1); break;
        case 2: chunk_wide<2>(wd, c, e0, e1); break;
        default: chunk_wide<3>(wd, c, e0, e1); break;
      }
      chunk_add(c, s, e0, e1, h0, h1);
    }
  }
  // g = h u^(B k) for the block's depth k (the tables hold u^(B e)), below
  // 2^61 + 5, then a plain prefix sum over the tile; a block whose request
  // starts inside the tile at index s subtracts the prefix before s.
  const uint64_t* T = a.tables;
  uint64_t v0 = 0, v1 = 0;
  if (live) {
    const uint32_t k = (uint32_t)(b - rs);
    v0 = p61_mul_lazy(h0, pow_at(T + 0 * 65536, T + 1 * 65536, k));
    v1 = p61_mul_lazy(h1, pow_at(T + 2 * 65536, T + 3 * 65536, k));
  }
  // warp scan with lazy reduction: from values below 2^61 + 5, two plain
  // steps stay below 2^63 + 20; a fold (x & p) + (x >> 61) brings such a sum
  // back below 2^61 + 4, so folding after d = 2 and d = 8 keeps every sum
  // below 2^64 and leaves the result below 2^62 + 8
#pragma unroll
  for (int d = 1; d < 32; d <<= 1) {
    const uint64_t y0 = __shfl_up_sync(kFull, v0, d), y1 = __shfl_up_sync(kFull, v1, d);
    if (lane >= (uint32_t)d) {
      v0 += y0;
      v1 += y1;
    }
    if (d == 2 || d == 8) {
      v0 = (v0 & kP61) + (v0 >> 61);
      v1 = (v1 & kP61) + (v1 >> 61);
    }
  }
  if (lane == 31) {
    s_w0[w] = v0;
    s_w1[w] = v1;
  }
  __syncthreads();
  if (w == 0) {  // exclusive prefix of the warp totals
    constexpr int NW = TB / 32;
    uint64_t z0 = lane < NW ? s_w0[lane] : 0, z1 = lane < NW ? s_w1[lane] : 0;
    const uint64_t o0 = z0, o1 = z1;
#pragma unroll
    for (int d = 1; d < NW; d <<= 1) {
      const uint64_t y0 = __shfl_up_sync(kFull, z0, d), y1 = __shfl_up_sync(kFull, z1, d);
      if (lane >= (uint32_t)d) {
        z0 += y0;
        z1 += y1;
      }
      z0 = (z0 & kP61) + (z0 >> 61);
      z1 = (z1 & kP61) + (z1 >> 61);
    }
    if (lane < NW) {
      s_w0[lane] = p61_fold(z0 + (kP61 << 2) - o0);  // z < 2^61 + 4, o < 2^62 + 8: stays in (0, 2^64)
      s_w1[lane] = p61_fold(z1 + (kP61 << 2) - o1);
    }
  }
  __syncthreads();
  v0 = p61_fold(v0 + s_w0[w]);
  v1 = p61_fold(v1 + s_w1[w]);
  s_p0[t] = v0;
  s_p1[t] = v1;
  __syncthreads();
  if (live && rs > b0) {  // the request starts inside the tile, after its first block
    const uint32_t sl = (uint32_t)(rs - b0) - 1;
    v0 = p61_add(v0, kP61 - s_p0[sl]);
    v1 = p61_add(v1, kP61 - s_p1[sl]);
  }
  if (live) a.keys[b] = make_ulonglong2(v0, v1);
  // the tile's aggregate for the carry: the last block's sum since its
  // request's start, and whether that start is in the tile; and the leading
  // blocks (before the tile's first request start)
  if (live && b + 1 == b_end) a.tile_agg[tile] = HashCarry{v0, v1, rs >= b0};
  if (t == 0) {
    uint32_t lead = (uint32_t)(b_end - b0);
    if (cached) {
      for (uint32_t i = 0; i < nreq; ++i)
        if (s_boff[i] >= b0 && s_boff[i] < b_end && s_boff[i + 1] > s_boff[i]) {
          lead = (uint32_t)(s_boff[i] - b0);
          break;
        }
    } else {
      for (uint32_t r = r_first; r <= r_last; ++r) {
        const uint64_t st0 = a.blk_off[r];
        if (st0 >= b0 && st0 < b_end && a.blk_off[r + 1] > st0) {
          lead = (uint32_t)(st0 - b0);
          break;
        }
      }
    }
    a.tile_lead[tile] = lead;
  }
}

// Carry of every tile = the segmented sum of the aggregates of the tiles
// before it, back to (and including) the nearest one where a request starts.
// All aggregates exist before this kernel starts, so nothing waits.  One warp
// per tile: each round reads 32 predecessors; then the carry is added to the
// tile's leading blocks (the tail of a request that started earlier).
constexpr int kChainWarps = 8;
__global__ void __launch_bounds__(kChainWarps * 32) k_hash_chain(ulonglong2* __restrict__ keys,
                                                                 const HashCarry* __restrict__ tile_agg,
                                                                 const uint32_t* __restrict__ tile_lead, uint32_t TB,
                                                                 const DevStatus* st, uint64_t keys_cap) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t tile = blockIdx.x * kChainWarps + (threadIdx.x >> 5);
  const uint64_t N = blocks_live(st, keys_cap);
  const uint64_t b0 = (uint64_t)tile * TB;
  if (b0 >= N || tile == 0) return;
  const uint32_t lead = tile_lead[tile];
  if (lead == 0 || !in_bounds(st, b0 + lead - 1, keys_cap)) return;
  uint64_t c0 = 0, c1 = 0;
  for (int64_t base = (int64_t)tile - 1; base >= 0; base -= 32) {
    const int64_t idx = base - (int64_t)lane;
    HashCarry g{0, 0, 0};
    if (idx >= 0) g = tile_agg[idx];
    const uint32_t heads = __ballot_sync(kFull, idx >= 0 && g.f);
    const uint32_t first = heads ? (uint32_t)(__ffs(heads) - 1) : 31u;
    uint64_t v0 = lane <= first ? g.v0 : 0, v1 = lane <= first ? g.v1 : 0;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      v0 = p61_add(v0, __shfl_xor_sync(kFull, v0, o));
      v1 = p61_add(v1, __shfl_xor_sync(kFull, v1, o));
    }
    c0 = p61_add(c0, v0);
    c1 = p61_add(c1, v1);
    if (heads) break;
  }
  for (uint32_t i = lane; i < lead; i += 32) {
    const ulonglong2 k = keys[b0 + i];
    keys[b0 + i] = make_ulonglong2(p61_add(k.x, c0), p61_add(k.y, c1));
  }
}

// The same carries as k_hash_chain, left for the keys' reader instead of
// added to the keys (a pipeline that does not return the keys saves the
// pass over them): carry[t] and lead[t] per tile, 0 where no key needs one.
// A warp takes kCarryPer consecutive tiles: the carry into the first from a
// look-back over the aggregates before it (all written, so nothing waits),
// then a segmented scan of its own tiles' aggregates across kCarryPer lanes.
constexpr int kCarryPer = 8;
__global__ void __launch_bounds__(kChainWarps * 32) k_hash_carry(const HashCarry* __restrict__ tile_agg,
                                                                 const uint32_t* __restrict__ tile_lead, uint32_t TB,
                                                                 const DevStatus* st, uint64_t keys_cap,
                                                                 uint32_t ntiles, ulonglong2* __restrict__ carry,
                                                                 uint32_t* __restrict__ lead_out) {
  grid_dep_sync();
  const uint32_t lane = threadIdx.x & 31;
  const uint32_t t0 = (blockIdx.x * kChainWarps + (threadIdx.x >> 5)) * kCarryPer;
  if (t0 >= ntiles) return;
  const uint64_t N = blocks_live(st, keys_cap);
  const uint64_t live = (N + TB - 1) / TB;  // tiles that hold blocks
  const SegSumOp op;
  HashCarry cin{0, 0, 0};
  if (t0 > 0 && t0 < live) {
    for (int64_t base = (int64_t)t0 - 1; base >= 0; base -= 32) {
      const int64_t idx = base - (int64_t)lane;
      HashCarry g{0, 0, 0};
      if (idx >= 0) g = tile_agg[idx];
      const uint32_t heads = __ballot_sync(kFull, idx >= 0 && g.f);
      const uint32_t first = heads ? (uint32_t)(__ffs(heads) - 1) : 31u;
      uint64_t v0 = lane <= first ? g.v0 : 0, v1 = lane <= first ? g.v1 : 0;
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) {
        v0 = p61_add(v0, __shfl_xor_sync(kFull, v0, o));
        v1 = p61_add(v1, __shfl_xor_sync(kFull, v1, o));
      }
      cin.v0 = p61_add(cin.v0, v0);
      cin.v1 = p61_add(cin.v1, v1);
      if (heads) break;
    }
  }
  const uint32_t t = t0 + lane;
  HashCarry g{0, 0, 0};
  if (lane < kCarryPer && t < live) g = tile_agg[t];
#pragma unroll
  for (int o = 1; o < kCarryPer; o <<= 1) {  // inclusive segmented sums over lanes 0 .. kCarryPer - 1
    HashCarry y;
    y.v0 = __shfl_up_sync(kFull, g.v0, o);
    y.v1 = __shfl_up_sync(kFull, g.v1, o);
    y.f = __shfl_up_sync(kFull, g.f, o);
    if (lane >= (uint32_t)o) g = op(y, g);
  }
  HashCarry before;  // this warp's tiles before tile t
  before.v0 = __shfl_up_sync(kFull, g.v0, 1);
  before.v1 = __shfl_up_sync(kFull, g.v1, 1);
  before.f = __shfl_up_sync(kFull, g.f, 1);
  if (lane == 0) before = HashCarry{0, 0, 0};
  const HashCarry c = op(cin, before);
  if (lane < kCarryPer && t < ntiles) {
    const uint64_t b0 = (uint64_t)t * TB;
    const uint32_t lead = (b0 >= N || t == 0) ? 0u : tile_lead[t];
    carry[t] = lead ? make_ulonglong2(c.v0, c.v1) : make_ulonglong2(0, 0);
    lead_out[t] = lead;
  }
}

template <int G>
void launch_hash(uint32_t grid, cudaStream_t s, const HashArgs& a, const HashConsts& c, bool full) {
  if (G == 1 && full && a.aligned) {
    PTC_KERNEL("k_hash16", s, k_hash16, grid, kHashThreads, 0, a, c);
    const uint32_t wgrid = grid < (uint32_t)(2 * num_sms()) ? grid : (uint32_t)(2 * num_sms());
    PTC_KERNEL("k_hash16_wide", s, k_hash16_wide, wgrid, kHashThreads, 0, a, c);
  }
  else if (a.aligned && a.B % 16 == 0)
    PTC_KERNEL("k_hash_tile", s, k_hash_tile, grid, kHashThreads, 0, a, c);
  else if (full)
    PTC_KERNEL("k_hash_local", s, (k_hash_local<G, true>), grid, kHashThreads, 0, a, c);
  else
    PTC_KERNEL("k_hash_local", s, (k_hash_local<G, false>), grid, kHashThreads, 0, a, c);
}

uint32_t chunks_per_block(uint32_t B) {  // G: power of two >= ceil(B / 16)
  uint32_t need = (B + 15) / 16, g = 1;
  while (g < need) g <<= 1;
  return g;
}

// Blocks per hash tile: kHashThreads for k_hash16 and k_hash_tile (B a
// multiple of 16 over 16-byte-aligned tokens), one CTA's kHashThreads / G for
// k_hash_local.  Arrays sized per tile take the smaller (the alignment of the
// tokens is not known there).
uint32_t tile_blocks(uint32_t B, bool aligned) {
  return aligned && B % 16 == 0 ? (uint32_t)kHashThreads : kHashThreads / chunks_per_block(B);
}
uint32_t min_tile_blocks(uint32_t B) { return tile_blocks(B, false); }

struct HashLayout {
  DevStatus* st;
  uint64_t* lb_off;
  HashCarry* tile_agg;
  uint32_t* tile_lead;
  uint64_t* tables;
  uint32_t* tile_req;
  uint32_t* wide_list;
  uint64_t hash_tiles;
  size_t zero_bytes;
  size_t total;
};

HashLayout hash_layout(void* ws, uint32_t n_req, uint64_t n_tok, uint32_t B, uint64_t keys_cap) {
  HashLayout L;
  Carver cv(ws);
  const uint32_t off_tiles = ceil_div_u32(n_req, kOffTile) + 1;
  const uint64_t nb = n_tok / B < keys_cap ? n_tok / B : keys_cap;
  const uint32_t tb = min_tile_blocks(B);
  const uint32_t hash_tiles = ceil_div_u32(nb, tb) + 1;
  L.st = cv.take<DevStatus>(1);
  L.lb_off = cv.take<uint64_t>(off_tiles);
  L.zero_bytes = cv.off;
  L.tile_agg = cv.take<HashCarry>(hash_tiles);
  L.tile_lead = cv.take<uint32_t>(hash_tiles);
  L.tables = cv.take<uint64_t>(4 * 65536);
  L.tile_req = cv.take<uint32_t>(hash_tiles + 1);
  L.wide_list = cv.take<uint32_t>(hash_tiles);
  L.hash_tiles = hash_tiles;
  L.total = cv.bytes();
  return L;
}

}  // namespace
}  // namespace ptc

using namespace ptc;

uint64_t ptc::hash_carry_tiles(uint64_t n_tok, uint32_t block_size) {
  if (block_size == 0) block_size = 1;
  return ceil_div_u32(n_tok / block_size, min_tile_blocks(block_size)) + 1;
}

extern "C" size_t ptc_hash_blocks_workspace_bytes(uint32_t n_req, uint64_t n_tok, uint32_t block_size) {
  if (block_size == 0) block_size = 1;
  return hash_layout(nullptr, n_req, n_tok, block_size, ~0ULL).total;
}

ptc_status ptc::hash_impl(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off,
                         const int64_t* req_ts_us, uint32_t n_req, uint32_t block_size, uint64_t seed,
                         ptc_u128* keys_out, uint64_t keys_cap, uint64_t* req_blk_off_out,
                         uint64_t* n_access_host_out, void* ws, size_t ws_bytes, cudaStream_t s, uint64_t* n_slot,
                         uint32_t* err_slot, KeyCarry* carry) {
  if (block_size < 1 || block_size > PTC_MAX_BLOCK_SIZE) return PTC_ERR_INVALID_ARG;
  if (req_tok_off == nullptr || req_blk_off_out == nullptr || n_access_host_out == nullptr)
    return PTC_ERR_INVALID_ARG;
  if (n_tok > 0 && tokens == nullptr) return PTC_ERR_INVALID_ARG;
  if (keys_cap > 0 && keys_out == nullptr) return PTC_ERR_INVALID_ARG;
  const bool deferred = n_slot != nullptr && err_slot != nullptr;
  const HashLayout need = hash_layout(nullptr, n_req, n_tok, block_size, ~0ULL);
  if (!ws_ok(ws, ws_bytes, need.total)) return PTC_ERR_WORKSPACE;
  const HashLayout L = hash_layout(ws, n_req, n_tok, block_size, ~0ULL);
  *n_access_host_out = 0;
  if (begin_call(ws, L.zero_bytes, s) != PTC_OK) return PTC_ERR_CUDA;
  const uint32_t wait_test = test_wait_polls();
  if (wait_test && fill_async(&L.st->wait_test, wait_test, sizeof(uint32_t), s) != PTC_OK) return PTC_ERR_CUDA;
  if (n_req == 0) {
    if (fill_async(req_blk_off_out, 0u, sizeof(uint64_t), s) != PTC_OK) return PTC_ERR_CUDA;
    if (deferred) return defer_status(L.st, err_slot, s, n_slot, 0);
    DevStatus h;
    return end_call(L.st, s, &h);
  }
  const uint32_t G = chunks_per_block(block_size);
  const bool aligned = (((uintptr_t)tokens) & 15) == 0;
  const uint32_t tb = tile_blocks(block_size, aligned);
  PTC_KERNEL("k_block_offsets", s, k_block_offsets, ceil_div_u32(n_req, kOffTile), kOffThreads, 0, req_tok_off, req_ts_us, n_req, n_tok, block_size, tb, req_blk_off_out, L.tile_req, L.hash_tiles, L.lb_off, L.st);

  // seeded bases and their derived constants
  PowBases pb;
  HashConsts hc;
  for (int b = 0; b < 2; ++b) {
    const uint64_t u = 2 + splitmix64_at(seed, (uint64_t)b) % (kP61 - 3);
    const uint64_t uB = p61_pow(u, block_size);
    pb.base[b * 2 + 0] = uB;
    pb.base[b * 2 + 1] = p61_pow(uB, 65536);
    uint64_t sum = 0;
    hc.csum[b][0] = 0;
    for (int j = 0; j < 16; ++j) {
      const uint64_t v = p61_pow(u, j + 1);
      hc.limb[b][0][j] = (uint32_t)(v & 0x1FFFFF);
      hc.limb[b][1][j] = (uint32_t)((v >> 21) & 0x1FFFFF);
      hc.limb[b][2][j] = (uint32_t)(v >> 42);
      hc.limb2[b][0][j] = (uint32_t)(v & 0x7FFFFFFF);
      hc.limb2[b][1][j] = (uint32_t)(v >> 31);
      sum = p61_add(sum, v);
      hc.csum[b][j + 1] = sum;
    }
    for (int q = 0; q < 32; ++q) hc.sub_mul[b][q] = p61_pow(u, 16ULL * q);
  }
  PTC_KERNEL("k_pow_tables", s, k_pow_tables, (4 * 8192) / 256, 256, 0, pb, L.tables, L.st);

  HashArgs a;
  a.tokens = tokens;
  a.n_tok = n_tok;
  a.tok_off = req_tok_off;
  a.blk_off = req_blk_off_out;
  a.R = n_req;
  a.B = block_size;
  a.keys = reinterpret_cast<ulonglong2*>(keys_out);
  a.keys_cap = keys_cap;
  a.tables = L.tables;
  a.tile_req = L.tile_req;
  a.tile_agg = L.tile_agg;
  a.tile_lead = L.tile_lead;
  a.wide_list = L.wide_list;
  a.st = L.st;
  a.aligned = aligned;
  const bool full = block_size == 16 * G;
  const uint64_t nb = n_tok / block_size < keys_cap ? n_tok / block_size : keys_cap;
  const uint32_t grid = ceil_div_u32(nb, tb);
  if (grid > 0) {
    switch (G) {
      case 1: launch_hash<1>(grid, s, a, hc, full); break;
      case 2: launch_hash<2>(grid, s, a, hc, full); break;
      case 4: launch_hash<4>(grid, s, a, hc, full); break;
      case 8: launch_hash<8>(grid, s, a, hc, full); break;
      case 16: launch_hash<16>(grid, s, a, hc, full); break;
      default: launch_hash<32>(grid, s, a, hc, full); break;
    }
    if (carry) {
      PTC_KERNEL("k_hash_carry", s, k_hash_carry, ceil_div_u32(grid, kChainWarps * kCarryPer), kChainWarps * 32, 0, L.tile_agg,
                 L.tile_lead, tb, L.st, keys_cap, grid, carry->carry, carry->lead);
      carry->tile_blocks = tb;
    } else {
      PTC_KERNEL("k_hash_chain", s, k_hash_chain, ceil_div_u32(grid, kChainWarps), kChainWarps * 32, 0, a.keys,
                 L.tile_agg, L.tile_lead, tb, L.st, keys_cap);
    }
  }
  if (deferred) return defer_status(L.st, err_slot, s, n_slot, 0);
  DevStatus h;
  ptc_status rc = end_call(L.st, s, &h);
  *n_access_host_out = h.value[0];
  if (rc != PTC_OK) return rc;
  if (h.value[0] > keys_cap) return PTC_ERR_INVALID_ARG;
  return PTC_OK;
}

extern "C" ptc_status ptc_hash_blocks(const uint32_t* tokens, uint64_t n_tok, const uint64_t* req_tok_off,
                                      const int64_t* req_ts_us, uint32_t n_req, uint32_t block_size, uint64_t seed,
                                      ptc_u128* keys_out, uint64_t keys_cap, uint64_t* req_blk_off_out,
                                      uint64_t* n_access_host_out, void* ws, size_t ws_bytes, void* stream) {
  return ptc::hash_impl(tokens, n_tok, req_tok_off, req_ts_us, n_req, block_size, seed, keys_out, keys_cap,
                        req_blk_off_out, n_access_host_out, ws, ws_bytes, (cudaStream_t)stream, nullptr, nullptr);
}
