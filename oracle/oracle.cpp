// CPU ORACLE — test infrastructure only.
//
// A plain, slow, obviously correct restatement of what the GPU path computes:
// block-level LRU prefix-cache hit curves and compute-saved curves over a
// request trace.  Only the tests, the package's smoke check and the bench's
// CPU-baseline leg may load this library.  It shares no code, header, table or
// constant generator with the CUDA path.
//
// Definitions followed (paper: "When Fancy Eviction Fails: Rethinking Cache
// Replacement For LLM Prefix Reuse"):
//   * Sec. 2.2: KV state is cached in fixed-size token blocks (16 tokens), and
//     a cached block is reusable iff its whole preceding sequence matches.
//     -> orc_block_ids: a trie keyed by (parent block id, the block's tokens),
//        compared token by token (no hashing decides identity).
//   * Sec. 3.1-3.2: block hit ratio of an LRU cache of C blocks replaying the
//     trace.  -> orc_lru_curves: one direct hashmap + recency-list LRU per
//        capacity; a block counts as a prefix hit only if it and every earlier
//        block of its request are resident (prefix reuse, Sec. 2.2).
//   * Sec. 5.2: compute-savings ratio = cost of hits / cost of all accesses,
//     with a per-block recompute cost that grows with depth.  -> cost_of().
//   * Appendix B: the stack distance between reuses ("reuses reachable within
//     C").  -> orc_sd_mattson (move-to-front list, Mattson et al. 1970) and
//        orc_sd_fenwick (Bennett & Kruskal 1975 counting), two independent ways.
//   * Belady's next use (Sec. 3.2, 5.2).  -> orc_reuse: previous and next
//     access of the same block.
//   * Sec. 5.3: session-level instead of block-level eviction.
//     -> orc_session_lru_curves: one direct simulation per capacity that evicts
//        the least recently touched session's blocks together.
//   * Sec. 3.2: Belady's optimum as the offline ceiling.  -> orc_belady_curves:
//     one direct MIN simulation (evict the farthest next access) per capacity,
//     with the same prefix rule as the LRU curves.
//   * Sec. 3.1 (the paper's simulator keeps a whole request resident and
//     makes room for it up front) and the order a request's blocks are
//     touched in.  -> orc_lru_curves_variant (direct LRU per capacity),
//        orc_sd_variant (Fenwick counting) and orc_sd_variant_mattson
//        (move-to-front list).
//   * Sec. 4.1-4.3 and App. B: block lifetimes, frequencies, reuse intervals,
//     block categories, session lengths and reuses reachable within a
//     capacity.  -> orc_trace_stats: two passes over the access stream with
//        per-block arrays, then loops over blocks and sessions.
// The GPU path's block keys are polynomial hashes of each block's whole
// prefix, sum over its tokens of (tok_t + 1) u^(t+1) mod 2^61 - 1 at two
// seeded bases u; orc_prefix_hash evaluates that sum token by token so the
// keys themselves can be compared.
//
// Readings where the paper is silent (listed with the design notes): requests
// are replayed in trace order and blocks root-first; a trailing partial block is
// not cached; ids are numbered by first occurrence; stack distances are 1-based
// with "never seen" = 0xFFFFFFFF; costs are summed in unsigned 128-bit integers.
#include <algorithm>
#include <atomic>
#include <cstdint>
#include <cstring>
#include <iterator>
#include <list>
#include <set>
#include <thread>
#include <unordered_map>
#include <vector>

typedef unsigned __int128 u128;
static const uint32_t NONE = 0xFFFFFFFFu;

// ---------------------------------------------------------------------------
// Exact block identity (Sec. 2.2).
// ---------------------------------------------------------------------------
namespace {
struct BlockKey {
  uint32_t parent;   // id of the previous block of the request, or NONE for the first block
  uint64_t tok_off;  // offset of the block's first token in the token array
};
struct BlockHash {
  const uint32_t* tok;
  uint32_t B;
  size_t operator()(const BlockKey& k) const {
    // FNV-1a over the parent id and the B token values (used only to bucket;
    // equality below compares the tokens themselves).
    uint64_t h = 1469598103934665603ULL;
    auto mix = [&](uint32_t v) {
      for (int b = 0; b < 4; ++b) { h ^= (v >> (8 * b)) & 0xFF; h *= 1099511628211ULL; }
    };
    mix(k.parent);
    for (uint32_t t = 0; t < B; ++t) mix(tok[k.tok_off + t]);
    return (size_t)h;
  }
};
struct BlockEq {
  const uint32_t* tok;
  uint32_t B;
  bool operator()(const BlockKey& a, const BlockKey& b) const {
    if (a.parent != b.parent) return false;
    for (uint32_t t = 0; t < B; ++t)
      if (tok[a.tok_off + t] != tok[b.tok_off + t]) return false;
    return true;
  }
};
}  // namespace

extern "C" {

// Number of full blocks of each request and their offsets in the access
// stream: req_blk_off[r] = sum over earlier requests of floor(len / B).
// Returns the total N.
uint64_t orc_block_offsets(const uint64_t* req_tok_off, uint32_t n_req, uint32_t B, uint64_t* req_blk_off) {
  req_blk_off[0] = 0;
  for (uint32_t r = 0; r < n_req; ++r) {
    uint64_t len = req_tok_off[r + 1] - req_tok_off[r];
    req_blk_off[r + 1] = req_blk_off[r] + len / B;  // a trailing partial block is not a cache object
  }
  return req_blk_off[n_req];
}

// Dense block ids in first-occurrence order of the access stream (requests in
// trace order, blocks root-first).  Two blocks get the same id iff their whole
// prefixes [0, B(k+1)) are equal token by token: by induction over k, since a
// block's trie key is (id of its parent, its own B tokens).
// ids must hold N entries (N from orc_block_offsets).  Returns D.
uint64_t orc_block_ids(const uint32_t* tokens, const uint64_t* req_tok_off, uint32_t n_req, uint32_t B,
                       uint32_t* ids) {
  BlockHash hasher{tokens, B};
  BlockEq eq{tokens, B};
  std::unordered_map<BlockKey, uint32_t, BlockHash, BlockEq> trie(16, hasher, eq);
  uint32_t next_id = 0;
  uint64_t i = 0;
  for (uint32_t r = 0; r < n_req; ++r) {
    uint64_t len = req_tok_off[r + 1] - req_tok_off[r];
    uint64_t nblk = len / B;
    uint32_t parent = NONE;
    for (uint64_t k = 0; k < nblk; ++k) {
      BlockKey key{parent, req_tok_off[r] + k * B};
      auto it = trie.find(key);
      uint32_t id;
      if (it == trie.end()) {
        id = next_id++;
        trie.emplace(key, id);
      } else {
        id = it->second;
      }
      ids[i++] = id;
      parent = id;
    }
  }
  return next_id;
}

// prev[i] = largest j < i with ids[j] == ids[i], else NONE;
// next[i] = smallest j > i with ids[j] == ids[i], else NONE (Belady's next use).
void orc_reuse(const uint32_t* ids, uint64_t n, uint64_t n_distinct, uint32_t* prev, uint32_t* next) {
  std::vector<uint32_t> last(n_distinct, NONE);
  for (uint64_t i = 0; i < n; ++i) {
    prev[i] = last[ids[i]];
    last[ids[i]] = (uint32_t)i;
  }
  std::fill(last.begin(), last.end(), NONE);
  for (uint64_t i = n; i-- > 0;) {
    next[i] = last[ids[i]];
    last[ids[i]] = (uint32_t)i;
  }
}

// LRU stack distance by Mattson's stack: keep blocks in recency order (most
// recent first); an access at depth d (1-based) has distance d, a block never
// seen has distance NONE, and the block moves to the top.  O(N * D): tiny
// inputs only.
void orc_sd_mattson(const uint32_t* ids, uint64_t n, uint32_t* sd) {
  std::vector<uint32_t> stack;  // stack[0] is the most recent
  for (uint64_t i = 0; i < n; ++i) {
    uint32_t x = ids[i];
    size_t pos = 0;
    while (pos < stack.size() && stack[pos] != x) ++pos;
    if (pos == stack.size()) {
      sd[i] = NONE;
      stack.insert(stack.begin(), x);
    } else {
      sd[i] = (uint32_t)(pos + 1);
      stack.erase(stack.begin() + pos);
      stack.insert(stack.begin(), x);
    }
  }
}

// LRU stack distance by counting (Bennett & Kruskal): mark, for every block,
// the position of its latest access so far; the distance of access i with
// previous access p is 1 + (number of marked positions strictly between p and
// i), i.e. 1 + the number of distinct blocks touched since p.  A Fenwick tree
// over positions holds the marks.
void orc_sd_fenwick(const uint32_t* prev, uint64_t n, uint32_t* sd) {
  std::vector<uint32_t> tree(n + 1, 0);
  auto add = [&](uint64_t pos, int32_t v) {
    for (uint64_t x = pos + 1; x <= n; x += x & (~x + 1)) tree[x] += (uint32_t)v;
  };
  auto prefix = [&](uint64_t cnt) {  // marks in positions [0, cnt)
    uint64_t s = 0;
    for (uint64_t x = cnt; x > 0; x -= x & (~x + 1)) s += tree[x];
    return s;
  };
  for (uint64_t i = 0; i < n; ++i) {
    uint32_t p = prev[i];
    if (p == NONE) {
      sd[i] = NONE;
    } else {
      uint64_t between = prefix(i) - prefix((uint64_t)p + 1);
      sd[i] = (uint32_t)(1 + between);
      add(p, -1);
    }
    add(i, +1);
  }
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Recompute cost of block k (0-based depth) of a request (Sec. 5.2, App. C).
//   kind 0 (uniform): every block costs 1, so compute saved = hits.
//   kind 1 (measured-shape): B*f_lin for the position-independent work plus
//           f_attn * (t+1) for each token t of the block (token t attends to
//           t+1 positions), t = Bk .. Bk+B-1.
//   kind 2 (linear): the attention term alone, proportional to depth.
// ---------------------------------------------------------------------------
static u128 cost_of(uint64_t k, uint32_t B, int kind, uint64_t f_lin, uint64_t f_attn) {
  if (kind == 0) return 1;
  u128 c = 0;
  if (kind == 1) c += (u128)B * f_lin;
  for (uint64_t t = (uint64_t)B * k; t < (uint64_t)B * k + B; ++t) c += (u128)f_attn * (t + 1);
  return c;
}

extern "C" {

// Direct LRU simulation, one capacity at a time (Sec. 3.1-3.2 with prefix
// reuse from Sec. 2.2).  For capacity C: replay requests in trace order and
// their blocks root-first; a resident block moves to the most-recent end, a
// missing block is inserted there and, if the cache then holds more than C
// blocks, the least recent one is evicted.  Block k of a request is a hit iff
// blocks 0..k of that request were all resident when touched.
//
// caps[G] are capacities in blocks (>= 1).  Outputs per capacity: hits[g] and
// the 128-bit compute saved as saved_lo[g] / saved_hi[g].  total_cost gets the
// 128-bit cost of every access.  Capacities are spread over `threads` host
// threads.  Returns 0, or -1 on a bad argument.
int orc_lru_curves(const uint32_t* ids, const uint64_t* req_blk_off, uint32_t n_req, uint32_t B, int kind,
                   uint64_t f_lin, uint64_t f_attn, const uint64_t* caps, uint32_t G, int threads, uint64_t* hits,
                   uint64_t* saved_lo, uint64_t* saved_hi, uint64_t* total_lo, uint64_t* total_hi) {
  for (uint32_t g = 0; g < G; ++g)
    if (caps[g] == 0) return -1;
  u128 total = 0;
  for (uint32_t r = 0; r < n_req; ++r)
    for (uint64_t k = 0; k < req_blk_off[r + 1] - req_blk_off[r]; ++k) total += cost_of(k, B, kind, f_lin, f_attn);
  *total_lo = (uint64_t)total;
  *total_hi = (uint64_t)(total >> 64);

  std::atomic<uint32_t> next_cap{0};
  auto simulate = [&]() {
    for (;;) {
      uint32_t g = next_cap.fetch_add(1);
      if (g >= G) return;
      uint64_t C = caps[g];
      std::list<uint32_t> recency;  // front = most recent
      std::unordered_map<uint32_t, std::list<uint32_t>::iterator> where;
      uint64_t h = 0;
      u128 saved = 0;
      for (uint32_t r = 0; r < n_req; ++r) {
        bool prefix_ok = true;
        for (uint64_t k = 0; k < req_blk_off[r + 1] - req_blk_off[r]; ++k) {
          uint32_t id = ids[req_blk_off[r] + k];
          auto it = where.find(id);
          bool resident = it != where.end();
          if (resident) {
            recency.splice(recency.begin(), recency, it->second);
          } else {
            recency.push_front(id);
            where[id] = recency.begin();
            if (recency.size() > C) {
              where.erase(recency.back());
              recency.pop_back();
            }
          }
          prefix_ok = prefix_ok && resident;
          if (prefix_ok) {
            ++h;
            saved += cost_of(k, B, kind, f_lin, f_attn);
          }
        }
      }
      hits[g] = h;
      saved_lo[g] = (uint64_t)saved;
      saved_hi[g] = (uint64_t)(saved >> 64);
    }
  };
  if (threads < 1) threads = 1;
  std::vector<std::thread> pool;
  for (int t = 1; t < threads; ++t) pool.emplace_back(simulate);
  simulate();
  for (auto& th : pool) th.join();
  return 0;
}

// Belady's offline optimum (Belady 1966), the paper's offline ceiling
// (Sec. 3.2, and the headroom in App. A-B), simulated directly, one capacity
// at a time.  For capacity C: replay requests in trace order and their blocks
// root-first; a resident block stays (a hit); a missing block is brought in
// and, if the cache then holds more than C blocks, the resident block other
// than the one just brought in whose next access lies farthest in the future
// (never again counts as farthest) is evicted.  Every accessed block is
// admitted: the demand-paging MIN that Mattson et al. (1970) show to be a
// stack algorithm.  Block k of a request counts as a hit iff blocks 0..k of
// that request were all resident when touched (Sec. 2.2 prefix reuse), as in
// orc_lru_curves; raw_hits[g] counts every resident access, without the
// prefix rule.  Next accesses come from a backward pass over the ids.
// Outputs per capacity as orc_lru_curves.  Returns 0, or -1 on a capacity
// of 0.
int orc_belady_curves(const uint32_t* ids, const uint64_t* req_blk_off, uint32_t n_req, uint32_t B, int kind,
                      uint64_t f_lin, uint64_t f_attn, const uint64_t* caps, uint32_t G, int threads, uint64_t* hits,
                      uint64_t* saved_lo, uint64_t* saved_hi, uint64_t* raw_hits) {
  for (uint32_t g = 0; g < G; ++g)
    if (caps[g] == 0) return -1;
  const uint64_t n = req_blk_off[n_req];
  uint32_t D = 0;
  for (uint64_t i = 0; i < n; ++i)
    if (ids[i] + 1 > D) D = ids[i] + 1;
  std::vector<uint32_t> nxt(n, NONE), last(D, NONE);
  for (uint64_t i = n; i-- > 0;) {
    nxt[i] = last[ids[i]];
    last[ids[i]] = (uint32_t)i;
  }
  const uint64_t kNever = 1ULL << 63;  // "never again": beyond every access index, ties broken by id
  const uint64_t kOut = ~0ULL;         // not resident
  std::atomic<uint32_t> next_cap{0};
  auto simulate = [&]() {
    for (;;) {
      uint32_t g = next_cap.fetch_add(1);
      if (g >= G) return;
      uint64_t C = caps[g];
      std::set<std::pair<uint64_t, uint32_t>> by_next;  // resident blocks by (next access, id)
      std::vector<uint64_t> key(D, kOut);                // each resident block's next access
      uint64_t h = 0, raw = 0;
      u128 saved = 0;
      for (uint32_t r = 0; r < n_req; ++r) {
        bool prefix_ok = true;
        for (uint64_t k = 0; k < req_blk_off[r + 1] - req_blk_off[r]; ++k) {
          uint64_t i = req_blk_off[r] + k;
          uint32_t id = ids[i];
          uint64_t nu = nxt[i] == NONE ? kNever + id : nxt[i];
          bool resident = key[id] != kOut;
          if (resident) by_next.erase({key[id], id});
          by_next.insert({nu, id});
          key[id] = nu;
          if (!resident && by_next.size() > C) {
            auto victim = std::prev(by_next.end());
            if (victim->second == id) victim = std::prev(victim);  // the block just brought in stays
            key[victim->second] = kOut;
            by_next.erase(victim);
          }
          raw += resident;
          prefix_ok = prefix_ok && resident;
          if (prefix_ok) {
            ++h;
            saved += cost_of(k, B, kind, f_lin, f_attn);
          }
        }
      }
      hits[g] = h;
      raw_hits[g] = raw;
      saved_lo[g] = (uint64_t)saved;
      saved_hi[g] = (uint64_t)(saved >> 64);
    }
  };
  if (threads < 1) threads = 1;
  std::vector<std::thread> pool;
  for (int t = 1; t < threads; ++t) pool.emplace_back(simulate);
  simulate();
  for (auto& th : pool) th.join();
  return 0;
}

// Session-level LRU eviction (Sec. 5.3: evicting whole sessions instead of
// blocks), one capacity at a time.  Readings (the paper gives no rules):
//   * a block brought in by a request belongs to that request's session until
//     it is evicted, even when other sessions hit it later (so evicting a
//     session also drops the shared prompts it brought in, as Sec. 5.3 notes);
//   * sessions are ordered by the arrival of their latest request; a session
//     is touched when its request arrives, before its blocks;
//   * a miss brings the block in; while more than C blocks are resident, all
//     blocks of the least recently touched session other than the current
//     one are evicted;
//   * if the current session is then the only one holding blocks and the
//     cache still holds more than C, all its blocks except the one just
//     brought in are evicted (a session larger than the cache restarts).
// Block k of a request counts as a hit iff blocks 0..k of that request were
// all resident (Sec. 2.2 prefix reuse); costs as in orc_lru_curves.
// req_session[r] < n_session.  Returns 0, or -1 on a bad argument.
int orc_session_lru_curves(const uint32_t* ids, const uint64_t* req_blk_off, const uint32_t* req_session,
                           uint32_t n_req, uint32_t n_session, uint32_t B, int kind, uint64_t f_lin, uint64_t f_attn,
                           const uint64_t* caps, uint32_t G, int threads, uint64_t* hits, uint64_t* saved_lo,
                           uint64_t* saved_hi) {
  for (uint32_t g = 0; g < G; ++g)
    if (caps[g] == 0) return -1;
  for (uint32_t r = 0; r < n_req; ++r)
    if (req_session[r] >= n_session) return -1;
  std::atomic<uint32_t> next_cap{0};
  auto simulate = [&]() {
    for (;;) {
      uint32_t g = next_cap.fetch_add(1);
      if (g >= G) return;
      uint64_t C = caps[g];
      std::unordered_map<uint32_t, uint32_t> owner;     // resident block -> its session
      std::vector<std::vector<uint32_t>> owned(n_session);  // each session's resident blocks
      std::list<uint32_t> order;                        // sessions, most recently touched first
      std::vector<std::list<uint32_t>::iterator> pos(n_session, order.end());
      uint64_t total = 0, h = 0;
      u128 saved = 0;
      for (uint32_t r = 0; r < n_req; ++r) {
        uint32_t s = req_session[r];
        if (pos[s] != order.end()) order.erase(pos[s]);
        order.push_front(s);
        pos[s] = order.begin();
        bool prefix_ok = true;
        for (uint64_t k = 0; k < req_blk_off[r + 1] - req_blk_off[r]; ++k) {
          uint32_t id = ids[req_blk_off[r] + k];
          bool resident = owner.count(id) != 0;
          if (!resident) {
            owner[id] = s;
            owned[s].push_back(id);
            ++total;
            while (total > C) {
              uint32_t victim = s;
              for (auto it = order.rbegin(); it != order.rend(); ++it)
                if (*it != s && !owned[*it].empty()) {
                  victim = *it;
                  break;
                }
              if (victim != s) {
                for (uint32_t b : owned[victim]) owner.erase(b);
                total -= owned[victim].size();
                owned[victim].clear();
              } else {  // only the current session holds blocks
                for (uint32_t b : owned[s])
                  if (b != id) owner.erase(b);
                total = 1;
                owned[s].assign(1, id);
              }
            }
          }
          prefix_ok = prefix_ok && resident;
          if (prefix_ok) {
            ++h;
            saved += cost_of(k, B, kind, f_lin, f_attn);
          }
        }
      }
      hits[g] = h;
      saved_lo[g] = (uint64_t)saved;
      saved_hi[g] = (uint64_t)(saved >> 64);
    }
  };
  if (threads < 1) threads = 1;
  std::vector<std::thread> pool;
  for (int t = 1; t < threads; ++t) pool.emplace_back(simulate);
  simulate();
  for (auto& th : pool) th.join();
  return 0;
}

// Curves from stack distances by Mattson inclusion (Mattson et al. 1970;
// App. B "reuses reachable within C"): LRU is a stack algorithm, so the
// access with stack distance sd is resident in every cache of at least sd
// blocks.  With the prefix rule of Sec. 2.2, block k of a request counts at
// capacity C iff the distances of blocks 0..k of that request are all at most
// C, i.e. iff e_k = max(sd_0, .., sd_k) <= C (sd = NONE never counts).  For
// each capacity: hits[g] = #{accesses with e <= caps[g]} and saved[g] = the
// 128-bit sum of their costs.  The same outputs as orc_lru_curves, reached
// through the distances instead of a cache simulation.  caps must be strictly
// ascending.  Returns 0, or -1 on a capacity of 0 or an unsorted grid.
int orc_curves_from_dist(const uint32_t* sd, const uint64_t* req_blk_off, uint32_t n_req, uint32_t B, int kind,
                         uint64_t f_lin, uint64_t f_attn, const uint64_t* caps, uint32_t G, uint64_t* hits,
                         uint64_t* saved_lo, uint64_t* saved_hi) {
  for (uint32_t g = 0; g < G; ++g)
    if (caps[g] == 0) return -1;
  for (uint32_t g = 1; g < G; ++g)
    if (caps[g] <= caps[g - 1]) return -1;
  // An access with running maximum e counts at every capacity from the
  // first grid point >= e on: add it to that point, then sum over the grid.
  std::vector<uint64_t> h(G, 0);
  std::vector<u128> saved(G, 0);
  for (uint32_t r = 0; r < n_req; ++r) {
    uint64_t e = 0;  // running maximum of the distances, NONE as 2^32 - 1
    for (uint64_t k = 0; k < req_blk_off[r + 1] - req_blk_off[r]; ++k) {
      uint32_t d = sd[req_blk_off[r] + k];
      if (d > e) e = d;
      if (e == NONE) continue;  // a cold block, or a deeper block of a request with one
      uint32_t g = (uint32_t)(std::lower_bound(caps, caps + G, e) - caps);
      if (g == G) continue;  // beyond the largest capacity
      ++h[g];
      saved[g] += cost_of(k, B, kind, f_lin, f_attn);
    }
  }
  uint64_t hs = 0;
  u128 ss = 0;
  for (uint32_t g = 0; g < G; ++g) {
    hs += h[g];
    ss += saved[g];
    hits[g] = hs;
    saved_lo[g] = (uint64_t)ss;
    saved_hi[g] = (uint64_t)(ss >> 64);
  }
  return 0;
}

// Polynomial prefix hash over GF(p), p = 2^61 - 1, evaluated token by token:
// the prefix tok_0 .. tok_{m-1} of a request maps to
//     S(m) = sum_{t<m} (tok_t + 1) * u^(t+1)   (mod p).
// Every coefficient tok_t + 1 is at least 1, so a prefix and any longer
// prefix are different polynomials and no leading term is needed to keep
// lengths apart.  For each block k of each request the key is
// (S(B(k+1)) at u_0, S(B(k+1)) at u_1), written as keys[2i], keys[2i+1].
// The two bases come from `seed` by SplitMix64 (Steele, Lea, Flood 2014):
// u_b = 2 + (output b of the stream seeded `seed`) mod (p - 3).
void orc_prefix_hash(const uint32_t* tokens, const uint64_t* req_tok_off, uint32_t n_req, uint32_t B, uint64_t seed,
                     uint64_t* keys) {
  const uint64_t P = (1ULL << 61) - 1;
  uint64_t u[2];
  for (int b = 0; b < 2; ++b) {
    uint64_t z = seed + (uint64_t)(b + 1) * 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    z = z ^ (z >> 31);
    u[b] = 2 + z % (P - 3);
  }
  uint64_t i = 0;
  for (uint32_t r = 0; r < n_req; ++r) {
    uint64_t len = req_tok_off[r + 1] - req_tok_off[r];
    uint64_t nblk = len / B;
    u128 s0 = 0, s1 = 0, p0 = u[0], p1 = u[1];  // p_b = u_b^(t+1)
    for (uint64_t t = 0; t < nblk * B; ++t) {
      u128 x = (u128)tokens[req_tok_off[r] + t] + 1;
      s0 = (s0 + x * p0) % P;
      s1 = (s1 + x * p1) % P;
      p0 = p0 * u[0] % P;
      p1 = p1 * u[1] % P;
      if ((t + 1) % B == 0) {
        keys[2 * i] = (uint64_t)s0;
        keys[2 * i + 1] = (uint64_t)s1;
        ++i;
      }
    }
  }
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Trace characterization (Sec. 4.1-4.3; App. B).  Each access of block d in
// request r happens at the request's arrival time ts[r] and belongs to the
// request's session sess[r].  Per block d: its frequency (number of
// accesses), its lifetime (time of its last access minus time of its first,
// zero for a block used once), and its category.  Per reuse (every access but
// a block's first): the reuse interval, its time minus the time of the
// previous access of the same block.  Per session: its request count and its
// duration (last minus first request time).
//
// Categories (Sec. 4.1 names three, by message role, which a token trace does
// not carry; the reading used here classifies by the sessions a block appears
// in):
//   0  shared across sessions: the block appears in two or more sessions and
//      at least one of them has two or more requests (system prompts reused
//      across conversations);
//   1  session history: the block appears in exactly one session, and that
//      session has two or more requests;
//   2  single-turn: every session the block appears in has one request.
// Histograms bin a value x >= 0 by the bit length of x (0 for x = 0, else
// floor(log2 x) + 1), 65 bins.  freq[c][k] counts blocks used exactly k times
// for 1 <= k < 256, and freq[c][0] those used 256 times or more.
// reach[g] counts reuses whose LRU stack distance is at most cap[g] (App. B:
// reuses reachable within a cache of cap[g] blocks); dist may be NULL.
// Returns 0, or 1 for malformed input (an id >= D, a session label >=
// n_session, offsets that are not a partition of [0, n)), or 2 if the
// timestamps decrease.
// ---------------------------------------------------------------------------
namespace {
int bit_length(uint64_t x) {
  int b = 0;
  while (x != 0) {
    ++b;
    x >>= 1;
  }
  return b;
}
}  // namespace

extern "C" {

int orc_trace_stats(const uint32_t* ids, uint64_t n, uint64_t D, const uint64_t* req_blk_off, const int64_t* ts,
                    const uint64_t* sess, uint32_t n_req, uint64_t n_session, const uint32_t* dist,
                    const uint64_t* caps, uint32_t n_cap, uint64_t* blocks, uint64_t* accesses, uint64_t* freq,
                    uint64_t* freq_log2, uint64_t* reuse_us, uint64_t* lifetime_us, uint64_t* reuse_by_freq,
                    uint64_t* lifetime_by_freq, uint64_t* dist_log2, uint64_t* reach, uint64_t* sess_requests,
                    uint64_t* sess_duration_us, uint64_t* scalars) {
  // inputs
  if (req_blk_off[0] != 0 || req_blk_off[n_req] != n) return 1;
  for (uint32_t r = 0; r < n_req; ++r) {
    if (req_blk_off[r + 1] < req_blk_off[r] || sess[r] >= n_session) return 1;
    if (r > 0 && ts[r] < ts[r - 1]) return 2;
  }
  for (uint64_t i = 0; i < n; ++i)
    if (ids[i] >= D) return 1;

  // sessions: request count, first and last request time
  std::vector<uint64_t> s_req(n_session, 0);
  std::vector<int64_t> s_first(n_session, 0), s_last(n_session, 0);
  for (uint32_t r = 0; r < n_req; ++r) {
    uint64_t s = sess[r];
    if (s_req[s] == 0) s_first[s] = ts[r];
    s_last[s] = ts[r];
    ++s_req[s];
  }

  // first pass over the accesses in stream order: frequency, first and last
  // access time, the first session seen, and the two category conditions
  std::vector<uint64_t> cnt(D, 0);
  std::vector<int64_t> t_first(D, 0), t_last(D, 0);
  std::vector<uint64_t> first_sess(D, 0);
  std::vector<char> in_multi(D, 0), in_two(D, 0);
  for (uint32_t r = 0; r < n_req; ++r) {
    for (uint64_t i = req_blk_off[r]; i < req_blk_off[r + 1]; ++i) {
      uint32_t d = ids[i];
      if (cnt[d] == 0) {
        t_first[d] = ts[r];
        first_sess[d] = sess[r];
      } else if (first_sess[d] != sess[r]) {
        in_two[d] = 1;
      }
      t_last[d] = ts[r];
      if (s_req[sess[r]] >= 2) in_multi[d] = 1;
      ++cnt[d];
    }
  }
  auto category = [&](uint32_t d) { return in_multi[d] ? (in_two[d] ? 0 : 1) : 2; };

  // per block
  for (uint64_t d = 0; d < D; ++d) {
    if (cnt[d] == 0) return 1;  // ids must be dense
    int c = category((uint32_t)d);
    uint64_t life = (uint64_t)(t_last[d] - t_first[d]);
    blocks[c] += 1;
    accesses[c] += cnt[d];
    freq[c * 256 + (cnt[d] < 256 ? cnt[d] : 0)] += 1;
    freq_log2[c * 65 + bit_length(cnt[d])] += 1;
    lifetime_us[c * 65 + bit_length(life)] += 1;
    lifetime_by_freq[bit_length(cnt[d]) * 65 + bit_length(life)] += 1;
  }

  // second pass: reuse intervals, binned by the category and the frequency of
  // the block (both final after the first pass)
  std::vector<char> seen(D, 0);
  std::vector<int64_t> t_prev(D, 0);
  uint64_t n_reuse = 0;
  for (uint32_t r = 0; r < n_req; ++r) {
    for (uint64_t i = req_blk_off[r]; i < req_blk_off[r + 1]; ++i) {
      uint32_t d = ids[i];
      if (seen[d]) {
        uint64_t gap = (uint64_t)(ts[r] - t_prev[d]);
        reuse_us[category(d) * 65 + bit_length(gap)] += 1;
        reuse_by_freq[bit_length(cnt[d]) * 65 + bit_length(gap)] += 1;
        ++n_reuse;
      }
      seen[d] = 1;
      t_prev[d] = ts[r];
    }
  }

  // stack distances of the reuses
  if (dist != nullptr) {
    for (uint64_t i = 0; i < n; ++i) {
      if (dist[i] == NONE) continue;
      dist_log2[bit_length(dist[i])] += 1;
      for (uint32_t g = 0; g < n_cap; ++g)
        if (dist[i] <= caps[g]) reach[g] += 1;
    }
  }

  // per session
  uint64_t used = 0, multi = 0;
  for (uint64_t s = 0; s < n_session; ++s) {
    if (s_req[s] == 0) continue;
    ++used;
    if (s_req[s] >= 2) ++multi;
    sess_requests[bit_length(s_req[s])] += 1;
    sess_duration_us[bit_length((uint64_t)(s_last[s] - s_first[s]))] += 1;
  }
  scalars[0] = n;
  scalars[1] = D;
  scalars[2] = n_reuse;
  scalars[3] = used;
  scalars[4] = multi;
  return 0;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Semantics variants (Sec. 3.1: the paper's simulator makes room for a whole
// request before its prefill, so every block of a request is resident at
// once; engines differ in the order they touch a request's blocks).
//   order      0: root-first (depth 0, 1, ...), the hot path's order
//              1: leaf-first (deepest block first, the root last)
//   residency  0: per block: each block is looked up when it is touched
//              1: per request: every block of the request is looked up at the
//                 request's arrival, before any of them is touched; then all
//                 are touched in `order`
// A block counts as a hit iff it and every shallower block of its request
// were found resident (prefix reuse, Sec. 2.2).  (order 0, residency 0) is
// orc_lru_curves.
// ---------------------------------------------------------------------------
extern "C" {

// Direct LRU simulation per capacity under a variant; arguments and outputs
// as for orc_lru_curves (without the total cost).  Returns 0, or -1 on a bad
// argument.
int orc_lru_curves_variant(const uint32_t* ids, const uint64_t* req_blk_off, uint32_t n_req, uint32_t B, int kind,
                           uint64_t f_lin, uint64_t f_attn, const uint64_t* caps, uint32_t G, int order,
                           int residency, int threads, uint64_t* hits, uint64_t* saved_lo, uint64_t* saved_hi) {
  if ((order != 0 && order != 1) || (residency != 0 && residency != 1)) return -1;
  for (uint32_t g = 0; g < G; ++g)
    if (caps[g] == 0) return -1;
  std::atomic<uint32_t> next_cap{0};
  auto simulate = [&]() {
    for (;;) {
      uint32_t g = next_cap.fetch_add(1);
      if (g >= G) return;
      uint64_t C = caps[g];
      std::list<uint32_t> recency;  // front = most recent
      std::unordered_map<uint32_t, std::list<uint32_t>::iterator> where;
      auto touch = [&](uint32_t id) {
        auto it = where.find(id);
        if (it != where.end()) {
          recency.splice(recency.begin(), recency, it->second);
        } else {
          recency.push_front(id);
          where[id] = recency.begin();
          if (recency.size() > C) {
            where.erase(recency.back());
            recency.pop_back();
          }
        }
      };
      uint64_t h = 0;
      u128 saved = 0;
      std::vector<char> resident;
      for (uint32_t r = 0; r < n_req; ++r) {
        const uint64_t a = req_blk_off[r], n = req_blk_off[r + 1] - a;
        resident.assign(n, 0);
        if (residency == 1)
          for (uint64_t k = 0; k < n; ++k) resident[k] = where.count(ids[a + k]) != 0;
        for (uint64_t s = 0; s < n; ++s) {
          const uint64_t k = order == 0 ? s : n - 1 - s;  // the s-th block touched
          if (residency == 0) resident[k] = where.count(ids[a + k]) != 0;
          touch(ids[a + k]);
        }
        for (uint64_t k = 0; k < n && resident[k]; ++k) {
          ++h;
          saved += cost_of(k, B, kind, f_lin, f_attn);
        }
      }
      hits[g] = h;
      saved_lo[g] = (uint64_t)saved;
      saved_hi[g] = (uint64_t)(saved >> 64);
    }
  };
  if (threads < 1) threads = 1;
  std::vector<std::thread> pool;
  for (int t = 1; t < threads; ++t) pool.emplace_back(simulate);
  simulate();
  for (auto& th : pool) th.join();
  return 0;
}

// Stack distance under a variant: the block's depth in the LRU stack (1 =
// most recent) when it is looked up, i.e. 1 + the number of distinct blocks
// touched since its own last touch; 0xFFFFFFFF for a block never seen.  Per
// block it is looked up when touched, per request at the request's arrival.
// Written in depth order (index req_blk_off[r] + k).  Counting as in
// orc_sd_fenwick: positions are numbered in touch order, and a Fenwick tree
// marks the position of every block's latest touch.
int orc_sd_variant(const uint32_t* ids, uint64_t n_distinct, const uint64_t* req_blk_off, uint32_t n_req, int order,
                   int residency, uint32_t* sd) {
  if ((order != 0 && order != 1) || (residency != 0 && residency != 1)) return -1;
  const uint64_t n = req_blk_off[n_req];
  std::vector<uint32_t> tree(n + 1, 0);
  auto add = [&](uint64_t pos, int32_t v) {
    for (uint64_t x = pos + 1; x <= n; x += x & (~x + 1)) tree[x] += (uint32_t)v;
  };
  auto prefix = [&](uint64_t cnt) {  // marks in positions [0, cnt)
    uint64_t s = 0;
    for (uint64_t x = cnt; x > 0; x -= x & (~x + 1)) s += tree[x];
    return s;
  };
  std::vector<uint64_t> last(n_distinct, UINT64_MAX);
  auto depth = [&](uint32_t id, uint64_t now) -> uint32_t {
    if (last[id] == UINT64_MAX) return NONE;
    return (uint32_t)(1 + prefix(now) - prefix(last[id] + 1));
  };
  uint64_t t = 0;  // touches so far
  for (uint32_t r = 0; r < n_req; ++r) {
    const uint64_t a = req_blk_off[r], m = req_blk_off[r + 1] - a;
    if (residency == 1)
      for (uint64_t k = 0; k < m; ++k) sd[a + k] = depth(ids[a + k], t);
    for (uint64_t s = 0; s < m; ++s) {
      const uint64_t k = order == 0 ? s : m - 1 - s;
      const uint32_t id = ids[a + k];
      if (residency == 0) sd[a + k] = depth(id, t);
      if (last[id] != UINT64_MAX) add(last[id], -1);
      add(t, +1);
      last[id] = t++;
    }
  }
  return 0;
}

// The same distances by a move-to-front list (Mattson et al. 1970): O(N * D),
// tiny inputs only.
int orc_sd_variant_mattson(const uint32_t* ids, const uint64_t* req_blk_off, uint32_t n_req, int order,
                           int residency, uint32_t* sd) {
  if ((order != 0 && order != 1) || (residency != 0 && residency != 1)) return -1;
  std::vector<uint32_t> stack;  // stack[0] is the most recent
  auto find = [&](uint32_t id) -> uint32_t {
    for (size_t pos = 0; pos < stack.size(); ++pos)
      if (stack[pos] == id) return (uint32_t)(pos + 1);
    return NONE;
  };
  auto touch = [&](uint32_t id) {
    uint32_t d = find(id);
    if (d != NONE) stack.erase(stack.begin() + (d - 1));
    stack.insert(stack.begin(), id);
  };
  for (uint32_t r = 0; r < n_req; ++r) {
    const uint64_t a = req_blk_off[r], m = req_blk_off[r + 1] - a;
    if (residency == 1)
      for (uint64_t k = 0; k < m; ++k) sd[a + k] = find(ids[a + k]);
    for (uint64_t s = 0; s < m; ++s) {
      const uint64_t k = order == 0 ? s : m - 1 - s;
      if (residency == 0) sd[a + k] = find(ids[a + k]);
      touch(ids[a + k]);
    }
  }
  return 0;
}

}  // extern "C"
