// Seeded synthetic request traces shaped like the paper's prefix-cache workloads.
//
// This module only draws INPUTS: it holds none of the arithmetic of the method
// (no hashing of blocks, no identity, no stack distances, no curves).  Both the
// CPU oracle and the GPU path read the arrays it writes, so a trace is the same
// bytes for both sides.
//
// A trace is four arrays:
//   tokens      u32[T]     every request's full context, concatenated in trace order
//   req_tok_off u64[R+1]   request r owns tokens[req_tok_off[r] : req_tok_off[r+1]]
//   req_ts_us   i64[R]     arrival time in microseconds, non-decreasing
//   req_session u64[R]     session id (carried for reference; not used by the math)
//
// Determinism.  All randomness is SplitMix64 (Steele, Lea, Flood, OOPSLA 2014)
// read as a counter-based generator: output n of the stream keyed k is
// mix64(k + (n+1)*gamma).  The few real-valued draws (lognormal lengths,
// exponential and jittered gaps, Zipf choices) use log/exp/cos written below as
// plain series with only +,-,*,/ and sqrt, and this file is compiled with
// -ffp-contract=off, so x86-64 and aarch64 hosts produce the same trace.
//
// Workload shapes follow the paper's description of its traces: 16-token
// blocks (Sec. 3.1), sessions of append-only turns (Sec. 2.3), system prompts
// shared across sessions (Table "trace-compare", global scope), short steady
// intra-session gaps (Sec. 4.2), heavy-tailed agentic session footprints
// (Sec. 4.5) and a 131,072-token context cap with oldest-turn truncation for
// the agentic generator.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <thread>
#include <vector>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ULL;
constexpr uint32_t kVocab = 151936;  // Qwen3 tokenizer vocabulary size
constexpr double kPi = 3.14159265358979323846;
constexpr double kLn2 = 0.693147180559945309417232121458;

inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}
// Output n (n >= 0) of the SplitMix64 stream keyed k.
inline uint64_t sm64_at(uint64_t k, uint64_t n) { return mix64(k + (n + 1) * kGamma); }
// Key of a sub-stream labelled `label` under stream key k.
inline uint64_t derive(uint64_t k, uint64_t label) { return mix64(k ^ mix64(label * kGamma + 0x632BE59BD9B4E019ULL)); }

// Token `pos` of the segment keyed `key`: Lemire's multiply-shift maps the
// 64-bit output uniformly onto [0, vocab).
inline uint32_t seg_token(uint64_t key, uint64_t pos) {
  return (uint32_t)(((unsigned __int128)sm64_at(key, pos) * kVocab) >> 64);
}

// ---- deterministic real functions (series; no libm transcendental calls) ----
double det_log(double x) {  // natural log, x > 0 finite
  int e = 0;
  double m = std::frexp(x, &e);  // exact: x = m * 2^e, m in [0.5, 1)
  if (m < 0.70710678118654752440) { m *= 2.0; e -= 1; }
  // log m = 2 atanh(s), s = (m-1)/(m+1), |s| < 0.1716
  double s = (m - 1.0) / (m + 1.0), s2 = s * s, term = s, sum = 0.0;
  for (int k = 1; k <= 41; k += 2) { sum += term / (double)k; term *= s2; }
  return 2.0 * sum + (double)e * kLn2;
}
double det_exp(double x) {  // |x| < 700
  double kf = std::floor(x / kLn2 + 0.5);
  double r = x - kf * kLn2;  // |r| <= ~0.35
  double p = 1.0;
  for (int n = 27; n >= 1; --n) p = 1.0 + r * p / (double)n;
  return std::ldexp(p, (int)kf);
}
double det_cos(double x) {
  double twopi = 2.0 * kPi;
  double y = x - twopi * std::floor(x / twopi);  // [0, 2pi)
  y -= kPi;                                       // cos(x) = -cos(y), y in [-pi, pi)
  double y2 = y * y, p = 1.0;
  for (int n = 22; n >= 1; --n) p = 1.0 - y2 * p / (double)((2 * n - 1) * (2 * n));
  return -p;
}

struct Rng {  // one structural draw stream
  uint64_t key, n = 0;
  explicit Rng(uint64_t k) : key(k) {}
  uint64_t u64() { return sm64_at(key, n++); }
  double u01() { return (double)(u64() >> 11) * 0x1.0p-53; }               // [0, 1)
  double u01_open0() { return (double)((u64() >> 11) + 1) * 0x1.0p-53; }  // (0, 1]
  double normal() {
    double u1 = u01_open0(), u2 = u01();
    return std::sqrt(-2.0 * det_log(u1)) * det_cos(2.0 * kPi * u2);
  }
  uint32_t lognormal_len(double median, double sigma) {
    double v = median * det_exp(sigma * normal());
    if (v < 1.0) v = 1.0;
    if (v > 4.0e6) v = 4.0e6;
    return (uint32_t)(v + 0.5);
  }
  double expo(double rate) { return -det_log(u01_open0()) / rate; }
  uint32_t geometric0(double mean) {  // support {0,1,...}
    if (mean <= 0) return 0;
    double q = mean / (1.0 + mean);  // failure probability
    double k = std::floor(det_log(u01_open0()) / det_log(q));
    return k > 1.0e6 ? 1000000u : (uint32_t)k;
  }
  uint32_t uniform_int(uint32_t lo, uint32_t hi) {  // inclusive
    return lo + (uint32_t)(((unsigned __int128)u64() * (uint64_t)(hi - lo + 1)) >> 64);
  }
};

struct Zipf {  // P(k) proportional to k^-s on k = 1..n
  std::vector<double> cdf;
  Zipf(uint32_t n, double s) {
    cdf.resize(n);
    double acc = 0.0;
    for (uint32_t k = 1; k <= n; ++k) { acc += det_exp(-s * det_log((double)k)); cdf[k - 1] = acc; }
  }
  uint32_t draw(Rng& r) const {  // 1-based
    double u = r.u01() * cdf.back();
    return (uint32_t)(std::upper_bound(cdf.begin(), cdf.end(), u) - cdf.begin()) + 1;
  }
};

struct Seg { uint64_t key; uint32_t len; };
struct Req {
  int64_t ts_us;
  uint64_t session;
  uint32_t turn;
  uint32_t seg_begin, seg_count;
  uint64_t ntok;
};

struct Trace {
  std::vector<Seg> segs;  // flattened per-request segment lists
  std::vector<Req> reqs;
  std::vector<uint32_t> order;  // trace order of reqs
  uint64_t n_tok = 0;
  uint64_t n_sessions = 0;
};

struct SysPool {  // shared system prompts (global block scope across sessions)
  std::vector<Seg> prompts;
  bool zipf = false;
  Zipf z{1, 1.0};
  SysPool(uint64_t key, uint32_t count, uint32_t lo, uint32_t hi, double zipf_s) : z(count, zipf_s > 0 ? zipf_s : 1.0) {
    Rng r(derive(key, 1));
    zipf = zipf_s > 0;
    for (uint32_t i = 0; i < count; ++i) prompts.push_back({derive(key, 1000 + i), r.uniform_int(lo, hi)});
  }
  Seg pick(Rng& r) const {
    uint32_t idx = zipf ? z.draw(r) - 1 : r.uniform_int(0, (uint32_t)prompts.size() - 1);
    return prompts[idx];
  }
};

// Conversational generator: a single-turn share, multi-turn sessions with
// 2 + Geometric turns, each turn appends a user message and a modelled reply.
struct ConvParams {
  uint64_t n_sessions;
  double window_s;            // session starts are Poisson over [0, window)
  bool diurnal;               // 24 h sinusoidal rate, peak/trough 3x (thinning)
  double single_frac;
  double extra_turns_mean;    // multi-turn sessions: turns = 2 + Geom0(mean)
  int gap_kind;               // 0: uniform mean*(1 +- jitter); 1: lognormal(median, sigma)
  double gap_a, gap_b;
  uint32_t sys_count, sys_lo, sys_hi;
  double sys_zipf;            // 0: uniform choice
  double user_med, reply_med, sigma;
};

// Agentic generator: Zipf turn counts (heavy-tailed footprints), each turn
// appends tool output and a reply, contexts capped by dropping oldest turns.
struct AgentParams {
  uint64_t n_sessions;
  double window_s;
  bool diurnal;
  double zipf_s;
  uint32_t max_turns;
  double tool_med, reply_med, sigma;
  uint64_t cap_tokens;
  double gap_lo, gap_hi;
  uint32_t sys_count, sys_lo, sys_hi;
};

double session_start(Rng& r, double window_s, bool diurnal, double& clock, double rate) {
  // Poisson arrivals at `rate`; with `diurnal`, thinned by 1 + 0.5 sin(2 pi t / 24h).
  for (;;) {
    clock += r.expo(diurnal ? rate * 1.5 : rate);
    if (!diurnal) return clock;
    double lam = 1.0 + 0.5 * det_cos(2.0 * kPi * clock / 86400.0 - kPi / 2.0);
    if (r.u01() * 1.5 < lam) return clock;
  }
  (void)window_s;
}

void push_request(Trace& tr, int64_t ts, uint64_t session, uint32_t turn, const std::vector<Seg>& ctx) {
  Req q;
  q.ts_us = ts;
  q.session = session;
  q.turn = turn;
  q.seg_begin = (uint32_t)tr.segs.size();
  q.seg_count = (uint32_t)ctx.size();
  q.ntok = 0;
  for (const Seg& s : ctx) { tr.segs.push_back(s); q.ntok += s.len; }
  tr.reqs.push_back(q);
}

void gen_conv(Trace& tr, const ConvParams& P, uint64_t key, uint64_t session_base) {
  SysPool pool(derive(key, 7), P.sys_count, P.sys_lo, P.sys_hi, P.sys_zipf);
  Rng arrivals(derive(key, 11));
  double clock = 0.0, rate = (double)P.n_sessions / P.window_s;
  std::vector<Seg> ctx;
  for (uint64_t s = 0; s < P.n_sessions; ++s) {
    double start = session_start(arrivals, P.window_s, P.diurnal, clock, rate);
    uint64_t sid = session_base + s;
    uint64_t skey = derive(key, 0x5E55000000ULL + s);
    Rng r(derive(skey, 1));
    bool single = r.u01() < P.single_frac;
    uint32_t turns = single ? 1u : 2u + r.geometric0(P.extra_turns_mean);
    ctx.clear();
    ctx.push_back(pool.pick(r));
    double t = start;
    for (uint32_t j = 0; j < turns; ++j) {
      if (j > 0) {
        double gap = P.gap_kind == 0 ? P.gap_a * (1.0 + P.gap_b * (2.0 * r.u01() - 1.0))
                                     : P.gap_a * det_exp(P.gap_b * r.normal());
        t += gap;
      }
      ctx.push_back({derive(skey, 100 + 2 * (uint64_t)j), r.lognormal_len(P.user_med, P.sigma)});
      ctx.push_back({derive(skey, 101 + 2 * (uint64_t)j), r.lognormal_len(P.reply_med, P.sigma)});
      push_request(tr, (int64_t)(t * 1e6), sid, j, ctx);
    }
  }
  tr.n_sessions += P.n_sessions;
}

void gen_agent(Trace& tr, const AgentParams& P, uint64_t key, uint64_t session_base) {
  SysPool pool(derive(key, 7), P.sys_count, P.sys_lo, P.sys_hi, 0.0);
  Zipf zt(P.max_turns, P.zipf_s);
  Rng arrivals(derive(key, 11));
  double clock = 0.0, rate = (double)P.n_sessions / P.window_s;
  std::vector<Seg> turns_kept;  // non-system segments currently in context
  std::vector<Seg> ctx;
  for (uint64_t s = 0; s < P.n_sessions; ++s) {
    double start = session_start(arrivals, P.window_s, P.diurnal, clock, rate);
    uint64_t sid = session_base + s;
    uint64_t skey = derive(key, 0xA6E0000000ULL + s);
    Rng r(derive(skey, 1));
    uint32_t turns = zt.draw(r);
    Seg sys = pool.pick(r);
    turns_kept.clear();
    uint64_t body = 0;  // tokens in turns_kept
    double t = start;
    for (uint32_t j = 0; j < turns; ++j) {
      if (j > 0) t += P.gap_lo + (P.gap_hi - P.gap_lo) * r.u01();
      Seg tool{derive(skey, 100 + 2 * (uint64_t)j), r.lognormal_len(P.tool_med, P.sigma)};
      Seg reply{derive(skey, 101 + 2 * (uint64_t)j), r.lognormal_len(P.reply_med, P.sigma)};
      turns_kept.push_back(tool);
      turns_kept.push_back(reply);
      body += (uint64_t)tool.len + reply.len;
      // Truncate: drop the oldest non-system turn (a tool/reply pair) while over the cap.
      while (sys.len + body > P.cap_tokens && turns_kept.size() > 2) {
        body -= (uint64_t)turns_kept[0].len + turns_kept[1].len;
        turns_kept.erase(turns_kept.begin(), turns_kept.begin() + 2);
      }
      ctx.clear();
      ctx.push_back(sys);
      for (const Seg& g : turns_kept) ctx.push_back(g);
      // A single turn longer than the cap keeps only its leading tokens.
      uint64_t total = sys.len + body;
      if (total > P.cap_tokens) {
        uint64_t over = total - P.cap_tokens;
        for (size_t i = ctx.size(); i-- > 1 && over > 0;) {
          uint64_t cut = std::min<uint64_t>(over, ctx[i].len > 1 ? ctx[i].len - 1 : 0);
          ctx[i].len -= (uint32_t)cut;
          over -= cut;
        }
      }
      push_request(tr, (int64_t)(t * 1e6), sid, j, ctx);
    }
  }
  tr.n_sessions += P.n_sessions;
}

void finish(Trace& tr) {
  tr.order.resize(tr.reqs.size());
  for (uint32_t i = 0; i < tr.order.size(); ++i) tr.order[i] = i;
  std::sort(tr.order.begin(), tr.order.end(), [&](uint32_t a, uint32_t b) {
    const Req &x = tr.reqs[a], &y = tr.reqs[b];
    if (x.ts_us != y.ts_us) return x.ts_us < y.ts_us;
    if (x.session != y.session) return x.session < y.session;
    return x.turn < y.turn;
  });
  tr.n_tok = 0;
  for (const Req& q : tr.reqs) tr.n_tok += q.ntok;
}

// ---- named workloads (the session counts are the scale knob; see the design notes) ----
ConvParams conv_tiny() {  // tiny conversational trace
  return ConvParams{444, 3600.0, false, 0.5, 6.0, 0, 30.0, 0.10, 10, 512, 2048, 0.0, 200.0, 400.0, 1.0};
}
ConvParams conv_chat() {  // conversational chat trace
  ConvParams p{5600, 0.0, false, 0.6, 4.0, 1, 45.0, 0.3, 50, 1024, 4096, 1.0, 300.0, 600.0, 1.0};
  p.window_s = 5.9 * (double)p.n_sessions;  // ~16 concurrent multi-turn sessions
  return p;
}
AgentParams agent_coding() {  // agentic coding trace
  AgentParams p{560, 0.0, false, 1.2, 400, 2048.0, 500.0, 1.0, 131072, 5.0, 20.0, 10, 2048, 8192};
  p.window_s = 31.4 * (double)p.n_sessions;  // ~14 concurrent sessions
  return p;
}

}  // namespace

extern "C" {

struct tg_trace;  // opaque

// Build the request plan for workload `cfg` (0 tiny conversational, 1 chat,
// 2 agentic coding, 3 mixed 24 h) from `seed`.  sessions_a / sessions_b,
// when > 0, override the session counts (b applies to the agentic half of
// the mixed workload).  Returns an opaque handle or null.
tg_trace* tg_make(int cfg, uint64_t seed, int64_t sessions_a, int64_t sessions_b) {
  Trace* tr = new Trace();
  uint64_t root = derive(0x7072656669786361ULL, seed);
  switch (cfg) {
    case 0: {
      ConvParams p = conv_tiny();
      if (sessions_a > 0) p.n_sessions = (uint64_t)sessions_a;
      gen_conv(*tr, p, derive(root, 0), 0);
      break;
    }
    case 1: {
      ConvParams p = conv_chat();
      if (sessions_a > 0) { p.n_sessions = (uint64_t)sessions_a; p.window_s = 5.9 * (double)p.n_sessions; }
      gen_conv(*tr, p, derive(root, 1), 0);
      break;
    }
    case 2: {
      AgentParams p = agent_coding();
      if (sessions_a > 0) { p.n_sessions = (uint64_t)sessions_a; p.window_s = 31.4 * (double)p.n_sessions; }
      gen_agent(*tr, p, derive(root, 2), 0);
      break;
    }
    case 3: {  // half the tokens from each generator, session starts over 24 h, diurnal rate
      ConvParams c = conv_chat();
      AgentParams a = agent_coding();
      c.n_sessions = sessions_a > 0 ? (uint64_t)sessions_a : 178000;
      a.n_sessions = sessions_b > 0 ? (uint64_t)sessions_b : 1300;
      c.window_s = a.window_s = 86400.0;
      c.diurnal = a.diurnal = true;
      gen_conv(*tr, c, derive(root, 31), 0);
      gen_agent(*tr, a, derive(root, 32), c.n_sessions);  // labels stay dense: 0 .. sessions - 1
      break;
    }
    default:
      delete tr;
      return nullptr;
  }
  finish(*tr);
  return (tg_trace*)tr;
}

void tg_sizes(const tg_trace* h, uint64_t* n_req, uint64_t* n_tok, uint64_t* n_sessions) {
  const Trace* tr = (const Trace*)h;
  *n_req = tr->reqs.size();
  *n_tok = tr->n_tok;
  *n_sessions = tr->n_sessions;
}

// Write the request table of the first n_req requests in trace order:
// req_tok_off[n_req+1], req_ts_us[n_req], req_session[n_req].
void tg_offsets(const tg_trace* h, uint64_t n_req, uint64_t* req_tok_off, int64_t* req_ts_us,
                uint64_t* req_session) {
  const Trace* tr = (const Trace*)h;
  if (n_req > tr->reqs.size()) n_req = tr->reqs.size();
  req_tok_off[0] = 0;
  for (uint64_t i = 0; i < n_req; ++i) {
    const Req& q = tr->reqs[tr->order[i]];
    req_tok_off[i + 1] = req_tok_off[i] + q.ntok;
    req_ts_us[i] = q.ts_us;
    req_session[i] = q.session;
  }
}

// Write the tokens of the first n_req requests; req_tok_off is the table that
// tg_offsets wrote.  Runs on `threads` host threads.
void tg_fill_tokens(const tg_trace* h, uint64_t n_req, const uint64_t* req_tok_off, uint32_t* tokens,
                    int threads) {
  const Trace* tr = (const Trace*)h;
  if (n_req > tr->reqs.size()) n_req = tr->reqs.size();
  if (threads < 1) threads = 1;
  std::atomic<uint64_t> next{0};
  auto work = [&]() {
    for (;;) {
      uint64_t i = next.fetch_add(1);
      if (i >= n_req) break;
      const Req& q = tr->reqs[tr->order[i]];
      uint32_t* out = tokens + req_tok_off[i];
      for (uint32_t g = 0; g < q.seg_count; ++g) {
        const Seg& s = tr->segs[q.seg_begin + g];
        for (uint32_t p = 0; p < s.len; ++p) *out++ = seg_token(s.key, p);
      }
    }
  };
  std::vector<std::thread> pool;
  for (int t = 1; t < threads; ++t) pool.emplace_back(work);
  work();
  for (auto& th : pool) th.join();
}

void tg_free(tg_trace* h) { delete (Trace*)h; }

// The deterministic real functions, exported so tests can check them against libm.
double tg_det_log(double x) { return det_log(x); }
double tg_det_exp(double x) { return det_exp(x); }
double tg_det_cos(double x) { return det_cos(x); }
uint64_t tg_sm64_at(uint64_t k, uint64_t n) { return sm64_at(k, n); }

}  // extern "C"
