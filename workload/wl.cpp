// wl.cpp -- seeded synthetic workload generator (see wl.h for the model).
// Input source shared by the oracle and the CUDA path; holds no radix-tree or routing arithmetic.
#include "wl.h"

#include <algorithm>
#include <cmath>
#include <cstring>
#include <thread>
#include <vector>

namespace {

// ---- published generators -------------------------------------------------------------------------
// SplitMix64 (Steele, Lea & Flood 2014; constants as published by Vigna).
inline uint64_t splitmix64(uint64_t& st) {
  uint64_t z = (st += 0x9E3779B97F4A7C15ull);
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
inline uint64_t rotl(uint64_t x, int k) { return (x << k) | (x >> (64 - k)); }

// xoshiro256** 1.0 (Blackman & Vigna 2018), seeded with four SplitMix64 outputs.
struct Rng {
  uint64_t s[4];
  explicit Rng(uint64_t seed) {
    uint64_t sm = seed;
    for (int i = 0; i < 4; ++i) s[i] = splitmix64(sm);
  }
  uint64_t next() {
    const uint64_t result = rotl(s[1] * 5, 7) * 9;
    const uint64_t t = s[1] << 17;
    s[2] ^= s[0];
    s[3] ^= s[1];
    s[1] ^= s[2];
    s[0] ^= s[3];
    s[2] ^= t;
    s[3] = rotl(s[3], 45);
    return result;
  }
  // Uniform integer in [0, range), range >= 1: Lemire, "Fast random integer generation in an interval"
  // (ACM TOMACS 2019), multiply-shift with rejection of the biased low part.
  uint64_t below(uint64_t range) {
    unsigned __int128 m = (unsigned __int128)next() * range;
    uint64_t lo = (uint64_t)m;
    if (lo < range) {
      const uint64_t thresh = (0 - range) % range;
      while (lo < thresh) {
        m = (unsigned __int128)next() * range;
        lo = (uint64_t)m;
      }
    }
    return (uint64_t)(m >> 64);
  }
  int64_t uniform(int64_t lo, int64_t hi) { return lo + (int64_t)below((uint64_t)(hi - lo) + 1); }
  double unit() { return (double)(next() >> 11) * 0x1.0p-53; }
};

enum : uint64_t { TAG_PREFIX = 1, TAG_ASSIGN = 2, TAG_SEQ = 3, TAG_REQ = 4, TAG_LOAD = 5, TAG_DELTA = 6 };
const int64_t STALE_STEP = -1;

inline uint64_t mix(uint64_t h, uint64_t v) {
  uint64_t st = h ^ v;
  return splitmix64(st);
}
// Independent stream keyed by (seed, tag, a, b).
inline Rng stream(uint64_t seed, uint64_t tag, uint64_t a, uint64_t b) {
  return Rng(mix(mix(mix(seed, tag), a), b));
}

// Cumulative Zipf weights (k+1)^-s over n ranks.
std::vector<double> zipf_cdf(int64_t n, double s) {
  std::vector<double> c((size_t)n);
  double acc = 0.0;
  for (int64_t k = 0; k < n; ++k) {
    acc += std::pow((double)(k + 1), -s);
    c[(size_t)k] = acc;
  }
  return c;
}
// Smallest index whose cumulative weight exceeds u * total.
inline int64_t zipf_pick(const std::vector<double>& cdf, double u) {
  if (cdf.empty()) return -1;
  const double x = u * cdf.back();
  int64_t k = (int64_t)(std::upper_bound(cdf.begin(), cdf.end(), x) - cdf.begin());
  return k < (int64_t)cdf.size() ? k : (int64_t)cdf.size() - 1;
}

template <class F>
void parallel_for(int64_t n, int32_t n_threads, F fn) {
  if (n <= 0) return;
  int64_t t = n_threads < 1 ? 1 : n_threads;
  if (t > n) t = n;
  if (t == 1) {
    fn(0, n);
    return;
  }
  std::vector<std::thread> th;
  th.reserve((size_t)t);
  for (int64_t i = 0; i < t; ++i) {
    const int64_t b = n * i / t, e = n * (i + 1) / t;
    th.emplace_back([=]() { fn(b, e); });
  }
  for (auto& x : th) x.join();
}

struct SeqRec {
  int32_t k;        // prefix index, -1 = none
  int32_t suf_len;  // suffix length
  int64_t j;        // sequence id within its tree (keys the suffix stream)
};
struct Op {
  int32_t code;  // 0 INSERT, 1 DELETE
  SeqRec seq;
};
struct Tree {
  std::vector<int32_t> assigned;  // assigned prefix ids, ascending
  std::vector<double> cdf;        // Zipf weights renormalised over `assigned`
  std::vector<SeqRec> live;       // sequences currently stored in the replica
  std::vector<SeqRec> exact;      // exact tree (stale replicas only)
  std::vector<Op> pending;        // last delta drawn for this tree
  int64_t next_j = 0;
};

}  // namespace

struct wl_gen {
  wl_params prm;
  uint64_t seed;
  std::vector<int64_t> pre_off;
  std::vector<int32_t> pre_len;
  std::vector<int32_t> pre_tok;
  std::vector<double> zipf_all;
  std::vector<Tree> trees;

  // Draws the identity of sequence j of tree p and leaves `r` positioned at its suffix tokens.
  SeqRec draw_seq(int32_t p, int64_t j, Rng& r) const {
    const Tree& t = trees[(size_t)p];
    SeqRec s;
    const int64_t pick = zipf_pick(t.cdf, r.unit());
    s.k = pick < 0 ? -1 : t.assigned[(size_t)pick];
    s.suf_len = (int32_t)r.uniform(prm.suf_lo, prm.suf_hi);
    s.j = j;
    return s;
  }
  void suffix_tokens(int32_t p, const SeqRec& s, int32_t* out) const {
    Rng r = stream(seed, TAG_SEQ, (uint64_t)p, (uint64_t)s.j);
    (void)draw_seq(p, s.j, r);
    for (int32_t i = 0; i < s.suf_len; ++i) out[i] = (int32_t)r.below((uint64_t)prm.vocab);
  }
  SeqRec new_seq(int32_t p, int64_t j) const {
    Rng r = stream(seed, TAG_SEQ, (uint64_t)p, (uint64_t)j);
    return draw_seq(p, j, r);
  }
  void make_delta(int32_t p, int64_t step, int64_t n_del, int64_t n_ins) {
    Tree& t = trees[(size_t)p];
    Rng r = stream(seed, TAG_DELTA, (uint64_t)p, (uint64_t)step);
    const int64_t n = (int64_t)t.live.size();
    if (n_del > n) n_del = n;
    t.pending.clear();
    t.pending.reserve((size_t)(n_del + n_ins));
    // n_del distinct stored sequences: partial Fisher-Yates moving the chosen ones to the back.
    for (int64_t i = 0; i < n_del; ++i) {
      const int64_t pick = (int64_t)r.below((uint64_t)(n - i));
      std::swap(t.live[(size_t)pick], t.live[(size_t)(n - 1 - i)]);
      t.pending.push_back(Op{1, t.live[(size_t)(n - 1 - i)]});
    }
    t.live.resize((size_t)(n - n_del));
    for (int64_t i = 0; i < n_ins; ++i) {
      const SeqRec s = new_seq(p, t.next_j++);
      t.pending.push_back(Op{0, s});
      t.live.push_back(s);
    }
    // Random interleaving of the ops (Fisher-Yates).
    for (int64_t i = (int64_t)t.pending.size() - 1; i > 0; --i) {
      const int64_t q = (int64_t)r.below((uint64_t)(i + 1));
      std::swap(t.pending[(size_t)i], t.pending[(size_t)q]);
    }
  }
  // Request b: kind, prefix choice and lengths are drawn first so that a length-only pass replays them.
  struct ReqShape {
    int32_t fresh;    // 1: fresh random prefix
    int32_t k;        // shared prefix id
    int32_t pre_len;  // tokens taken from the prefix (fresh: random prefix length)
    int32_t forced;   // diverge mode: the forced token after pre_len tokens, -1 = none
    int32_t tail;     // random tail length
    int64_t len() const { return (int64_t)pre_len + (forced >= 0 ? 1 : 0) + tail; }
  };
  ReqShape req_shape(int64_t b, Rng& r) const {
    ReqShape s{0, -1, 0, -1, 0};
    const double u = r.unit();
    if (u < prm.fresh_frac || prm.n_prefix == 0) {
      s.fresh = 1;
      s.pre_len = (int32_t)r.uniform(prm.pre_lo, prm.pre_hi);
    } else {
      s.k = (int32_t)zipf_pick(zipf_all, r.unit());
      const int32_t L = pre_len[(size_t)s.k];
      if (prm.diverge && L > 0) {
        s.pre_len = (int32_t)r.uniform(0, L - 1);
        const int32_t avoid = pre_tok[(size_t)(pre_off[(size_t)s.k] + s.pre_len)];
        const int32_t t = (int32_t)r.below((uint64_t)(prm.vocab - 1));
        s.forced = t + (t >= avoid ? 1 : 0);
      } else {
        s.pre_len = L;
      }
    }
    s.tail = (int32_t)r.uniform(prm.req_suf_lo, prm.req_suf_hi);
    (void)b;
    return s;
  }
};

static bool params_ok(const wl_params* p) {
  if (!p) return false;
  if (p->P < 1 || p->vocab < 2 || p->n_seq < 0 || p->n_prefix < 0 || p->B < 0) return false;
  if (p->pre_lo < 0 || p->pre_hi < p->pre_lo || p->suf_lo < 0 || p->suf_hi < p->suf_lo) return false;
  if (p->req_suf_lo < 0 || p->req_suf_hi < p->req_suf_lo) return false;
  if (p->load_hi < 0 || p->alpha < 0) return false;
  if (p->diverge && p->pre_lo < 1) return false;
  return true;
}

extern "C" {

uint64_t wl_default_seed(int32_t cfg_id) { return 0x9E3779B97F4A7C15ull ^ (uint64_t)(int64_t)cfg_id; }

int wl_preset(int32_t cfg_id, wl_params* o) {
  if (!o) return -1;
  std::memset(o, 0, sizeof(*o));
  o->vocab = 32000;
  o->assign_prob = 0.5;
  o->fresh_frac = 0.2;
  o->suf_lo = 32;
  o->suf_hi = 128;
  o->req_suf_lo = 32;
  o->req_suf_hi = 128;
  o->load_hi = 255;
  o->alpha = 2;
  switch (cfg_id) {
    case 0:  // P=4, 1,000 sequences, 57 prefixes of 256-1,024 tokens, 4,096 requests, load 0-63, alpha 4
      o->P = 4; o->n_seq = 1000; o->n_prefix = 57; o->pre_lo = 256; o->pre_hi = 1024; o->zipf_s = 1.1;
      o->B = 4096; o->load_hi = 63; o->alpha = 4;
      return 0;
    case 1:  // P=16, 20,000 sequences, 512 prefixes of 128-2,048 tokens, 65,536 requests
      o->P = 16; o->n_seq = 20000; o->n_prefix = 512; o->pre_lo = 128; o->pre_hi = 2048; o->zipf_s = 1.1;
      o->B = 65536;
      return 0;
    case 2:  // stale replicas: P=64, 2,000 prefixes, Zipf 1.5, 262,144 requests, -10% / +5% per replica
      o->P = 64; o->n_seq = 20000; o->n_prefix = 2000; o->pre_lo = 128; o->pre_hi = 2048; o->zipf_s = 1.5;
      o->B = 262144; o->stale_del_frac = 0.10; o->stale_ins_frac = 0.05;
      return 0;
    case 3:  // long-context deep walks: P=32, 5,000 sequences, prefixes 4,096-32,768, suffixes 256-1,024
      o->P = 32; o->n_seq = 5000; o->n_prefix = 256; o->pre_lo = 4096; o->pre_hi = 32768; o->zipf_s = 1.1;
      o->suf_lo = 256; o->suf_hi = 1024; o->req_suf_lo = 256; o->req_suf_hi = 1024;
      o->B = 16384; o->fresh_frac = 0.1; o->diverge = 1;
      return 0;
    case 4:  // scale + anti-entropy: P=256, 100,000 sequences, 10,000 prefixes of 128-4,096, 1,048,576 requests
      o->P = 256; o->n_seq = 100000; o->n_prefix = 10000; o->pre_lo = 128; o->pre_hi = 4096; o->zipf_s = 1.2;
      o->B = 1048576; o->delta_frac = 0.05;
      return 0;
    default:
      return -1;
  }
}

wl_gen* wl_create(const wl_params* prm, uint64_t seed) {
  if (!params_ok(prm)) return nullptr;
  wl_gen* g = new wl_gen();
  g->prm = *prm;
  g->seed = seed;
  const wl_params& P = g->prm;
  // Prefix table.
  g->pre_off.resize((size_t)P.n_prefix);
  g->pre_len.resize((size_t)P.n_prefix);
  int64_t total = 0;
  for (int32_t k = 0; k < P.n_prefix; ++k) {
    Rng r = stream(seed, TAG_PREFIX, (uint64_t)k, 0);
    g->pre_off[(size_t)k] = total;
    g->pre_len[(size_t)k] = (int32_t)r.uniform(P.pre_lo, P.pre_hi);
    total += g->pre_len[(size_t)k];
  }
  g->pre_tok.resize((size_t)total);
  for (int32_t k = 0; k < P.n_prefix; ++k) {
    Rng r = stream(seed, TAG_PREFIX, (uint64_t)k, 0);
    (void)r.uniform(P.pre_lo, P.pre_hi);
    int32_t* dst = g->pre_tok.data() + g->pre_off[(size_t)k];
    for (int32_t i = 0; i < g->pre_len[(size_t)k]; ++i) dst[i] = (int32_t)r.below((uint64_t)P.vocab);
  }
  g->zipf_all = zipf_cdf(P.n_prefix, P.zipf_s);
  // Assignment of prefixes to trees and per-tree sequence lists.
  g->trees.resize((size_t)P.P);
  for (int32_t p = 0; p < P.P; ++p) {
    Tree& t = g->trees[(size_t)p];
    Rng r = stream(seed, TAG_ASSIGN, (uint64_t)p, 0);
    double acc = 0.0;
    for (int32_t k = 0; k < P.n_prefix; ++k) {
      if (r.unit() < P.assign_prob) {
        t.assigned.push_back(k);
        acc += std::pow((double)(k + 1), -P.zipf_s);
        t.cdf.push_back(acc);
      }
    }
  }
  const bool stale = P.stale_del_frac > 0.0 || P.stale_ins_frac > 0.0;
  parallel_for(P.P, (int32_t)std::min<int64_t>(P.P, 16), [&](int64_t b, int64_t e) {
    for (int64_t p = b; p < e; ++p) {
      Tree& t = g->trees[(size_t)p];
      t.live.reserve((size_t)P.n_seq);
      for (int64_t j = 0; j < P.n_seq; ++j) t.live.push_back(g->new_seq((int32_t)p, j));
      t.next_j = P.n_seq;
      if (stale && p >= 1) {
        t.exact = t.live;
        const int64_t n = (int64_t)t.live.size();
        g->make_delta((int32_t)p, STALE_STEP, (int64_t)std::ceil(P.stale_del_frac * (double)n),
                      (int64_t)std::ceil(P.stale_ins_frac * (double)n));
      }
    }
  });
  return g;
}

void wl_free(wl_gen* g) { delete g; }
void wl_get_params(const wl_gen* g, wl_params* out) { *out = g->prm; }

int64_t wl_prefix_pool_size(const wl_gen* g) { return (int64_t)g->pre_tok.size(); }
void wl_prefix_pool(const wl_gen* g, int32_t* pool, int64_t* pre_off, int32_t* pre_len) {
  if (pool && !g->pre_tok.empty()) std::memcpy(pool, g->pre_tok.data(), g->pre_tok.size() * sizeof(int32_t));
  if (pre_off) std::copy(g->pre_off.begin(), g->pre_off.end(), pre_off);
  if (pre_len) std::copy(g->pre_len.begin(), g->pre_len.end(), pre_len);
}

static const std::vector<SeqRec>* tree_list(const wl_gen* g, int32_t p, int32_t which) {
  if (!g || p < 0 || p >= g->prm.P) return nullptr;
  const Tree& t = g->trees[(size_t)p];
  if (which == 1 && !t.exact.empty()) return &t.exact;
  if (which == 0 || which == 1) return &t.live;
  return nullptr;
}

int wl_tree_size(const wl_gen* g, int32_t p, int32_t which, int64_t* n_seq, int64_t* n_segs, int64_t* n_suf) {
  const std::vector<SeqRec>* L = tree_list(g, p, which);
  if (!L) return -1;
  int64_t segs = 0, suf = 0;
  for (const SeqRec& s : *L) {
    segs += 1 + (s.k >= 0 ? 1 : 0);
    suf += s.suf_len;
  }
  if (n_seq) *n_seq = (int64_t)L->size();
  if (n_segs) *n_segs = segs;
  if (n_suf) *n_suf = suf;
  return 0;
}

// Emits the segments of one sequence: the prefix run (if any), then its suffix run.
static void emit_seq(const wl_gen* g, int32_t p, const SeqRec& s, int64_t* seg_off, int32_t* seg_len, int64_t& si,
                     int32_t* suffix_out, int64_t& cur, int64_t suffix_base) {
  if (s.k >= 0) {
    seg_off[si] = g->pre_off[(size_t)s.k];
    seg_len[si] = g->pre_len[(size_t)s.k];
    ++si;
  }
  seg_off[si] = suffix_base + cur;
  seg_len[si] = s.suf_len;
  ++si;
  g->suffix_tokens(p, s, suffix_out + cur);
  cur += s.suf_len;
}

int wl_tree_fill(const wl_gen* g, int32_t p, int32_t which, int64_t* seg_begin, int64_t* seg_off, int32_t* seg_len,
                 int32_t* suffix_out, int64_t suffix_base) {
  const std::vector<SeqRec>* L = tree_list(g, p, which);
  if (!L) return -1;
  int64_t si = 0, cur = 0;
  for (size_t i = 0; i < L->size(); ++i) {
    seg_begin[i] = si;
    emit_seq(g, p, (*L)[i], seg_off, seg_len, si, suffix_out, cur, suffix_base);
  }
  seg_begin[L->size()] = si;
  return 0;
}

static void req_lengths(const wl_gen* g, int64_t b0, int64_t b1, int64_t* len, int32_t n_threads) {
  parallel_for(b1 - b0, n_threads, [&](int64_t s, int64_t e) {
    for (int64_t i = s; i < e; ++i) {
      Rng r = stream(g->seed, TAG_REQ, (uint64_t)(b0 + i), 0);
      len[i] = g->req_shape(b0 + i, r).len();
    }
  });
}

int64_t wl_requests_size(const wl_gen* g, int64_t b0, int64_t b1, int32_t n_threads) {
  if (!g || b0 < 0 || b1 < b0) return -1;
  std::vector<int64_t> len((size_t)(b1 - b0));
  req_lengths(g, b0, b1, len.data(), n_threads);
  int64_t tot = 0;
  for (int64_t x : len) tot += x;
  return tot;
}

int wl_requests_fill(const wl_gen* g, int64_t b0, int64_t b1, int32_t* tokens, int64_t* offsets, int32_t n_threads) {
  if (!g || b0 < 0 || b1 < b0) return -1;
  const int64_t n = b1 - b0;
  std::vector<int64_t> len((size_t)n);
  req_lengths(g, b0, b1, len.data(), n_threads);
  offsets[0] = 0;
  for (int64_t i = 0; i < n; ++i) offsets[i + 1] = offsets[i] + len[(size_t)i];
  const wl_params& P = g->prm;
  parallel_for(n, n_threads, [&](int64_t s, int64_t e) {
    for (int64_t i = s; i < e; ++i) {
      Rng r = stream(g->seed, TAG_REQ, (uint64_t)(b0 + i), 0);
      const wl_gen::ReqShape sh = g->req_shape(b0 + i, r);
      int32_t* dst = tokens + offsets[i];
      if (sh.fresh) {
        for (int32_t t = 0; t < sh.pre_len; ++t) dst[t] = (int32_t)r.below((uint64_t)P.vocab);
      } else if (sh.pre_len > 0) {
        std::memcpy(dst, g->pre_tok.data() + g->pre_off[(size_t)sh.k], (size_t)sh.pre_len * sizeof(int32_t));
      }
      int64_t c = sh.pre_len;
      if (sh.forced >= 0) dst[c++] = sh.forced;
      for (int32_t t = 0; t < sh.tail; ++t) dst[c++] = (int32_t)r.below((uint64_t)P.vocab);
    }
  });
  return 0;
}

int wl_load_fill(const wl_gen* g, int64_t step, int32_t vary, int32_t* load) {
  if (!g) return -1;
  Rng r = stream(g->seed, TAG_LOAD, vary ? (uint64_t)step : 0, 0);
  for (int32_t p = 0; p < g->prm.P; ++p) load[p] = (int32_t)r.uniform(0, g->prm.load_hi);
  return 0;
}

int wl_delta_make(wl_gen* g, int32_t p0, int32_t p1, int64_t step, double del_frac, double ins_frac, int32_t n_threads) {
  if (!g || p0 < 0 || p1 > g->prm.P || p1 < p0 || step < 0 || del_frac < 0 || ins_frac < 0) return -1;
  parallel_for(p1 - p0, n_threads, [&](int64_t s, int64_t e) {
    for (int64_t i = s; i < e; ++i) {
      const int32_t p = (int32_t)(p0 + i);
      const double n = (double)g->trees[(size_t)p].live.size();
      g->make_delta(p, step, (int64_t)std::ceil(del_frac * n), (int64_t)std::ceil(ins_frac * n));
    }
  });
  return 0;
}

int wl_delta_size(const wl_gen* g, int32_t p0, int32_t p1, int64_t* n_ops, int64_t* n_segs, int64_t* n_suf) {
  if (!g || p0 < 0 || p1 > g->prm.P || p1 < p0) return -1;
  int64_t ops = 0, segs = 0, suf = 0;
  for (int32_t p = p0; p < p1; ++p) {
    for (const Op& o : g->trees[(size_t)p].pending) {
      ++ops;
      segs += 1 + (o.seq.k >= 0 ? 1 : 0);
      suf += o.seq.suf_len;
    }
  }
  if (n_ops) *n_ops = ops;
  if (n_segs) *n_segs = segs;
  if (n_suf) *n_suf = suf;
  return 0;
}

int wl_delta_fill(const wl_gen* g, int32_t p0, int32_t p1, int32_t* op, int64_t* seg_begin, int64_t* seg_off,
                  int32_t* seg_len, int32_t* suffix_out, int64_t suffix_base, int64_t* peer_begin, int32_t n_threads) {
  if (!g || p0 < 0 || p1 > g->prm.P || p1 < p0) return -1;
  const int32_t np = p1 - p0;
  // Per-tree starting offsets of ops, segments and suffix tokens.
  std::vector<int64_t> o0((size_t)np + 1, 0), s0((size_t)np + 1, 0), t0((size_t)np + 1, 0);
  for (int32_t i = 0; i < np; ++i) {
    int64_t ops = 0, segs = 0, suf = 0;
    for (const Op& o : g->trees[(size_t)(p0 + i)].pending) {
      ++ops;
      segs += 1 + (o.seq.k >= 0 ? 1 : 0);
      suf += o.seq.suf_len;
    }
    o0[(size_t)i + 1] = o0[(size_t)i] + ops;
    s0[(size_t)i + 1] = s0[(size_t)i] + segs;
    t0[(size_t)i + 1] = t0[(size_t)i] + suf;
  }
  if (peer_begin)
    for (int32_t i = 0; i <= np; ++i) peer_begin[i] = o0[(size_t)i];
  parallel_for(np, n_threads, [&](int64_t s, int64_t e) {
    for (int64_t i = s; i < e; ++i) {
      const int32_t p = (int32_t)(p0 + i);
      int64_t oi = o0[(size_t)i], si = s0[(size_t)i], cur = t0[(size_t)i];
      for (const Op& o : g->trees[(size_t)p].pending) {
        op[oi] = o.code;
        seg_begin[oi] = si;
        emit_seq(g, p, o.seq, seg_off, seg_len, si, suffix_out, cur, suffix_base);
        ++oi;
      }
    }
  });
  seg_begin[o0[(size_t)np]] = s0[(size_t)np];
  return 0;
}

uint64_t wl_splitmix64(uint64_t* state) { return splitmix64(*state); }
void wl_xoshiro_seed(uint64_t seed, uint64_t s[4]) {
  Rng r(seed);
  for (int i = 0; i < 4; ++i) s[i] = r.s[i];
}
uint64_t wl_xoshiro_next(uint64_t s[4]) {
  Rng r(0);
  for (int i = 0; i < 4; ++i) r.s[i] = s[i];
  const uint64_t v = r.next();
  for (int i = 0; i < 4; ++i) s[i] = r.s[i];
  return v;
}
uint64_t wl_bounded(uint64_t s[4], uint64_t range) {
  Rng r(0);
  for (int i = 0; i < 4; ++i) r.s[i] = s[i];
  const uint64_t v = r.below(range);
  for (int i = 0; i < 4; ++i) s[i] = r.s[i];
  return v;
}
int32_t wl_zipf_index(int32_t n, double s, double u) { return (int32_t)zipf_pick(zipf_cdf(n, s), u); }

}  // extern "C"
