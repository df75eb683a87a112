// snapshot.cpp -- host side of the full-snapshot format (Section 2, sendTrie): the canonical builder,
// the validity check of received snapshots, and the canonical export of a device tree.
#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "internal.h"

namespace p2p {

static thread_local std::string g_error;
void set_global_error(const std::string& msg) { g_error = msg; }
const char* global_error() { return g_error.c_str(); }

// ---- segmented sequences ---------------------------------------------------------------------------

bool check_seqs(const p2p_seqs* s, std::string& err, int64_t* max_len, std::vector<int64_t>* lens) {
  if (!s) return err = "seqs is NULL", false;
  if (s->n < 0 || s->n_segs < 0 || s->n_pool < 0) return err = "negative size in seqs", false;
  if (!s->seg_begin) return err = "seg_begin is NULL", false;
  if ((s->n_segs > 0 && (!s->seg_off || !s->seg_len)) || (s->n_pool > 0 && !s->pool))
    return err = "NULL array in seqs", false;
  if (s->seg_begin[0] != 0 || s->seg_begin[s->n] != s->n_segs) return err = "seg_begin must run from 0 to n_segs", false;
  int64_t mx = 0;
  if (lens) lens->assign((size_t)s->n, 0);
  for (int64_t i = 0; i < s->n; ++i) {
    const int64_t a = s->seg_begin[i], b = s->seg_begin[i + 1];
    if (b < a) return err = "seg_begin not non-decreasing at sequence " + std::to_string(i), false;
    int64_t L = 0;
    for (int64_t g = a; g < b; ++g) {
      const int64_t off = s->seg_off[g], len = s->seg_len[g];
      if (len < 0 || off < 0 || off > s->n_pool - len) return err = "segment " + std::to_string(g) + " outside the pool", false;
      L += len;
    }
    if (L > INT32_MAX) return err = "sequence " + std::to_string(i) + " longer than 2^31-1 tokens", false;
    if (lens) (*lens)[(size_t)i] = L;
    mx = std::max(mx, L);
  }
  if (max_len) *max_len = mx;
  return true;
}

namespace {

// Lexicographic comparison of two segmented sequences.  Runs that start at the same pool address are
// identical and skipped whole, so sequences sharing a referenced prefix compare in O(1) per run.
void compare(const p2p_seqs& S, int64_t a, int64_t b, int64_t& lcp, int& cmp) {
  int64_t sa = S.seg_begin[a], ea = S.seg_begin[a + 1], sb = S.seg_begin[b], eb = S.seg_begin[b + 1];
  int64_t oa = 0, ob = 0;
  lcp = 0;
  for (;;) {
    while (sa < ea && oa == S.seg_len[sa]) ++sa, oa = 0;
    while (sb < eb && ob == S.seg_len[sb]) ++sb, ob = 0;
    if (sa == ea || sb == eb) {
      cmp = (sa == ea) ? (sb == eb ? 0 : -1) : 1;
      return;
    }
    const int32_t* pa = S.pool + S.seg_off[sa] + oa;
    const int32_t* pb = S.pool + S.seg_off[sb] + ob;
    const int64_t m = std::min<int64_t>(S.seg_len[sa] - oa, S.seg_len[sb] - ob);
    int64_t k = 0;
    if (pa != pb) {
      while (k + 64 <= m && std::memcmp(pa + k, pb + k, 64 * sizeof(int32_t)) == 0) k += 64;
      while (k < m && pa[k] == pb[k]) ++k;
      if (k < m) {
        lcp += k;
        cmp = pa[k] < pb[k] ? -1 : 1;
        return;
      }
    }
    lcp += m;
    oa += m;
    ob += m;
  }
}

// Copies tokens [from, to) of sequence i.
void copy_range(const p2p_seqs& S, int64_t i, int64_t from, int64_t to, int32_t* out) {
  int64_t pos = 0;
  for (int64_t g = S.seg_begin[i]; g < S.seg_begin[i + 1] && pos < to; ++g) {
    const int64_t L = S.seg_len[g];
    const int64_t lo = std::max(from, pos), hi = std::min(to, pos + L);
    if (lo < hi) std::memcpy(out + (lo - from), S.pool + S.seg_off[g] + (lo - pos), (size_t)(hi - lo) * sizeof(int32_t));
    pos += L;
  }
}

int32_t token_at(const p2p_seqs& S, int64_t i, int64_t at) {
  int64_t pos = 0;
  for (int64_t g = S.seg_begin[i]; g < S.seg_begin[i + 1]; ++g) {
    if (at < pos + S.seg_len[g]) return S.pool[S.seg_off[g] + (at - pos)];
    pos += S.seg_len[g];
  }
  return 0;
}

struct BNode {
  int64_t depth;   // tokens from the root to the end of this node's edge
  int64_t src;     // a sequence whose path passes through this node (gives the label tokens)
  int64_t parent;
  int64_t term;
  std::vector<int64_t> kids;  // ascending by first token (appended in sorted order)
};

}  // namespace

// Canonical snapshot of a multiset: sort the sequences, then build the compressed trie from the sorted
// order and the LCPs of neighbours (the rightmost path is kept on a stack; an LCP that ends inside an edge
// splits it).  Finally number the nodes in preorder and pack labels and child lists in node order.
bool build_snapshot(const p2p_seqs& S, p2p_snapshot& out, std::string& err) {
  std::vector<int64_t> lens;
  if (!check_seqs(&S, err, nullptr, &lens)) return false;
  const int64_t n = S.n;
  std::vector<int64_t> ord((size_t)n);
  for (int64_t i = 0; i < n; ++i) ord[(size_t)i] = i;
  std::sort(ord.begin(), ord.end(), [&](int64_t a, int64_t b) {
    int64_t l;
    int c;
    compare(S, a, b, l, c);
    return c < 0 || (c == 0 && a < b);
  });
  std::vector<BNode> T;
  T.reserve((size_t)(2 * n + 1));
  T.push_back(BNode{0, -1, -1, 0, {}});
  std::vector<int64_t> stack{0};
  for (int64_t r = 0; r < n; ++r) {
    const int64_t i = ord[(size_t)r];
    int64_t l = 0;
    if (r > 0) {
      int c;
      compare(S, ord[(size_t)r - 1], i, l, c);
    }
    int64_t last = -1;
    while (T[(size_t)stack.back()].depth > l) {
      last = stack.back();
      stack.pop_back();
    }
    int64_t top = stack.back();
    if (T[(size_t)top].depth < l) {
      // The previous sequence's path leaves `top` through `last`; split that edge at depth l.
      const int64_t mid = (int64_t)T.size();
      T.push_back(BNode{l, T[(size_t)last].src, top, 0, {last}});
      T[(size_t)top].kids.back() = mid;
      T[(size_t)last].parent = mid;
      stack.push_back(mid);
      top = mid;
    }
    if (lens[(size_t)i] == l) {
      T[(size_t)top].term += 1;
    } else {
      const int64_t leaf = (int64_t)T.size();
      T.push_back(BNode{lens[(size_t)i], i, top, 1, {}});
      T[(size_t)top].kids.push_back(leaf);
      stack.push_back(leaf);
    }
  }
  if ((int64_t)T.size() > INT32_MAX) return err = "snapshot has more than 2^31-1 nodes", false;
  // Preorder numbering.
  std::vector<int64_t> order;
  order.reserve(T.size());
  std::vector<int64_t> st{0};
  while (!st.empty()) {
    const int64_t v = st.back();
    st.pop_back();
    order.push_back(v);
    const auto& k = T[(size_t)v].kids;
    for (auto it = k.rbegin(); it != k.rend(); ++it) st.push_back(*it);
  }
  std::vector<int32_t> id(T.size());
  for (size_t j = 0; j < order.size(); ++j) id[(size_t)order[j]] = (int32_t)j;
  const size_t N = order.size();
  int64_t total_label = 0;
  for (int64_t v : order)
    if (v != 0) total_label += T[(size_t)v].depth - T[(size_t)T[(size_t)v].parent].depth;
  if (total_label > INT32_MAX) return err = "snapshot has more than 2^31-1 label tokens", false;
  out.n_nodes = (int32_t)N;
  out.n_labels = (int32_t)total_label;
  out.label_off.assign(N, 0);
  out.label_len.assign(N, 0);
  out.child_begin.assign(N, 0);
  out.child_count.assign(N, 0);
  out.term_count.assign(N, 0);
  out.child_first_tok.assign(N - 1, 0);
  out.child_idx.assign(N - 1, 0);
  out.labels.assign((size_t)total_label, 0);
  int64_t lab = 0, ch = 0;
  for (size_t j = 0; j < N; ++j) {
    const BNode& b = T[(size_t)order[j]];
    if (b.term > INT32_MAX) return err = "a sequence is stored more than 2^31-1 times", false;
    out.label_off[j] = (int32_t)lab;
    if (order[j] != 0) {
      const int64_t d0 = T[(size_t)b.parent].depth;
      out.label_len[j] = (int32_t)(b.depth - d0);
      copy_range(S, b.src, d0, b.depth, out.labels.data() + lab);
      lab += b.depth - d0;
    }
    out.child_begin[j] = (int32_t)ch;
    out.child_count[j] = (int32_t)b.kids.size();
    out.term_count[j] = (int32_t)b.term;
    for (int64_t k : b.kids) {
      out.child_first_tok[(size_t)ch] = token_at(S, T[(size_t)k].src, b.depth);
      out.child_idx[(size_t)ch] = id[(size_t)k];
      ++ch;
    }
  }
  return true;
}

// Validity rules of p2p_flat_tree (see p2p_router.h).
bool validate_flat(const p2p_flat_tree* t, std::string& err) {
  if (!t) return err = "tree is NULL", false;
  const int64_t N = t->n_nodes, NL = t->n_labels;
  if (N < 1 || NL < 0) return err = "n_nodes must be >= 1 and n_labels >= 0", false;
  if (!t->label_off || !t->label_len || !t->child_begin || !t->child_count || !t->term_count)
    return err = "NULL node array", false;
  if ((N > 1 && (!t->child_first_tok || !t->child_idx)) || (NL > 0 && !t->labels)) return err = "NULL array", false;
  if (t->label_len[0] != 0) return err = "root label must be empty", false;
  std::vector<int64_t> parent((size_t)N, -1);
  for (int64_t v = 0; v < N; ++v) {
    const int64_t off = t->label_off[v], len = t->label_len[v];
    if (off < 0 || len < 0 || off > NL - len) return err = "label of node " + std::to_string(v) + " out of range", false;
    if (v > 0 && len < 1) return err = "non-root node " + std::to_string(v) + " has an empty label", false;
    if (t->term_count[v] < 0) return err = "negative term_count", false;
    const int64_t cb = t->child_begin[v], cc = t->child_count[v];
    if (cb < 0 || cc < 0 || cb > (N - 1) - cc) return err = "child range of node " + std::to_string(v) + " out of range", false;
    for (int64_t e = cb; e < cb + cc; ++e) {
      const int64_t c = t->child_idx[e];
      if (c < 1 || c >= N) return err = "child index out of range", false;
      if (parent[(size_t)c] != -1) return err = "node " + std::to_string(c) + " has two parents", false;
      parent[(size_t)c] = v;
      if (t->child_first_tok[e] != t->labels[t->label_off[c]])
        return err = "child_first_tok differs from the child's first label token", false;
      if (e > cb && !(t->child_first_tok[e - 1] < t->child_first_tok[e]))
        return err = "children of node " + std::to_string(v) + " not strictly ascending", false;
    }
    if (v > 0 && cc <= 1 && t->term_count[v] == 0)
      return err = "non-root node " + std::to_string(v) + " with <= 1 child stores no sequence (not compressed)", false;
  }
  // Reachability from the root and path lengths (a path of more than 2^31-1 tokens is rejected).
  std::vector<int64_t> depth((size_t)N, -1);
  std::vector<int64_t> st{0};
  depth[0] = 0;
  int64_t seen = 0;
  while (!st.empty()) {
    const int64_t v = st.back();
    st.pop_back();
    ++seen;
    for (int64_t e = t->child_begin[v]; e < t->child_begin[v] + t->child_count[v]; ++e) {
      const int64_t c = t->child_idx[e];
      if (depth[(size_t)c] != -1) return err = "cycle in child lists", false;
      depth[(size_t)c] = depth[(size_t)v] + t->label_len[c];
      if (depth[(size_t)c] > INT32_MAX) return err = "a path is longer than 2^31-1 tokens", false;
      st.push_back(c);
    }
  }
  if (seen != N) return err = "nodes unreachable from the root", false;
  return true;
}

// Canonical snapshot of a device tree copied to the host (node, child and label arrays as laid out on the
// device, see internal.h): every node's children are the live slots of its table, sorted by first token.
bool snapshot_from_device_layout(const int4* node, int64_t n_node, const int4* child, int64_t n_child,
                                 const int32_t* label, int64_t n_label, const int32_t* shared, int64_t n_shared,
                                 p2p_snapshot& out, std::string& err) {
  if (n_node < 1) return err = "corrupt device tree (no root)", false;
  auto kids = [&](int64_t v, std::vector<int4>& k) -> bool {
    k.clear();
    const int4 nd = node[v];
    const int32_t bits = tab_bits(nd.y);
    if (bits == 0) return nd.z == 0;
    if (bits > kMaxTabBits || nd.x < 0 || (int64_t)nd.x + ((int64_t)1 << bits) > n_child) return false;
    for (int64_t s = 0; s < ((int64_t)1 << bits); ++s)
      if (child[nd.x + s].y >= 1) k.push_back(child[nd.x + s]);
    std::sort(k.begin(), k.end(), [](const int4& a, const int4& b) { return a.x < b.x; });
    for (size_t i = 1; i < k.size(); ++i)
      if (k[i - 1].x == k[i].x) return false;
    return (int64_t)k.size() == nd.z;
  };
  // Preorder DFS; each stacked item carries the slot through which the node was reached.  A non-root node
  // with one child and no sequence (an LRU tree keeps such nodes where an access ended inside an edge) is
  // merged with its child, so the export is canonical whatever the device layout: an exported node carries
  // the chain of slots whose labels it concatenates, and `order` holds the chain's last node.
  std::vector<int64_t> order, first;  // an exported node's last and first device node
  std::vector<std::vector<int4>> via;
  std::vector<std::vector<int4>> children;
  std::vector<std::pair<int64_t, int4>> st{{0, make_int4(0, 0, 0, 0)}};
  std::vector<int4> k;
  int64_t total_label = 0, visited = 0;
  auto check_label = [&](const int4& e) {
    const bool own = e.z >= 0;
    const int64_t start = own ? e.z : ~(int64_t)e.z;
    return e.w >= 1 && start + e.w <= (own ? n_label : n_shared);
  };
  while (!st.empty()) {
    auto [v, e] = st.back();
    st.pop_back();
    const int64_t v0 = v;
    std::vector<int4> chain;
    for (;;) {
      if (v < 0 || v >= n_node || ++visited > n_node) return err = "corrupt device tree (node index)", false;
      if (v != 0) {
        if (!check_label(e)) return err = "corrupt device tree (label)", false;
        total_label += e.w;
        chain.push_back(e);
      }
      if (!kids(v, k)) return err = "corrupt device tree (children table)", false;
      if (v == 0 || k.size() != 1 || node[v].w != 0) break;
      e = k[0];
      v = e.y;
    }
    order.push_back(v);
    first.push_back(v0);
    via.push_back(chain);
    children.push_back(k);
    for (auto it = k.rbegin(); it != k.rend(); ++it) st.push_back({it->y, *it});
  }
  if (total_label > INT32_MAX) return err = "tree has more than 2^31-1 label tokens", false;
  const size_t N = order.size();
  std::vector<int32_t> id((size_t)n_node, -1);
  for (size_t j = 0; j < N; ++j) id[(size_t)first[j]] = (int32_t)j;  // child entries name a chain's first node
  out.n_nodes = (int32_t)N;
  out.n_labels = (int32_t)total_label;
  out.label_off.assign(N, 0);
  out.label_len.assign(N, 0);
  out.child_begin.assign(N, 0);
  out.child_count.assign(N, 0);
  out.term_count.assign(N, 0);
  out.child_first_tok.assign(N - 1, 0);
  out.child_idx.assign(N - 1, 0);
  out.labels.assign((size_t)total_label, 0);
  int64_t lab = 0, ch = 0;
  for (size_t j = 0; j < N; ++j) {
    const int64_t v = order[j];
    out.label_off[j] = (int32_t)lab;
    if (v != 0) {
      int32_t len = 0;
      for (const int4& ce : via[j]) {
        std::memcpy(out.labels.data() + lab, label_ptr(label, shared, ce.z), (size_t)ce.w * sizeof(int32_t));
        lab += ce.w;
        len += ce.w;
      }
      out.label_len[j] = len;
    }
    const std::vector<int4>& kk = children[j];
    out.child_begin[j] = (int32_t)ch;
    out.child_count[j] = (int32_t)kk.size();
    out.term_count[j] = node[v].w;
    for (const int4& c : kk) {
      out.child_first_tok[(size_t)ch] = c.x;
      out.child_idx[(size_t)ch] = id[(size_t)c.y];
      ++ch;
    }
  }
  return true;
}

}  // namespace p2p

extern "C" {

int p2p_snapshot_build(const p2p_seqs* seqs, p2p_snapshot** out) {
  if (!out) {
    p2p::set_global_error("out is NULL");
    return P2P_E_INVAL;
  }
  *out = nullptr;
  std::string err;
  p2p_snapshot* s = new (std::nothrow) p2p_snapshot();
  if (!s) {
    p2p::set_global_error("out of host memory");
    return P2P_E_NOMEM;
  }
  if (!seqs || !p2p::check_seqs(seqs, err, nullptr, nullptr)) {
    delete s;
    p2p::set_global_error(seqs ? err : "seqs is NULL");
    return P2P_E_INVAL;
  }
  if (!p2p::build_snapshot(*seqs, *s, err)) {
    delete s;
    p2p::set_global_error(err);
    return P2P_E_NOMEM;
  }
  *out = s;
  return P2P_OK;
}

void p2p_snapshot_view(const p2p_snapshot* s, p2p_flat_tree* o) {
  if (!s || !o) return;
  o->n_nodes = s->n_nodes;
  o->n_labels = s->n_labels;
  o->label_off = s->label_off.data();
  o->label_len = s->label_len.data();
  o->child_begin = s->child_begin.data();
  o->child_count = s->child_count.data();
  o->term_count = s->term_count.data();
  o->child_first_tok = s->child_first_tok.data();
  o->child_idx = s->child_idx.data();
  o->labels = s->labels.data();
}

void p2p_snapshot_free(p2p_snapshot* s) { delete s; }

int p2p_flat_tree_validate(const p2p_flat_tree* t) {
  std::string err;
  if (!p2p::validate_flat(t, err)) {
    p2p::set_global_error(err);
    return P2P_E_FORMAT;
  }
  return P2P_OK;
}

}  // extern "C"
