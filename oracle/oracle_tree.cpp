// oracle_tree.cpp -- CPU oracle for the prefix-cache-aware router.
//
// TEST INFRASTRUCTURE.  Only the tests, the package smoke check and the bench's CPU-baseline leg may load
// this library.  It shares no code, header or constant with the CUDA path and is never a fallback for it.
//
// What it computes (all integer, exact):
//   * A radix tree (edge-compressed trie over tokens) per node of the paper's system (Section 2: each node
//     keeps a radix tree of the prefixes it caches and one estimate per peer).  A tree stores a multiset
//     S(T) of token sequences; term counts record multiplicity.
//   * insert  = updateTrie(req) / updateTrieEstimate(req, k) (Section 2 primitive list; Algorithm 1).
//   * remove  = drop one occurrence of a stored sequence (anti-entropy delta, the DELETE half; the
//     structural part of evictLRUTrie in Section 2).
//   * match   = PrefixMatch(r, T) of Algorithm 1: the number of leading tokens of r found along a path
//     of T, counting a partially matched edge.  Because every leaf is terminal this equals
//     max over s in S(T) of LCP(r, s), and 0 for the empty tree.
//   * route   = the argmax over all N trees in Algorithm 1 (getBestNode), extended with a load term:
//     score_p = match_p - alpha * load_p, ties to the lower load, then to the lower tree index.
//   * export  = a canonical flat form (the full-snapshot broadcast of sendTrie, Section 3 "Trie-broadcast
//     loss"): nodes in preorder, children ascending by first token, labels and child lists packed in
//     node order.  Two trees holding the same multiset export identical arrays.
//
// Touched-byte counters follow the accounting used for the roofline: per lookup, 4 bytes per token
// compared (every matched token plus the mismatching one when the walk stops inside an edge with
// request tokens left), 20 bytes per node visited (the root included), and 4*ceil(log2(deg+1)) bytes
// per child search at a node with deg >= 1 children; the route adds 4 bytes per request token.
//
// Plain and slow on purpose: pointer nodes, std::vector labels, sorted std::vector children.
#include <algorithm>
#include <array>
#include <cstdint>
#include <cstring>
#include <thread>
#include <unordered_map>
#include <vector>

namespace {

struct Node {
  std::vector<int32_t> label;  // edge label from the parent (empty only for the root)
  int64_t term = 0;            // number of stored sequences that end exactly here
  std::vector<Node*> kids;     // sorted ascending by kid->label[0]
};

struct Tree {
  Node* root;
  Tree() : root(new Node()) {}
  ~Tree() {
    std::vector<Node*> st{root};
    while (!st.empty()) {
      Node* n = st.back();
      st.pop_back();
      for (Node* k : n->kids) st.push_back(k);
      delete n;
    }
  }
};

// Position of the child whose label starts with `tok`, or of the slot where it would be inserted.
std::vector<Node*>::iterator child_slot(Node* n, int32_t tok) {
  return std::lower_bound(n->kids.begin(), n->kids.end(), tok,
                          [](const Node* k, int32_t t) { return k->label[0] < t; });
}
Node* find_child(const Node* n, int32_t tok) {
  auto it = std::lower_bound(n->kids.begin(), n->kids.end(), tok,
                             [](const Node* k, int32_t t) { return k->label[0] < t; });
  if (it != n->kids.end() && (*it)->label[0] == tok) return *it;
  return nullptr;
}

void insert(Tree& t, const int32_t* s, int64_t n) {
  Node* cur = t.root;
  int64_t i = 0;
  for (;;) {
    if (i == n) {
      cur->term += 1;
      return;
    }
    auto it = child_slot(cur, s[i]);
    if (it == cur->kids.end() || (*it)->label[0] != s[i]) {
      Node* leaf = new Node();
      leaf->label.assign(s + i, s + n);
      leaf->term = 1;
      cur->kids.insert(it, leaf);
      return;
    }
    Node* c = *it;
    const int64_t L = (int64_t)c->label.size();
    int64_t k = 0;
    while (k < L && i + k < n && c->label[(size_t)k] == s[i + k]) ++k;
    if (k == L) {
      cur = c;
      i += k;
      continue;
    }
    // The sequence leaves the edge after k tokens (1 <= k < L): split the edge there.
    Node* mid = new Node();
    mid->label.assign(c->label.begin(), c->label.begin() + k);
    c->label.erase(c->label.begin(), c->label.begin() + k);
    mid->kids.push_back(c);
    *it = mid;
    i += k;
    if (i == n) {
      mid->term = 1;
      return;
    }
    Node* leaf = new Node();
    leaf->label.assign(s + i, s + n);
    leaf->term = 1;
    mid->kids.insert(child_slot(mid, leaf->label[0]), leaf);
    return;
  }
}

// x has exactly one child y and no sequence ends at x: fold y's edge into x's.
void merge_with_only_child(Node* x) {
  Node* y = x->kids[0];
  x->label.insert(x->label.end(), y->label.begin(), y->label.end());
  x->term = y->term;
  x->kids = std::move(y->kids);
  y->kids.clear();
  delete y;
}

// Removes one occurrence of s.  Returns 1 if removed, 0 if s was not stored.
int remove(Tree& t, const int32_t* s, int64_t n) {
  std::vector<Node*> path{t.root};
  Node* cur = t.root;
  int64_t i = 0;
  while (i < n) {
    Node* c = find_child(cur, s[i]);
    if (!c) return 0;
    const int64_t L = (int64_t)c->label.size();
    if (i + L > n) return 0;
    for (int64_t k = 0; k < L; ++k)
      if (c->label[(size_t)k] != s[i + k]) return 0;
    i += L;
    cur = c;
    path.push_back(c);
  }
  if (cur->term == 0) return 0;
  cur->term -= 1;
  if (cur == t.root || cur->term > 0) return 1;
  Node* parent = path[path.size() - 2];
  if (cur->kids.empty()) {
    parent->kids.erase(child_slot(parent, cur->label[0]));
    delete cur;
    if (parent != t.root && parent->term == 0 && parent->kids.size() == 1) merge_with_only_child(parent);
  } else if (cur->kids.size() == 1) {
    merge_with_only_child(cur);
  }
  return 1;
}

int64_t ceil_log2_plus1(int64_t deg) {  // ceil(log2(deg + 1)), deg >= 1
  int64_t b = 0;
  while (((int64_t)1 << b) < deg + 1) ++b;
  return b;
}

// counters: [0] tokens compared, [1] nodes visited, [2] child-search bytes.
int64_t match(const Tree& t, const int32_t* r, int64_t n, int64_t* ctr) {
  const Node* cur = t.root;
  int64_t i = 0, compared = 0, visited = 1, search = 0;
  for (;;) {
    if (i == n) break;
    const int64_t deg = (int64_t)cur->kids.size();
    if (deg == 0) break;
    search += 4 * ceil_log2_plus1(deg);
    const Node* c = find_child(cur, r[i]);
    if (!c) break;
    visited += 1;
    const int64_t L = (int64_t)c->label.size();
    int64_t k = 0;
    while (k < L && i + k < n && c->label[(size_t)k] == r[i + k]) ++k;
    compared += k;
    if (k < L && i + k < n) compared += 1;
    i += k;
    if (k < L) break;
    cur = c;
  }
  if (ctr) {
    ctr[0] += compared;
    ctr[1] += visited;
    ctr[2] += search;
  }
  return i;
}

// Route decision for one request: lexicographic max of (match - alpha*load, -load, -p).
int32_t argmax_peer(int32_t P, const int32_t* m, const int32_t* load, int32_t alpha) {
  int32_t best = 0;
  for (int32_t p = 1; p < P; ++p) {
    const int64_t sp = (int64_t)m[p] - (int64_t)alpha * load[p];
    const int64_t sb = (int64_t)m[best] - (int64_t)alpha * load[best];
    if (sp > sb || (sp == sb && (load[p] < load[best] || (load[p] == load[best] && p < best)))) best = p;
  }
  return best;
}

void preorder(const Tree& t, std::vector<const Node*>& out) {
  std::vector<const Node*> st{t.root};
  while (!st.empty()) {
    const Node* n = st.back();
    st.pop_back();
    out.push_back(n);
    for (auto it = n->kids.rbegin(); it != n->kids.rend(); ++it) st.push_back(*it);
  }
}

std::vector<int32_t> gather(const int64_t* seg_begin, const int64_t* seg_off, const int32_t* seg_len,
                            const int32_t* pool, int64_t i) {
  std::vector<int32_t> s;
  for (int64_t g = seg_begin[i]; g < seg_begin[i + 1]; ++g)
    s.insert(s.end(), pool + seg_off[g], pool + seg_off[g] + seg_len[g]);
  return s;
}

}  // namespace

extern "C" {

typedef struct otree otree;

otree* otree_new(void) { return reinterpret_cast<otree*>(new Tree()); }
void otree_free(otree* t) { delete reinterpret_cast<Tree*>(t); }

void otree_insert(otree* t, const int32_t* s, int64_t n) { insert(*reinterpret_cast<Tree*>(t), s, n); }
int otree_remove(otree* t, const int32_t* s, int64_t n) { return remove(*reinterpret_cast<Tree*>(t), s, n); }

int64_t otree_match(const otree* t, const int32_t* r, int64_t n, int64_t* counters) {
  return match(*reinterpret_cast<const Tree*>(t), r, n, counters);
}

// Inserts sequences [i0, i1) of a segmented list (sequence i = concatenation of its pool runs).
void otree_insert_segmented(otree* t, const int64_t* seg_begin, const int64_t* seg_off, const int32_t* seg_len,
                            const int32_t* pool, int64_t i0, int64_t i1) {
  Tree& T = *reinterpret_cast<Tree*>(t);
  for (int64_t i = i0; i < i1; ++i) {
    const std::vector<int32_t> s = gather(seg_begin, seg_off, seg_len, pool, i);
    insert(T, s.data(), (int64_t)s.size());
  }
}

// Applies ops [i0, i1) in order (0 = INSERT, 1 = DELETE); returns the number of DELETEs of absent sequences.
int64_t otree_apply_ops(otree* t, const int32_t* op, const int64_t* seg_begin, const int64_t* seg_off,
                        const int32_t* seg_len, const int32_t* pool, int64_t i0, int64_t i1) {
  Tree& T = *reinterpret_cast<Tree*>(t);
  int64_t absent = 0;
  for (int64_t i = i0; i < i1; ++i) {
    const std::vector<int32_t> s = gather(seg_begin, seg_off, seg_len, pool, i);
    if (op[i] == 0)
      insert(T, s.data(), (int64_t)s.size());
    else if (remove(T, s.data(), (int64_t)s.size()) == 0)
      ++absent;
  }
  return absent;
}

// As otree_apply_ops, with the touched-byte counters of an anti-entropy delta: before each op, the read-only
// PrefixMatch walk of its sequence adds to ctr[0..2] (tokens compared, nodes visited, child-search bytes,
// as for a lookup); then ctr[3] += sequence tokens, ctr[4] += pool runs, ctr[5] += INSERTs, ctr[6] += label
// tokens an INSERT adds (sequence length - match), ctr[7] += DELETEs.
int64_t otree_apply_ops_counted(otree* t, const int32_t* op, const int64_t* seg_begin, const int64_t* seg_off,
                                const int32_t* seg_len, const int32_t* pool, int64_t i0, int64_t i1, int64_t* ctr) {
  Tree& T = *reinterpret_cast<Tree*>(t);
  int64_t absent = 0;
  for (int64_t i = i0; i < i1; ++i) {
    const std::vector<int32_t> s = gather(seg_begin, seg_off, seg_len, pool, i);
    const int64_t n = (int64_t)s.size();
    const int64_t m = match(T, s.data(), n, ctr);
    ctr[3] += n;
    ctr[4] += seg_begin[i + 1] - seg_begin[i];
    if (op[i] == 0) {
      ctr[5] += 1;
      ctr[6] += n - m;
      insert(T, s.data(), n);
    } else {
      ctr[7] += 1;
      if (remove(T, s.data(), n) == 0) ++absent;
    }
  }
  return absent;
}

// out[0] = nodes (root included), out[1] = label tokens, out[2] = stored sequences (sum of term counts).
void otree_stats(const otree* t, int64_t* out) {
  std::vector<const Node*> nodes;
  preorder(*reinterpret_cast<const Tree*>(t), nodes);
  int64_t lab = 0, seqs = 0;
  for (const Node* n : nodes) {
    lab += (int64_t)n->label.size();
    seqs += n->term;
  }
  out[0] = (int64_t)nodes.size();
  out[1] = lab;
  out[2] = seqs;
}

// Canonical flat export; arrays sized from otree_stats (child arrays hold nodes-1 entries).
// Returns 0, or -1 if a count does not fit int32.
int otree_export(const otree* t, int32_t* label_off, int32_t* label_len, int32_t* child_begin, int32_t* child_count,
                 int32_t* term_count, int32_t* child_first_tok, int32_t* child_idx, int32_t* labels) {
  std::vector<const Node*> nodes;
  preorder(*reinterpret_cast<const Tree*>(t), nodes);
  std::unordered_map<const Node*, int64_t> id;
  for (size_t i = 0; i < nodes.size(); ++i) id[nodes[i]] = (int64_t)i;
  int64_t lab = 0, ch = 0;
  for (size_t i = 0; i < nodes.size(); ++i) {
    const Node* n = nodes[i];
    if (n->term > INT32_MAX || lab > INT32_MAX || ch > INT32_MAX) return -1;
    label_off[i] = (int32_t)lab;
    label_len[i] = (int32_t)n->label.size();
    if (!n->label.empty()) std::memcpy(labels + lab, n->label.data(), n->label.size() * sizeof(int32_t));
    lab += (int64_t)n->label.size();
    child_begin[i] = (int32_t)ch;
    child_count[i] = (int32_t)n->kids.size();
    term_count[i] = (int32_t)n->term;
    for (const Node* k : n->kids) {
      child_first_tok[ch] = k->label[0];
      child_idx[ch] = (int32_t)id[k];
      ++ch;
    }
  }
  return 0;
}

int32_t oracle_argmax(int32_t P, const int32_t* match_row, const int32_t* load, int32_t alpha) {
  return argmax_peer(P, match_row, load, alpha);
}

// Routes requests [0, B): out_match[b*P + p] = PrefixMatch(r_b, T_p), out_peer[b] = the route decision.
// counters (nullable) receive [tokens compared, nodes visited, child-search bytes, request tokens].
void oracle_route(const otree* const* trees, int32_t P, const int32_t* tokens, const int64_t* offsets, int64_t B,
                  const int32_t* load, int32_t alpha, int32_t* out_match, int32_t* out_peer, int32_t n_threads,
                  int64_t* counters) {
  int64_t nt = n_threads < 1 ? 1 : n_threads;
  if (nt > B) nt = B < 1 ? 1 : B;
  std::vector<std::array<int64_t, 4>> part((size_t)nt, std::array<int64_t, 4>{0, 0, 0, 0});
  auto work = [&](int64_t ti) {
    const int64_t b0 = B * ti / nt, b1 = B * (ti + 1) / nt;
    int64_t* c = part[(size_t)ti].data();
    for (int64_t b = b0; b < b1; ++b) {
      const int32_t* r = tokens + offsets[b];
      const int64_t n = offsets[b + 1] - offsets[b];
      int32_t* row = out_match + b * P;
      for (int32_t p = 0; p < P; ++p)
        row[p] = (int32_t)match(*reinterpret_cast<const Tree*>(trees[p]), r, n, c);
      out_peer[b] = argmax_peer(P, row, load, alpha);
      c[3] += n;
    }
  };
  if (nt == 1) {
    work(0);
  } else {
    std::vector<std::thread> th;
    for (int64_t i = 0; i < nt; ++i) th.emplace_back(work, i);
    for (auto& x : th) x.join();
  }
  if (counters) {
    for (int j = 0; j < 4; ++j) counters[j] = 0;
    for (auto& c : part)
      for (int j = 0; j < 4; ++j) counters[j] += c[(size_t)j];
  }
}

}  // extern "C"
