// internal.h -- device layout of the trees and the kernel launchers shared by the library's sources.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <cstring>
#include <string>
#include <vector>

#include "p2p_router.h"

// Host snapshot object handed out by p2p_snapshot_build / p2p_tree_download (layout of p2p_flat_tree).
struct p2p_snapshot {
  int32_t n_nodes = 0, n_labels = 0;
  std::vector<int32_t> label_off, label_len, child_begin, child_count, term_count, child_first_tok, child_idx, labels;
};

namespace p2p {

// Device layout of one tree (HBM, one allocation per array):
//   node[v]  = {child_begin, child_count, child_cap, term_count}          (int4, 16 B)
//   child[e] = {first_tok, node, label_off, label_len} of one child edge   (int4, 16 B)
//   label[]  = int32 tokens; an edge's label is label[label_off .. +label_len)
// Node 0 is the root.  A node's children occupy child[child_begin .. +child_count), ascending by
// first_tok, inside a reserved range of child_cap entries.  Keeping the child's label position in the
// parent's entry lets a walk start comparing the label as soon as the child search returns.
struct TreeView {
  const int4* node;
  const int4* child;
  const int32_t* label;
};

// Mutable state of one tree, owned by the delta kernel while it runs and mirrored on the host.
struct TreeState {
  int4* node;
  int4* child;
  int32_t* label;
  int32_t n_node, cap_node;    // node slots used (high-water mark) / capacity
  int32_t n_child, cap_child;  // child entries used (bump arena) / capacity
  int32_t n_label, cap_label;  // label tokens used (bump arena) / capacity
  int32_t free_head, n_free;   // free node slots, linked through node[v].x
  int32_t status;              // DELTA_OK, DELTA_NEED_SPACE, DELTA_CORRUPT
  int32_t need_node, need_child, need_label;  // room the first unapplied op needs
  int64_t op_next, op_end;     // ops still to apply: [op_next, op_end)
  int64_t n_absent;            // DELETEs of sequences that were not stored
  int64_t stale_child, stale_label;  // unreachable child entries / label tokens
};

enum { DELTA_OK = 0, DELTA_NEED_SPACE = 1, DELTA_CORRUPT = 2 };

// Bits of the router's device error word.
enum { ERR_BAD_OFFSETS = 1, ERR_CORRUPT_TREE = 2 };

// Route kernel (lookup + route decision), see route_kernel.cu.
cudaError_t launch_route(const TreeView* d_trees, int32_t P, const int32_t* tokens, int64_t n_tokens,
                         int64_t tok_base, const int64_t* offsets, int64_t B, const int32_t* d_load, int32_t alpha,
                         int32_t* out_match, int32_t* out_peer, int32_t* d_err, int num_sms, cudaStream_t st);

// Delta kernel: applies the ops [op_next, op_end) of states[0 .. n_trees) (one warp per tree).
// scratch holds n_trees * scratch_stride tokens (each op's sequence is gathered there).
cudaError_t launch_delta(TreeState* d_states, int32_t n_trees, const int32_t* op, const int64_t* seg_begin,
                         const int64_t* seg_off, const int32_t* seg_len, const int32_t* pool, int32_t* scratch,
                         int64_t scratch_stride, cudaStream_t st);

// Writes a tree's state and view on the device (values passed as kernel parameters, so no host buffer
// has to outlive the call).
cudaError_t launch_set_tree(TreeState* d_state, TreeView* d_view, TreeState value, cudaStream_t st);

// Rewrites views[0 .. n) from states[0 .. n) (after a delta moved some trees' arrays).
cudaError_t launch_refresh_views(const TreeState* d_states, TreeView* d_views, int32_t n, cudaStream_t st);

// Static scratch of the allocation-free delta call (delta_static.cu).
enum { STATIC_BAD_OP = 1, STATIC_BAD_SEGMENT = 2, STATIC_BAD_PEER_BEGIN = 4, STATIC_TOO_LONG = 8 };
int64_t static_scratch_tokens();
cudaError_t static_scratch(int device, int32_t** header, int32_t** tokens);
cudaError_t launch_validate_static(int32_t* header, const p2p_delta* d, int32_t peer, int32_t P, cudaStream_t st);
cudaError_t launch_init_ranges(TreeState* d_states, int32_t nt, const int64_t* peer_begin, int64_t n, cudaStream_t st);

// Host-side helpers in snapshot.cpp.
void set_global_error(const std::string& msg);
const char* global_error();
// Checks a segmented sequence list (ranges only; the pool is not read).  max_len / lens: optional outputs.
bool check_seqs(const p2p_seqs* s, std::string& err, int64_t* max_len, std::vector<int64_t>* lens);
bool build_snapshot(const p2p_seqs& S, p2p_snapshot& out, std::string& err);
bool validate_flat(const p2p_flat_tree* t, std::string& err);
bool snapshot_from_device_layout(const int4* node, int64_t n_node, const int4* child, int64_t n_child,
                                 const int32_t* label, int64_t n_label, p2p_snapshot& out, std::string& err);

}  // namespace p2p
