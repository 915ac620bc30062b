// Rollout-level prefix trees (Sec. 3.2.1, "Prefix Tree Construction"; Sec. 3.2.2,
// "Trajectory Extraction and Filtering"), built on the host and written out as one packed,
// deduplicated token stream for a batch of rollouts: every shared prefix once, harness content
// (tool outputs, environment feedback, the prompt) untrainable, responses trainable, with the
// previous-token link and the depth of every token on its path and the rollout that owns it.
//
// Per rollout (one worker thread per rollout at a time):
//   1. each call (x_i, y_i), in capture order, becomes a node under the node whose accumulated
//      history is the longest prefix of x_i (earliest node on ties). Matching histories are
//      closed under ancestors (a child's history extends its parent's), so a depth-first walk
//      that only enters children whose own tokens continue x_i finds all of them;
//   2. leaves of the whole tree are counted; more than max_leaves (> 0) discards the rollout;
//   3. auxiliary calls leave with their subtrees; the root's children are grouped into
//      segments by equal input; in each segment the leaf with the longest history is kept;
//   4. the kept leaves' ancestors are laid out in depth-first preorder, children in creation
//      order.
// A second pass writes every rollout at its offset of the packed stream.
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <exception>
#include <mutex>
#include <new>
#include <string>
#include <thread>
#include <unordered_map>
#include <vector>

#include "rl_host.h"

namespace rl {
namespace tree {

struct Span {
  const int32_t* p;
  int64_t n;
};

struct Node {
  int32_t parent;
  int32_t call;        // global call index, -1 for the root
  int64_t hist_len;    // accumulated history length
  int64_t inter_len;   // harness tokens at the start of the node
  Span x, y;           // the call's input and response (own tokens: x[parent hist_len:] + y)
  std::vector<int32_t> children;
};

struct Rollout {
  std::vector<Node> nodes;
  std::vector<int32_t> order;      // kept nodes in preorder
  std::vector<int32_t> kept_leaves;
  int32_t n_leaves = 0, n_unplaced = 0;
  bool valid = true;
  int64_t n_tokens = 0, n_trainable = 0;
};

// token k of node n's own tokens
static inline int32_t own_token(const Node& n, int64_t parent_hist, int64_t k) {
  const int64_t xi = parent_hist + k;
  return xi < n.x.n ? n.x.p[xi] : n.y.p[xi - n.x.n];
}

static inline int64_t own_len(const Node& n, int64_t parent_hist) { return n.x.n - parent_hist + n.y.n; }

// Is the accumulated history of `child` a prefix of x, given that its parent's is?
static bool child_matches(const Node& child, int64_t parent_hist, const Span& x) {
  if (child.hist_len > x.n) return false;
  // own tokens are child.x[parent_hist:] then child.y; compare with x[parent_hist:]
  const int64_t nx = child.x.n - parent_hist;
  if (nx > 0 && std::memcmp(child.x.p + parent_hist, x.p + parent_hist, nx * sizeof(int32_t)) != 0) return false;
  if (child.y.n > 0 && std::memcmp(child.y.p, x.p + child.x.n, child.y.n * sizeof(int32_t)) != 0) return false;
  return true;
}

static void build_one(const Span& prompt, int32_t call0, int32_t call1, const int64_t* xo, const int32_t* xt,
                      const int64_t* yo, const int32_t* yt, const uint8_t* aux, int32_t max_leaves, Rollout& R) {
  R.nodes.clear();
  Node root;
  root.parent = -1;
  root.call = -1;
  root.hist_len = prompt.n;
  root.inter_len = prompt.n;
  root.x = prompt;
  root.y = Span{nullptr, 0};
  R.nodes.push_back(root);
  std::vector<int32_t> stack;
  for (int32_t c = call0; c < call1; ++c) {
    const Span x{xt + xo[c], xo[c + 1] - xo[c]};
    const Span y{yt + yo[c], yo[c + 1] - yo[c]};
    if (x.n < prompt.n || (prompt.n > 0 && std::memcmp(x.p, prompt.p, prompt.n * sizeof(int32_t)) != 0)) {
      ++R.n_unplaced;
      continue;
    }
    // longest matching history; earliest node on ties
    int32_t best = 0;
    stack.assign(1, 0);
    while (!stack.empty()) {
      const int32_t n = stack.back();
      stack.pop_back();
      const Node& nd = R.nodes[n];
      if (nd.hist_len > R.nodes[best].hist_len || (nd.hist_len == R.nodes[best].hist_len && n < best)) best = n;
      for (int32_t ch : nd.children)
        if (child_matches(R.nodes[ch], nd.hist_len, x)) stack.push_back(ch);
    }
    Node nn;
    nn.parent = best;
    nn.call = c;
    nn.hist_len = x.n + y.n;
    nn.inter_len = x.n - R.nodes[best].hist_len;
    nn.x = x;
    nn.y = y;
    const int32_t id = static_cast<int32_t>(R.nodes.size());
    R.nodes.push_back(nn);
    R.nodes[best].children.push_back(id);
  }
  const int32_t N = static_cast<int32_t>(R.nodes.size());
  for (int32_t n = 1; n < N; ++n) R.n_leaves += R.nodes[n].children.empty() ? 1 : 0;
  if (max_leaves > 0 && R.n_leaves > max_leaves) {
    R.valid = false;
    return;
  }
  // auxiliary calls leave with their subtrees (parents precede children in creation order)
  std::vector<uint8_t> main(N, 1);
  for (int32_t n = 1; n < N; ++n)
    main[n] = main[R.nodes[n].parent] && !(aux && aux[R.nodes[n].call]);
  // segments: root children grouped by equal input (first such child is the representative)
  std::vector<int32_t> seg(N, -1);
  std::unordered_map<uint64_t, std::vector<int32_t>> by_hash;
  for (int32_t ch : R.nodes[0].children) {
    if (!main[ch]) continue;
    const Span& x = R.nodes[ch].x;
    uint64_t h = 1469598103934665603ull ^ static_cast<uint64_t>(x.n);
    for (int64_t k = 0; k < x.n; ++k) h = (h ^ static_cast<uint32_t>(x.p[k])) * 1099511628211ull;
    int32_t rep = ch;
    for (int32_t other : by_hash[h]) {
      const Span& xo2 = R.nodes[other].x;
      if (xo2.n == x.n && (x.n == 0 || std::memcmp(xo2.p, x.p, x.n * sizeof(int32_t)) == 0)) {
        rep = other;
        break;
      }
    }
    if (rep == ch) by_hash[h].push_back(ch);
    seg[ch] = rep;
  }
  for (int32_t n = 1; n < N; ++n)
    if (R.nodes[n].parent > 0) seg[n] = seg[R.nodes[n].parent];
  // per segment, the main leaf with the longest history (earliest on ties)
  std::unordered_map<int32_t, int32_t> best_leaf;
  std::vector<int32_t> seg_order;
  for (int32_t n = 1; n < N; ++n) {
    if (!main[n]) continue;
    bool leaf = true;
    for (int32_t ch : R.nodes[n].children)
      if (main[ch]) {
        leaf = false;
        break;
      }
    if (!leaf) continue;
    auto it = best_leaf.find(seg[n]);
    if (it == best_leaf.end()) {
      best_leaf[seg[n]] = n;
      seg_order.push_back(seg[n]);
    } else if (R.nodes[n].hist_len > R.nodes[it->second].hist_len) {
      it->second = n;
    }
  }
  std::vector<uint8_t> keep(N, 0), is_kept_leaf(N, 0);
  keep[0] = 1;
  for (int32_t s : seg_order) {
    int32_t n = best_leaf[s];
    is_kept_leaf[n] = 1;
    while (n >= 0 && !keep[n]) {
      keep[n] = 1;
      n = R.nodes[n].parent;
    }
  }
  // preorder over kept nodes, children in creation order
  R.order.clear();
  R.kept_leaves.clear();
  stack.assign(1, 0);
  while (!stack.empty()) {
    const int32_t n = stack.back();
    stack.pop_back();
    R.order.push_back(n);
    if (is_kept_leaf[n]) R.kept_leaves.push_back(n);
    const Node& nd = R.nodes[n];
    const int64_t ph = n ? R.nodes[nd.parent].hist_len : 0;
    const int64_t len = n ? own_len(nd, ph) : nd.x.n;
    R.n_tokens += len;
    R.n_trainable += nd.y.n;
    for (auto it = nd.children.rbegin(); it != nd.children.rend(); ++it)
      if (keep[*it]) stack.push_back(*it);
  }
}

struct Out {
  int32_t* tokens;
  uint8_t* mask;
  int64_t* parent;
  int32_t* depth;
  int32_t* owner;
  int32_t* node_call;
  int32_t* leaf_call;
  int64_t* leaf_end;
};

// Write rollout r's kept nodes at token offset base and leaf offset lbase.
static void emit(const Rollout& R, int32_t r, int64_t base, int64_t lbase, const Out& o) {
  const int32_t N = static_cast<int32_t>(R.nodes.size());
  std::vector<int64_t> path_end(N, -1);
  int64_t pos = base, li = lbase;
  for (int32_t n : R.order) {
    const Node& nd = R.nodes[n];
    const int64_t ph = n ? R.nodes[nd.parent].hist_len : 0;
    const int64_t len = n ? own_len(nd, ph) : nd.x.n;
    const int64_t inter = n ? nd.inter_len : nd.x.n;
    int64_t prev = n ? path_end[nd.parent] : -1;
    for (int64_t k = 0; k < len; ++k, ++pos) {
      o.tokens[pos] = n ? own_token(nd, ph, k) : nd.x.p[k];
      o.mask[pos] = k >= inter ? 1 : 0;
      o.parent[pos] = prev;
      if (o.depth) o.depth[pos] = prev >= 0 ? o.depth[prev] + 1 : 0;
      if (o.owner) o.owner[pos] = r;
      if (o.node_call) o.node_call[pos] = nd.call;
      prev = pos;
    }
    path_end[n] = prev;
    if (o.leaf_call && std::find(R.kept_leaves.begin(), R.kept_leaves.end(), n) != R.kept_leaves.end()) {
      o.leaf_call[li] = nd.call;
      if (o.leaf_end) o.leaf_end[li] = path_end[n];
      ++li;
    }
  }
}

// Runs f(0..n-1) on up to `threads` host threads. An exception in a worker is kept and
// rethrown after every thread has joined; so is a failure to start a thread (the threads
// already started are joined first).
template <class F>
static void parallel_for(int32_t n, int32_t threads, F f) {
  if (threads <= 1 || n <= 1) {
    for (int32_t i = 0; i < n; ++i) f(i);
    return;
  }
  std::mutex mu;
  std::exception_ptr first;
  const int32_t T = std::min(threads, n);
  auto work = [&](int32_t w) {
    try {
      for (int32_t i = w; i < n; i += T) f(i);
    } catch (...) {
      std::lock_guard<std::mutex> lock(mu);
      if (!first) first = std::current_exception();
    }
  };
  std::vector<std::thread> pool;
  try {
    for (int32_t w = 0; w < T; ++w) pool.emplace_back(work, w);
  } catch (...) {
    for (auto& th : pool) th.join();
    throw;
  }
  for (auto& th : pool) th.join();
  if (first) std::rethrow_exception(first);
}

}  // namespace tree
}  // namespace rl

namespace rl {
namespace tree {
static rl_status build_batch(int32_t n_rollouts, const int64_t* prompt_offsets, const int32_t* prompt_tokens,
                             const int32_t* call_offsets, const int64_t* x_offsets, const int32_t* x_tokens,
                             const int64_t* y_offsets, const int32_t* y_tokens, const uint8_t* aux, int32_t max_leaves,
                             int32_t n_threads, int64_t capacity, int32_t* tokens_out, uint8_t* mask_out,
                             int64_t* parent_out, int32_t* depth_out, int32_t* owner_out, int32_t* node_call_out,
                             int32_t* leaf_call_out, int64_t* leaf_end_out, int64_t* leaf_offsets_out,
                             rl_tree_stats* stats_out, int64_t* rollout_offsets_out, int64_t* n_tokens_out);
}  // namespace tree
}  // namespace rl

// C entry point: no C++ exception (an allocation or a thread that cannot be created) may
// cross the C ABI; it becomes an error status instead.
extern "C" rl_status rl_prefix_tree_build_batch(
    int32_t n_rollouts, const int64_t* prompt_offsets, const int32_t* prompt_tokens, const int32_t* call_offsets,
    const int64_t* x_offsets, const int32_t* x_tokens, const int64_t* y_offsets, const int32_t* y_tokens,
    const uint8_t* aux, int32_t max_leaves, int32_t n_threads, int64_t capacity, int32_t* tokens_out,
    uint8_t* mask_out, int64_t* parent_out, int32_t* depth_out, int32_t* owner_out, int32_t* node_call_out,
    int32_t* leaf_call_out, int64_t* leaf_end_out, int64_t* leaf_offsets_out, rl_tree_stats* stats_out,
    int64_t* rollout_offsets_out, int64_t* n_tokens_out) {
  try {
    return rl::tree::build_batch(n_rollouts, prompt_offsets, prompt_tokens, call_offsets, x_offsets, x_tokens,
                                 y_offsets, y_tokens, aux, max_leaves, n_threads, capacity, tokens_out, mask_out,
                                 parent_out, depth_out, owner_out, node_call_out, leaf_call_out, leaf_end_out,
                                 leaf_offsets_out, stats_out, rollout_offsets_out, n_tokens_out);
  } catch (const std::bad_alloc&) {
    return rl::set_error(RL_ERR_UNSUPPORTED, "rl_prefix_tree_build_batch: out of host memory");
  } catch (const std::exception& e) {
    return rl::set_error(RL_ERR_UNSUPPORTED, std::string("rl_prefix_tree_build_batch: ") + e.what());
  } catch (...) {
    return rl::set_error(RL_ERR_UNSUPPORTED, "rl_prefix_tree_build_batch: unexpected host error");
  }
}

static rl_status rl::tree::build_batch(
    int32_t n_rollouts, const int64_t* prompt_offsets, const int32_t* prompt_tokens, const int32_t* call_offsets,
    const int64_t* x_offsets, const int32_t* x_tokens, const int64_t* y_offsets, const int32_t* y_tokens,
    const uint8_t* aux, int32_t max_leaves, int32_t n_threads, int64_t capacity, int32_t* tokens_out,
    uint8_t* mask_out, int64_t* parent_out, int32_t* depth_out, int32_t* owner_out, int32_t* node_call_out,
    int32_t* leaf_call_out, int64_t* leaf_end_out, int64_t* leaf_offsets_out, rl_tree_stats* stats_out,
    int64_t* rollout_offsets_out, int64_t* n_tokens_out) {
  clear_error();
  if (n_rollouts < 0) return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: n_rollouts < 0");
  if (!n_tokens_out) return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: n_tokens_out is NULL");
  *n_tokens_out = 0;
  if (n_rollouts == 0) {
    if (rollout_offsets_out) rollout_offsets_out[0] = 0;
    if (leaf_offsets_out) leaf_offsets_out[0] = 0;
    return RL_OK;
  }
  if (!prompt_offsets || !call_offsets || !x_offsets || !y_offsets)
    return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: NULL offsets");
  // host-side validation of the CSR arrays
  if (call_offsets[0] < 0 || prompt_offsets[0] < 0)
    return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: negative first offset");
  for (int32_t r = 0; r < n_rollouts; ++r) {
    if (call_offsets[r + 1] < call_offsets[r] || prompt_offsets[r + 1] < prompt_offsets[r])
      return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: offsets must be non-decreasing");
  }
  const int32_t n_calls = call_offsets[n_rollouts];
  if (x_offsets[0] < 0 || y_offsets[0] < 0)
    return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: negative first offset");
  for (int32_t c = 0; c < n_calls; ++c)
    if (x_offsets[c + 1] < x_offsets[c] || y_offsets[c + 1] < y_offsets[c])
      return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: offsets must be non-decreasing");
  if ((prompt_offsets[n_rollouts] > 0 && !prompt_tokens) || (x_offsets[n_calls] > 0 && !x_tokens) ||
      (y_offsets[n_calls] > 0 && !y_tokens))
    return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: NULL token array");

  std::vector<Rollout> R(n_rollouts);
  parallel_for(n_rollouts, n_threads, [&](int32_t r) {
    const Span prompt{prompt_tokens ? prompt_tokens + prompt_offsets[r] : nullptr,
                      prompt_offsets[r + 1] - prompt_offsets[r]};
    build_one(prompt, call_offsets[r], call_offsets[r + 1], x_offsets, x_tokens, y_offsets, y_tokens, aux,
              max_leaves, R[r]);
  });
  std::vector<int64_t> base(n_rollouts + 1, 0), lbase(n_rollouts + 1, 0);
  for (int32_t r = 0; r < n_rollouts; ++r) {
    base[r + 1] = base[r] + (R[r].valid ? R[r].n_tokens : 0);
    lbase[r + 1] = lbase[r] + (R[r].valid ? static_cast<int64_t>(R[r].kept_leaves.size()) : 0);
  }
  *n_tokens_out = base[n_rollouts];
  if (stats_out)
    for (int32_t r = 0; r < n_rollouts; ++r) {
      stats_out[r].valid = R[r].valid ? 1 : 0;
      stats_out[r].n_leaves = R[r].n_leaves;
      stats_out[r].n_kept_leaves = R[r].valid ? static_cast<int32_t>(R[r].kept_leaves.size()) : 0;
      stats_out[r].n_unplaced = R[r].n_unplaced;
      stats_out[r].n_tokens = R[r].valid ? R[r].n_tokens : 0;
      stats_out[r].n_trainable = R[r].valid ? R[r].n_trainable : 0;
    }
  if (rollout_offsets_out) std::copy(base.begin(), base.end(), rollout_offsets_out);
  if (leaf_offsets_out) std::copy(lbase.begin(), lbase.end(), leaf_offsets_out);
  if (base[n_rollouts] > capacity)
    return set_error(RL_ERR_WORKSPACE_TOO_SMALL,
                     "rl_prefix_tree_build_batch: capacity below the packed length (see *n_tokens_out)");
  if (base[n_rollouts] > 0 && (!tokens_out || !mask_out || !parent_out))
    return set_error(RL_ERR_INVALID_ARG, "rl_prefix_tree_build_batch: NULL token output");
  const Out o{tokens_out, mask_out, parent_out, depth_out, owner_out, node_call_out, leaf_call_out, leaf_end_out};
  parallel_for(n_rollouts, n_threads, [&](int32_t r) {
    if (R[r].valid) emit(R[r], r, base[r], lbase[r], o);
  });
  return RL_OK;
}
