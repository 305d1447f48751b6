// Algorithm 2 (Sec. III): optimal chunk ordering for a delta-regular
// assignment with N == m, by delta successive perfect matchings of the
// bipartite graph of A (Claim 1).  Host code; one-time set-up.
#include <string.h>

#include <vector>

#include "gc_internal.cuh"

namespace gc {
namespace {

// Perfect matching of rows to columns in the graph adj (adjacency lists,
// columns ascending), by augmenting paths (Kuhn): rows in increasing order,
// a depth-first search over alternating paths that tries each row's columns
// in increasing order.  match_row[i] = column of row i.  Returns false if
// some row stays unmatched.
bool perfect_matching(const std::vector<std::vector<int>>& adj, int m, std::vector<int>& match_row) {
  std::vector<int> match_col(m, -1), seen(m, -1), prev_row(m, -1);
  match_row.assign(m, -1);
  std::vector<std::pair<int, int>> stack;  // (row, index of its next column)
  for (int r0 = 0; r0 < m; ++r0) {
    stack.clear();
    stack.push_back({r0, 0});
    int free_col = -1;
    while (!stack.empty()) {
      const int r = stack.back().first;
      const int k = stack.back().second;
      if (k >= (int)adj[r].size()) {
        stack.pop_back();
        continue;
      }
      stack.back().second = k + 1;
      const int c = adj[r][k];
      if (seen[c] == r0) continue;
      seen[c] = r0;
      prev_row[c] = r;
      if (match_col[c] < 0) {
        free_col = c;
        break;
      }
      stack.push_back({match_col[c], 0});
    }
    if (free_col < 0) return false;
    // flip the alternating path r0 -> c1 -> r1 -> ... -> free_col
    int c = free_col;
    while (true) {
      const int r = prev_row[c];
      const int old = match_row[r];
      match_row[r] = c;
      match_col[c] = r;
      if (r == r0) break;
      c = old;
    }
  }
  return true;
}

}  // namespace
}  // namespace gc

using namespace gc;

extern "C" int gc_chunk_ordering(const uint8_t* A_h, int N, int m, int delta, int32_t* order_h,
                                 uint8_t* O_h) {
  if (!A_h) return fail(GC_ERR_ARG, "A_h is NULL");
  if (N < 1 || m < 1 || delta < 1) return fail(GC_ERR_SHAPE, "N, m, delta must be >= 1");
  if (N != m) return fail(GC_ERR_SHAPE, "Algorithm 2 needs N == m (N=%d, m=%d)", N, m);
  if (delta > GC_MAX_DELTA) return fail(GC_ERR_UNSUPPORTED, "delta=%d exceeds %d", delta, GC_MAX_DELTA);
  if (delta > 255) return fail(GC_ERR_UNSUPPORTED, "delta=%d does not fit O's uint8", delta);
  std::vector<std::vector<int>> adj(N);
  std::vector<int> colsum(m, 0);
  for (int i = 0; i < N; ++i) {
    for (int j = 0; j < m; ++j)
      if (A_h[(size_t)i * m + j]) {
        adj[i].push_back(j);
        ++colsum[j];
      }
    if ((int)adj[i].size() != delta)
      return fail(GC_ERR_SHAPE, "row %d of A has %d non-zeros, not delta=%d", i, (int)adj[i].size(), delta);
  }
  for (int j = 0; j < m; ++j)
    if (colsum[j] != delta)
      return fail(GC_ERR_SHAPE, "column %d of A has %d non-zeros, not delta=%d", j, colsum[j], delta);
  std::vector<uint8_t> O((size_t)N * m, 0);
  std::vector<int> match;
  for (int p = 1; p <= delta; ++p) {
    if (!perfect_matching(adj, m, match))
      return fail(GC_ERR_DATA, "no perfect matching at level %d (A not regular?)", p);
    for (int i = 0; i < N; ++i) {
      const int j = match[i];
      O[(size_t)i * m + j] = (uint8_t)p;
      // remove the matched edge (lists stay sorted)
      auto& a = adj[i];
      for (size_t k = 0; k < a.size(); ++k)
        if (a[k] == j) {
          a.erase(a.begin() + (long)k);
          break;
        }
    }
  }
  if (O_h) memcpy(O_h, O.data(), O.size());
  if (order_h) {
    for (size_t k = 0; k < (size_t)m * delta; ++k) order_h[k] = -1;
    for (int i = 0; i < N; ++i)
      for (int j = 0; j < m; ++j) {
        const int p = O[(size_t)i * m + j];
        if (p) order_h[(size_t)j * delta + (p - 1)] = i;
      }
  }
  return GC_OK;
}
