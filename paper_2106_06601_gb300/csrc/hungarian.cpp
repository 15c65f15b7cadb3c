// Exact linear assignment for the process relabeling (Thm. 1 / Thm. 2,
// Sec. 4): the Hungarian method (Kuhn 1955; Munkres 1957) in its O(n^3)
// shortest-augmenting-path form.
//
// Rows are inserted one at a time.  Each insertion grows a Dijkstra-like
// search over columns under the reduced costs c[i][j] - u[i] - v[j] >= 0,
// updating the potentials (u, v) so that the edges of the matching stay
// tight, until it reaches a free column; the matching is then flipped along
// the alternating path.  After n insertions the matching is a minimum-cost
// perfect assignment and (u, v) is a feasible dual solution whose objective
// equals its cost (LP duality, the certificate of optimality).
#include <algorithm>
#include <cstdint>
#include <limits>
#include <vector>

namespace costa {

// cost: row-major n x n (integer or floating-point weights).  row_to_col[i]
// receives the column assigned to row i.
// Returns the minimum total cost.  u (n rows) and v (n columns) receive the
// dual potentials when non-null: u[i] + v[j] <= cost[i][j] for all (i, j),
// with equality on the assignment.
template <typename W>
W assign_min_t(int n, const std::vector<W> &cost, std::vector<int> &row_to_col, std::vector<W> *u_out,
               std::vector<W> *v_out) {
    const W INF = std::numeric_limits<W>::max() / 4;
    // 1-based internally; column 0 is a virtual source column.
    std::vector<W> u(n + 1, 0), v(n + 1, 0), dist(n + 1);
    std::vector<int> col_row(n + 1, 0), prev(n + 1, 0);
    std::vector<char> done(n + 1);
    for (int i = 1; i <= n; ++i) {
        col_row[0] = i;
        int j0 = 0;
        std::fill(dist.begin(), dist.end(), INF);
        std::fill(done.begin(), done.end(), 0);
        do {
            done[j0] = 1;
            const int i0 = col_row[j0];
            W delta = INF;
            int j1 = 0;
            const W *crow = cost.data() + static_cast<size_t>(i0 - 1) * n;
            for (int j = 1; j <= n; ++j) {
                if (done[j]) continue;
                const W red = crow[j - 1] - u[i0] - v[j];
                if (red < dist[j]) {
                    dist[j] = red;
                    prev[j] = j0;
                }
                if (dist[j] < delta) {
                    delta = dist[j];
                    j1 = j;
                }
            }
            for (int j = 0; j <= n; ++j) {
                if (done[j]) {
                    u[col_row[j]] += delta;
                    v[j] -= delta;
                } else {
                    dist[j] -= delta;
                }
            }
            j0 = j1;
        } while (col_row[j0] != 0);
        do {  // flip the alternating path back to the source column
            const int j1 = prev[j0];
            col_row[j0] = col_row[j1];
            j0 = j1;
        } while (j0 != 0);
    }
    row_to_col.assign(n, -1);
    W total = 0;
    for (int j = 1; j <= n; ++j) {
        row_to_col[col_row[j] - 1] = j - 1;
        total += cost[static_cast<size_t>(col_row[j] - 1) * n + (j - 1)];
    }
    if (u_out) u_out->assign(u.begin() + 1, u.end());
    if (v_out) v_out->assign(v.begin() + 1, v.end());
    return total;
}

int64_t assign_min(int n, const std::vector<int64_t> &cost, std::vector<int> &row_to_col,
                   std::vector<int64_t> *u_out, std::vector<int64_t> *v_out) {
    return assign_min_t<int64_t>(n, cost, row_to_col, u_out, v_out);
}

double assign_min_f(int n, const std::vector<double> &cost, std::vector<int> &row_to_col) {
    return assign_min_t<double>(n, cost, row_to_col, nullptr, nullptr);
}

}  // namespace costa

namespace costa {

// Greedy maximum-weight matching (Sec. 6: "a simple greedy algorithm, which
// is a 2-approximation"): pairs (p, q) by decreasing V[p][q], ties broken by
// smaller p then smaller q; a pair is kept when p and q are both unmatched.
// Target labels left unmatched take the unmatched processes, both in
// increasing order.  sigma[q] = p.  Returns sum_q V[sigma[q]][q].
int64_t greedy_max(int P, const int64_t *V, std::vector<int> &sigma) {
    const int64_t n = static_cast<int64_t>(P) * P;
    std::vector<int64_t> order(static_cast<size_t>(n));
    for (int64_t k = 0; k < n; ++k) order[static_cast<size_t>(k)] = k;
    std::stable_sort(order.begin(), order.end(), [V](int64_t a, int64_t b) { return V[a] > V[b]; });
    std::vector<char> used_p(P, 0), used_q(P, 0);
    sigma.assign(P, -1);
    for (int64_t k : order) {
        const int p = static_cast<int>(k / P), q = static_cast<int>(k % P);
        if (used_p[p] || used_q[q]) continue;
        used_p[p] = used_q[q] = 1;
        sigma[q] = p;
    }
    int next = 0;
    for (int q = 0; q < P; ++q) {
        if (sigma[q] >= 0) continue;
        while (used_p[next]) ++next;
        sigma[q] = next;
        used_p[next] = 1;
    }
    int64_t total = 0;
    for (int q = 0; q < P; ++q) total += V[static_cast<int64_t>(sigma[q]) * P + q];
    return total;
}

}  // namespace costa

#include <queue>

namespace costa {

// Exact maximum of sum_q V[sigma[q]][q] over permutations for a sparse V
// (Thm. 1 objective), by successive shortest augmenting paths (Dijkstra with
// potentials) on the bipartite graph of the nonzero entries.  Each target
// row q may also take a private "unmatched" column at weight 0; at the end
// the rows left unmatched take the unused processes in increasing order,
// which adds nothing to the objective (their V entries on the remaining
// pairs are whatever they are; see below).  Work per row is a Dijkstra over
// the rows and nonzero edges its search reaches, instead of the dense
// method's O(P^2) scan.
//
// Why the completion is optimal: a maximum-weight matching that may leave
// rows unmatched is at least as heavy as any permutation's objective
// restricted to nonzero entries, which is the permutation's objective; and
// completing it cannot lower its weight (V >= 0).  The returned objective is
// recomputed on the completed permutation.
int64_t assign_max_sparse(int P, const int64_t *V, std::vector<int> &sigma) {
    // adjacency by row q: (p, weight V[p][q] > 0)
    std::vector<int> start(static_cast<size_t>(P) + 1, 0);
    for (int p = 0; p < P; ++p)
        for (int q = 0; q < P; ++q)
            if (V[static_cast<size_t>(p) * P + q] > 0) ++start[q + 1];
    for (int q = 0; q < P; ++q) start[q + 1] += start[q];
    std::vector<int> col(static_cast<size_t>(start[P]));
    std::vector<int64_t> w(static_cast<size_t>(start[P]));
    {
        std::vector<int> fill(start.begin(), start.end() - 1);
        for (int p = 0; p < P; ++p)
            for (int q = 0; q < P; ++q) {
                const int64_t v = V[static_cast<size_t>(p) * P + q];
                if (v > 0) {
                    col[fill[q]] = p;
                    w[fill[q]++] = v;
                }
            }
    }
    // columns 0..P-1 are processes; column P + q is row q's private
    // "unmatched" column.  Costs: -V for real edges, 0 for the private one.
    const int NC = 2 * P;
    const int64_t INF = std::numeric_limits<int64_t>::max() / 4;
    std::vector<int64_t> u(P, 0), v(NC, 0);  // potentials: cost - u - v >= 0
    for (int q = 0; q < P; ++q) {
        int64_t m = 0;
        for (int e = start[q]; e < start[q + 1]; ++e) m = std::min(m, -w[e]);
        u[q] = m;
    }
    std::vector<int> col_row(NC, -1), row_col(P, -1);
    std::vector<int64_t> dist(NC, INF);
    std::vector<int> prev_row(NC, -1), touched;
    std::vector<char> done(NC, 0);
    typedef std::pair<int64_t, int> Item;  // (distance, column)
    for (int s = 0; s < P; ++s) {
        std::priority_queue<Item, std::vector<Item>, std::greater<Item>> pq;
        touched.clear();
        auto relax_row = [&](int r, int64_t dr) {  // dr: distance at row r
            for (int e = start[r]; e < start[r + 1]; ++e) {
                const int c = col[e];
                const int64_t nd = dr + (-w[e] - u[r] - v[c]);
                if (nd < dist[c]) {
                    if (dist[c] == INF) touched.push_back(c);
                    dist[c] = nd;
                    prev_row[c] = r;
                    pq.push({nd, c});
                }
            }
            const int c = P + r;  // the private column
            const int64_t nd = dr + (0 - u[r] - v[c]);
            if (nd < dist[c]) {
                if (dist[c] == INF) touched.push_back(c);
                dist[c] = nd;
                prev_row[c] = r;
                pq.push({nd, c});
            }
        };
        relax_row(s, 0);
        int end_col = -1;
        int64_t end_dist = 0;
        std::vector<int> done_cols;
        while (!pq.empty()) {
            const Item it = pq.top();
            pq.pop();
            const int c = it.second;
            if (done[c] || it.first != dist[c]) continue;
            done[c] = 1;
            done_cols.push_back(c);
            if (col_row[c] < 0) {
                end_col = c;
                end_dist = it.first;
                break;
            }
            relax_row(col_row[c], it.first);
        }
        // potentials: keep reduced costs non-negative for the next search
        u[s] += end_dist;
        for (int c : done_cols) {
            if (c == end_col) continue;
            const int r = col_row[c];
            v[c] -= end_dist - dist[c];
            u[r] += end_dist - dist[c];
        }
        // augment along prev_row back to s
        for (int c = end_col; c >= 0;) {
            const int r = prev_row[c];
            const int next = row_col[r];
            col_row[c] = r;
            row_col[r] = c;
            c = (r == s) ? -1 : next;
        }
        for (int c : touched) {
            dist[c] = INF;
            done[c] = 0;
            prev_row[c] = -1;
        }
    }
    // complete: rows on their private column take the unused processes
    sigma.assign(P, -1);
    std::vector<char> used(P, 0);
    for (int q = 0; q < P; ++q)
        if (row_col[q] >= 0 && row_col[q] < P) {
            sigma[q] = row_col[q];
            used[row_col[q]] = 1;
        }
    int next = 0;
    for (int q = 0; q < P; ++q) {
        if (sigma[q] >= 0) continue;
        while (used[next]) ++next;
        sigma[q] = next;
        used[next] = 1;
    }
    int64_t total = 0;
    for (int q = 0; q < P; ++q) total += V[static_cast<size_t>(sigma[q]) * P + q];
    return total;
}

}  // namespace costa
