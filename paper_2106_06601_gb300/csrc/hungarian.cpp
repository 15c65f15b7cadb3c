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
