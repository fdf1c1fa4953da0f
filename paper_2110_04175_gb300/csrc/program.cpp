// program.cpp -- tree validation and the visit program of the fused kernel.
//
// The method needs a tree (Algorithm 1 runs on a tree network; Section 3
// "Setup": undirected links without self loops).  This file checks that,
// numbers the directed edges (2u: edges[u][0] -> edges[u][1], 2u+1: the
// reverse), sorts every worker's neighbours by id, and then lays out the
// depth-first walk described in program.h so that it needs as few
// shared-memory slots per thread as possible:
//   - children are ordered so that the costliest subtree comes last (a
//     parent's slots die at its last child's visit, so that subtree runs
//     almost free) and the others in decreasing need (fewer sibling messages
//     wait while a large subtree is walked);
//   - every worker is tried as the root and the cheapest walk is kept.
#include "program.h"

#include <algorithm>
#include <cstring>
#include <functional>
#include <queue>
#include <vector>

#include "relaysum.h"

namespace relaysum {
namespace {

struct Tree {
    int n = 0;
    std::vector<std::vector<int>> nbr;      // ascending neighbour ids
    std::vector<std::vector<int>> in_edge;  // edge nbr[i][s] -> i
    std::vector<std::vector<int>> out_edge; // edge i -> nbr[i][s]
};

int validate(int n, const int32_t* edges, int n_edges, Tree* t, Program* p) {
    if (n < 1) return RELAY_EINVAL;
    if (n > kMaxN) return RELAY_EUNSUPPORTED;
    if (n_edges != n - 1) return RELAY_ENOTTREE;
    if (n_edges > 0 && edges == nullptr) return RELAY_EINVAL;
    t->n = n;
    t->nbr.assign(n, {});
    for (int u = 0; u < n_edges; ++u) {
        const int a = edges[2 * u], b = edges[2 * u + 1];
        if (a < 0 || b < 0 || a >= n || b >= n || a == b) return RELAY_ENOTTREE;
        p->edge_src[2 * u] = static_cast<int16_t>(a);
        p->edge_dst[2 * u] = static_cast<int16_t>(b);
        p->edge_src[2 * u + 1] = static_cast<int16_t>(b);
        p->edge_dst[2 * u + 1] = static_cast<int16_t>(a);
        t->nbr[a].push_back(b);
        t->nbr[b].push_back(a);
    }
    for (auto& l : t->nbr) {
        std::sort(l.begin(), l.end());
        if (std::adjacent_find(l.begin(), l.end()) != l.end()) return RELAY_ENOTTREE;
    }
    // n - 1 distinct edges + connected <=> tree
    std::vector<char> seen(n, 0);
    std::vector<int> stack{0};
    seen[0] = 1;
    int reached = 1;
    while (!stack.empty()) {
        const int i = stack.back();
        stack.pop_back();
        for (int j : t->nbr[i])
            if (!seen[j]) {
                seen[j] = 1;
                ++reached;
                stack.push_back(j);
            }
    }
    if (reached != n) return RELAY_ENOTTREE;
    // edge numbers per neighbour position
    const int E = 2 * n_edges;
    t->in_edge.assign(n, {});
    t->out_edge.assign(n, {});
    for (int i = 0; i < n; ++i) {
        t->in_edge[i].resize(t->nbr[i].size());
        t->out_edge[i].resize(t->nbr[i].size());
    }
    for (int e = 0; e < E; ++e) {
        const int a = p->edge_src[e], b = p->edge_dst[e];
        const auto& la = t->nbr[a];
        const auto& lb = t->nbr[b];
        const int sa = static_cast<int>(std::lower_bound(la.begin(), la.end(), b) - la.begin());
        const int sb = static_cast<int>(std::lower_bound(lb.begin(), lb.end(), a) - lb.begin());
        t->out_edge[a][sa] = e;  // a -> b leaves a towards position sa
        t->in_edge[b][sb] = e;   // and arrives at b from position sb
    }
    return RELAY_OK;
}

// A walk from one root: parent, children in visit order, pre-order.
struct Walk {
    std::vector<int> parent, order;
    std::vector<std::vector<int>> children;
};

Walk make_walk(const Tree& t, int root, bool received_sums) {
    const int n = t.n;
    Walk w;
    w.parent.assign(n, -1);
    w.children.assign(n, {});
    // BFS to orient the tree, then need() bottom-up in reverse BFS order.
    std::vector<int> bfs{root};
    std::vector<char> seen(n, 0);
    seen[root] = 1;
    for (size_t q = 0; q < bfs.size(); ++q) {
        const int i = bfs[q];
        for (int j : t.nbr[i])
            if (!seen[j]) {
                seen[j] = 1;
                w.parent[j] = i;
                w.children[i].push_back(j);
                bfs.push_back(j);
            }
    }
    // need[i]: peak slots live during i's visit and its subtree, counting i's
    // incoming slot.  A parent's accumulator (and a wide parent's total) dies
    // at the end of its LAST child's visit, and no sibling message is pending
    // then, so the last child's subtree runs almost free: the best order puts
    // the costliest child last and the others in decreasing need.  Every
    // child is tried as the last one.
    std::vector<int> need(n, 0), vpeak(n, 0);
    for (int q = n - 1; q >= 0; --q) {
        const int i = bfs[q];
        auto& ch = w.children[i];
        const int m = static_cast<int>(ch.size());
        const int D = static_cast<int>(t.nbr[i].size());
        const bool wide = D > kRegDeg;
        const int has_parent = w.parent[i] >= 0 ? 1 : 0;
        // accumulator (+ total, + received sum)
        const int own = (m > 0) ? (wide ? (received_sums ? 3 : 2) : 1) : 0;
        vpeak[i] = std::max(has_parent, own + (wide ? 0 : m));     // slots at i's own visit
        std::stable_sort(ch.begin(), ch.end(), [&](int a, int b) { return need[a] > need[b]; });
        auto peak_of = [&](const std::vector<int>& order) {
            int peak = vpeak[i];
            for (int k = 0; k < m; ++k) {
                const int c = order[k];
                const int pending = wide ? 0 : (m - 1 - k);        // messages to later children
                const int shared = wide ? 1 : 0;                   // a wide parent's total is c's input
                if (k < m - 1) {
                    peak = std::max(peak, own + pending + need[c] - shared);
                } else {  // last child: i's slots live only through c's own visit
                    peak = std::max(peak, own + vpeak[c] - shared);
                    peak = std::max(peak, need[c]);
                }
            }
            return peak;
        };
        int best = peak_of(ch);
        std::vector<int> best_order = ch;
        for (int last = 0; last < m; ++last) {
            std::vector<int> order;
            for (int k = 0; k < m; ++k)
                if (k != last) order.push_back(ch[k]);
            order.push_back(ch[last]);
            const int p = peak_of(order);
            if (p < best) {
                best = p;
                best_order = order;
            }
        }
        ch = best_order;
        need[i] = std::max(best, 1);
    }
    // pre-order
    std::vector<int> stack{root};
    while (!stack.empty()) {
        const int i = stack.back();
        stack.pop_back();
        w.order.push_back(i);
        const auto& ch = w.children[i];
        for (auto it = ch.rbegin(); it != ch.rend(); ++it) stack.push_back(*it);
    }
    return w;
}

// Assigns slots along the walk (lowest free id first) and fills the
// program; returns the number of slots used.
int assign_slots(const Tree& t, const Walk& w, int root, bool received_sums, Program* p) {
    const int n = t.n;
    std::priority_queue<int, std::vector<int>, std::greater<int>> free_ids;
    int next_id = 0;
    auto alloc = [&]() {
        if (!free_ids.empty()) {
            const int s = free_ids.top();
            free_ids.pop();
            return s;
        }
        return next_id++;
    };
    auto release = [&](int s) {
        if (s >= 0) free_ids.push(s);
    };
    std::vector<int> recv(n, -1), acc(n, -1), tot(n, -1), rsum(n, -1), pos_base(n, 0);
    int base = 0;
    for (int i = 0; i < n; ++i) {
        pos_base[i] = base;
        base += static_cast<int>(t.nbr[i].size());
    }
    for (int v = 0; v < n; ++v) {
        const int i = w.order[v];
        const int par = w.parent[i];
        const int D = static_cast<int>(t.nbr[i].size());
        const int m = static_cast<int>(w.children[i].size());
        const bool wide = D > kRegDeg;
        const bool par_wide = par >= 0 && static_cast<int>(t.nbr[par].size()) > kRegDeg;
        // a message slot is read at the start of the visit and freed; a
        // wide parent's total stays live until its last child
        if (!par_wide) release(recv[i]);
        acc[i] = (m > 0) ? alloc() : -1;
        tot[i] = (wide && m > 0) ? alloc() : -1;
        rsum[i] = (wide && m > 0 && received_sums) ? alloc() : -1;
        p->rsum_slot[i] = static_cast<int8_t>(rsum[i]);
        int parent_pos = -1;
        for (int s = 0; s < D; ++s) {
            const int k = t.nbr[i][s];
            const int pos = pos_base[i] + s;
            p->pos_in[pos] = static_cast<int16_t>(t.in_edge[i][s]);
            p->pos_out[pos] = static_cast<int16_t>(t.out_edge[i][s]);
            if (k == par) parent_pos = s;
            int slot = -1;
            if (k != par) {
                if (wide) {
                    recv[k] = tot[i];
                } else {
                    slot = alloc();
                    recv[k] = slot;
                }
            }
            p->pos_slot[pos] = static_cast<int16_t>(slot);
        }
        NodeRec& r = p->node[i];
        r.deg = static_cast<int16_t>(D);
        r.pos_base = static_cast<int16_t>(pos_base[i]);
        r.parent_pos = static_cast<int16_t>(parent_pos);
        r.recv_slot = static_cast<int16_t>(recv[i]);
        r.acc_slot = static_cast<int16_t>(acc[i]);
        r.parent_acc = static_cast<int16_t>(par >= 0 ? acc[par] : -1);
        const bool last = par >= 0 && w.children[par].back() == i;
        r.fin_parent = static_cast<int16_t>(last ? par : -1);
        r.parent = static_cast<int16_t>(par);
        r.tot_slot = static_cast<int16_t>(tot[i]);
        r.flags = static_cast<int16_t>(par_wide ? kRecvFromTotal : 0);
        if (last) {
            release(acc[par]);
            release(tot[par]);
            release(rsum[par]);
        }
        p->order[v] = static_cast<int16_t>(i);
    }
    // rebuild order of every worker's incoming messages: the walk adds the
    // DFS parent's message at the worker's visit, then each child's at the
    // child's visit
    auto in_from = [&](int i, int k) {
        const auto& l = t.nbr[i];
        return t.in_edge[i][std::lower_bound(l.begin(), l.end(), k) - l.begin()];
    };
    for (int i = 0; i < n; ++i) {
        int k = pos_base[i];
        if (w.parent[i] >= 0) p->rb_in[k++] = static_cast<int16_t>(in_from(i, w.parent[i]));
        for (int c : w.children[i]) p->rb_in[k++] = static_cast<int16_t>(in_from(i, c));
    }
    (void)root;
    return next_id;
}

}  // namespace

int build_program(int n, const int32_t* edges, int n_edges, Program* out, bool received_sums) {
    std::memset(out, 0, sizeof(Program));
    Tree t;
    const int rc = validate(n, edges, n_edges, &t, out);
    if (rc != RELAY_OK) return rc;
    out->n = n;
    out->E = 2 * (n - 1);
    // rows of received sums: the wide nodes in ascending id
    std::memset(out->rsum_row, -1, sizeof(out->rsum_row));
    std::memset(out->rsum_slot, -1, sizeof(out->rsum_slot));
    out->nwide = 0;
    if (received_sums)
        for (int i = 0; i < n; ++i)
            if (static_cast<int>(t.nbr[i].size()) > kRegDeg) out->rsum_row[i] = static_cast<int8_t>(out->nwide++);
    int best_root = 0, best_slots = -1;
    Program trial;
    for (int r = 0; r < n; ++r) {
        std::memcpy(&trial, out, sizeof(Program));
        const Walk w = make_walk(t, r, received_sums);
        const int s = assign_slots(t, w, r, received_sums, &trial);
        if (best_slots < 0 || s < best_slots) {
            best_slots = s;
            best_root = r;
        }
    }
    const Walk w = make_walk(t, best_root, received_sums);
    out->nslots = assign_slots(t, w, best_root, received_sums, out);
    out->root = best_root;
    // a received-sum slot must fit its int8 field
    if (received_sums && out->nwide > 0 && out->nslots > 127) return RELAY_EUNSUPPORTED;
    return RELAY_OK;
}

}  // namespace relaysum
