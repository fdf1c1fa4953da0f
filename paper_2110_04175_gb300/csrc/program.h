// program.h -- the visit program that drives the fused RelaySum kernel.
//
// Every coordinate of Algorithm 1 (RelaySGD) is independent, so one GPU
// thread owns a quad of coordinates for ALL workers and walks the tree once
// per step.  The walk is a depth-first pre-order from a chosen root.  At the
// visit of worker i the thread forms x_i^{t+1/2}, reads the D = |N(i)|
// incoming messages m^{t-1}_{k->i} and produces the D outgoing messages
// m^t_{i->k} (each the sum of x_i^{t+1/2} and the OTHER D-1 incoming
// messages), routing them into the rebuild sums: the message to the DFS
// parent goes straight into the parent's accumulator, a message to a child
// waits in a shared-memory slot until that child is visited.  A worker's
// rebuild finishes at the visit of its last child (or its own, for a leaf).
//
// Two ways to form the outgoing messages:
//   - degree <= kRegDeg ("narrow"): the incoming messages stay in registers
//     and message s is a prefix sum plus a suffix sum over the others;
//   - degree > kRegDeg ("wide", e.g. a star's hub): one streaming pass forms
//     the total T_i = x_i^{t+1/2} + sum_k m^{t-1}_{k->i}; only T_i is kept
//     (one slot), and each child c forms its own incoming message as
//     m^t_{i->c} = T_i - m^{t-1}_{c->i} at its visit (re-reading that one
//     message) and writes it out.  This keeps the slots per thread O(1)
//     instead of O(degree).
//
// Received sums (optional, relay_set_received_sums).  The sum a wide node
// needs, S_i^{t-1} = sum_k m^{t-1}_{k->i}, is the sum of received messages
// that Alg. 1's rebuild line formed one step earlier.  With received sums
// on, every message buffer carries one more row per wide node holding it:
// the walk forms T_i = x_i^{t+1/2} + S_i^{t-1} from that one row instead of
// reading all D incoming rows, each child's m^{t-1}_{c->i} is then read
// once (at the child's visit) rather than twice, and S_i^t is summed in one
// more slot (rsum_slot) as the new messages arrive and written to row
// E + rsum_row[i] of the output buffer at the visit of i's last child.
//
// The same program drives the node-parallel kernel for short vectors (one
// thread per worker and quad): it forms each worker's messages with the
// walk's arithmetic and adds the incoming ones in the walk's order (rb_in),
// so both kernels give the same bits.
//
// The program is a plain-old-data struct passed by value as a
// __grid_constant__ kernel parameter (warp-uniform reads from the constant
// bank), so a handle owns no device memory.
#pragma once

#include <cstdint>

namespace relaysum {

constexpr int kMaxN = 256;               // == RELAY_MAX_N
constexpr int kMaxE = 2 * (kMaxN - 1);
constexpr int kRegDeg = 4;               // degrees up to this keep messages in registers

enum NodeFlags : int16_t {
    kRecvFromTotal = 1,  // recv_slot holds the wide parent's total T_p
};

struct NodeRec {        // 20 bytes; indexed by worker id
    int16_t deg;        // D = |N(i)|
    int16_t pos_base;   // first of i's D positions (ascending neighbour id)
    int16_t parent_pos; // position of the DFS parent among i's neighbours; -1 at the root
    int16_t recv_slot;  // slot holding m^t_{parent->i} (or T_parent); -1 at the root
    int16_t acc_slot;   // slot of i's rebuild accumulator; -1 for a leaf
    int16_t parent_acc; // the parent's accumulator slot; -1 at the root
    int16_t fin_parent; // parent id when i is the parent's last child, else -1
    int16_t parent;     // DFS parent id; -1 at the root
    int16_t tot_slot;   // wide node with children: slot of its total T_i; else -1
    int16_t flags;      // NodeFlags
};

struct Program {
    int32_t n, E, nslots, root;
    int16_t order[kMaxN];        // DFS pre-order of the workers
    NodeRec node[kMaxN];
    int16_t pos_in[kMaxE];       // position s of i: edge k_s -> i
    int16_t pos_out[kMaxE];      // position s of i: edge i -> k_s
    int16_t pos_slot[kMaxE];     // narrow node: slot of the message to child k_s; else -1
    int16_t edge_src[kMaxE];     // directed edge e: edge_src[e] -> edge_dst[e]
    int16_t edge_dst[kMaxE];
    int16_t rb_in[kMaxE];        // i's positions: its incoming edges in the walk's rebuild
                                 // order (from the DFS parent, then from the children in
                                 // visit order); the node-parallel kernel adds them so
    // received sums (built only when they are on; else -1): a wide node's
    // slot of its running sum S_i^t, and its row among the sum rows (row
    // E + rsum_row[i] of a message buffer).  int8 keeps two programs within
    // one launch's parameter space.
    int8_t rsum_slot[kMaxN];
    int8_t rsum_row[kMaxN];
    int32_t nwide;               // rows of received sums (0 when they are off)
};

// Where the kernel takes the quadratic centres mu_i from.
constexpr int kMaxMixNnz = 1024;        // non-zero mixture weights in a kernel parameter
constexpr int kMaxCachedCentres = 16;   // centres kept per thread in shared memory

enum ObjectiveSource : int32_t {
    kMuStored = 0,      // read the caller's mu array
    kMuPerRow = 1,      // regenerate: one Philox block per non-zero weight of the row
    kMuCachedCentres = 2,  // regenerate the K centres once per quad, then mix per row
};

struct Objective {
    int32_t source;     // ObjectiveSource
    int32_t K;          // centres
    float scale;        // mu_i = scale * sum_k w_ik N_k
    uint32_t k0, k1;    // Philox key of the centres (stream 1)
    int16_t row_off[kMaxN + 1];   // row i's non-zeros: [row_off[i], row_off[i+1])
    int16_t col[kMaxMixNnz];      // centre index, ascending within a row
    float w[kMaxMixNnz];          // weight
};

// Status codes mirror relaysum.h.  received_sums: lay out the walk for
// received-sum rows (one more slot per wide node).
int build_program(int n, const int32_t* edges, int n_edges, Program* out, bool received_sums = false);

}  // namespace relaysum
