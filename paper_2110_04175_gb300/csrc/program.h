// program.h -- the visit program that drives the fused RelaySum kernel.
//
// Every coordinate of Algorithm 1 (RelaySGD) is independent, so one GPU
// thread owns a quad of coordinates for ALL workers and walks the tree once
// per step.  The walk is a depth-first pre-order from a chosen root.  At the
// visit of worker i the thread forms x_i^{t+1/2}, reads the D = |N(i)|
// incoming messages m^{t-1}_{k->i}, writes the D outgoing messages
// m^t_{i->k} (each the sum of x_i^{t+1/2} and the OTHER D-1 incoming
// messages), and routes them into the rebuild sums: the message to the DFS
// parent goes straight into the parent's accumulator, a message to a child
// waits in a shared-memory slot until that child is visited.  A worker's
// rebuild finishes at the visit of its last child (or its own, for a leaf).
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

struct NodeRec {        // 16 bytes; indexed by worker id
    int16_t deg;        // D = |N(i)|
    int16_t pos_base;   // first of i's D positions (ascending neighbour id)
    int16_t parent_pos; // position of the DFS parent among i's neighbours; -1 at the root
    int16_t recv_slot;  // slot holding m^t_{parent->i}; -1 at the root
    int16_t acc_slot;   // slot of i's rebuild accumulator; -1 for a leaf
    int16_t parent_acc; // the parent's accumulator slot; -1 at the root
    int16_t fin_parent; // parent id when i is the parent's last child, else -1
    int16_t parent;     // DFS parent id; -1 at the root
};

struct Program {
    int32_t n, E, nslots, root;
    int16_t order[kMaxN];        // DFS pre-order of the workers
    NodeRec node[kMaxN];
    int16_t pos_in[kMaxE];       // position s of i: edge k_s -> i
    int16_t pos_out[kMaxE];      // position s of i: edge i -> k_s
    int16_t pos_slot[kMaxE];     // slot of the message to child k_s (every
                                 // position when D > kRegDeg: suffix-sum scratch)
    int16_t edge_src[kMaxE];     // directed edge e: edge_src[e] -> edge_dst[e]
    int16_t edge_dst[kMaxE];
};

// Status codes mirror relaysum.h.
int build_program(int n, const int32_t* edges, int n_edges, Program* out);

}  // namespace relaysum
