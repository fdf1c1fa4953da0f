// handle.h -- the library's handle (relay_handle of relaysum.h): the visit
// program of the tree, the objective and the settings every launch copies
// into its arguments.  Host memory only; shared by the kernel translation
// unit and the host-state step (host_step.cpp).
#pragma once

#include <cstdint>

#include "program.h"
#include "relaysum.h"

struct relay_handle {
    relaysum::Program prog;
    relaysum::Objective obj;
    int64_t d = 0, ld = 0, nquads = 0, c0 = 0;
    int64_t ld_x = 0, ld_m = 0;  // row strides (floats) of x / mu and of the messages
    int32_t mode = 1;
    const float* mu = nullptr;
    float sigma = 0.0f;
    bool has_objective = false;
    // local optimiser of Alg. 1's local step (appendix "RelaySGD with momentum / Adam")
    int32_t opt = 0;
    float beta1 = 0.0f, beta2 = 0.0f, eps = 0.0f;
    float* s1 = nullptr;  // momentum buffer / Adam first moment, [n][ld_x]
    float* s2 = nullptr;  // Adam second moment, [n][ld_x]
    // algorithm on the relay: 0 RelaySGD (Alg. 1), 1 RelaySum/Grad (Alg. 6), 2 DME (Alg. 5)
    int32_t algo = 0;
    int64_t* dme_count = nullptr;  // algo 2: s_i, device int64 [n]
    // step kernel: RELAY_KERNEL_AUTO / _WALK / _NODES
    int32_t kernel = RELAY_KERNEL_AUTO;
    // messages lost in transit (Section 4.4), one bit per directed edge
    bool has_lost = false;
    // message buffers carry the received sums of the wide nodes (program.h)
    bool rsum = false;
    uint32_t lost[relaysum::kMaxE / 32 + 1] = {};
};
