// relaysum.cu -- GB300 (sm_103a) kernels and C ABI of the RelaySum step.
//
// Vogels et al., "RelaySum for Decentralized Deep Learning on Heterogeneous
// Data" (arXiv 2110.04175), Algorithm 1 (RelaySGD) with the robust rebuild of
// Section 4.4, local momentum / Adam, lost messages, and the appendix's
// RelaySum/Grad and mean-estimation algorithms on the same relay, for n
// virtual workers on one GPU.  See relaysum.h for the equations and the ABI
// contract, program.h for the visit program.
//
// Kernels:
//   relay_counts_kernel   Alg. 1 counters, int32, one CTA, in place (lost
//                         messages count 0; mean estimation's counts s_i).
//   relay_models_kernel   everything per coordinate, in ONE pass over d:
//                         local step (SGD / Nesterov / Adam) with Philox noise,
//                         every outgoing relay message, every rebuild.  Each
//                         x_i, mu_i and incoming message quad is read from HBM
//                         once and each outgoing message / new model quad
//                         written once (a child of a node of degree > 4
//                         re-reads the one message it sent that node, see
//                         program.h).  The path is bandwidth-bound streaming
//                         arithmetic: no tensor cores.
//   relay_nodes_kernel    the same step for short vectors, one thread per
//                         (worker, quad) with the new messages exchanged in
//                         shared memory; same bits as relay_models_kernel.
//   relay_init_kernel     x^0 (shared Philox draw) and zeroed messages.
//   relay_fill_mu_kernel  mu_i = scale * sum_k mix[i][k] N_k.
//   relay_metrics_kernel  consensus distance and distance to the optimum,
//   (+ _finish_kernel)    two fixed-order passes in double.
#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <new>

#include "handle.h"
#include "program.h"
#include "relaysum.h"

using relaysum::kMaxE;
using relaysum::kMaxN;
using relaysum::kRegDeg;
using relaysum::NodeRec;
using relaysum::Objective;
using relaysum::Program;


namespace {

// ------------------------------------------------------------ random numbers

// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11): round multipliers and
// Weyl key increments of the published definition.
constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

// The ten round keys (k0 + r W0, k1 + r W1), computed once on the host.
struct PhiloxKey {
    uint32_t k[10][2];
};

PhiloxKey philox_key(uint64_t seed) {
    PhiloxKey key;
    uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
    for (int r = 0; r < 10; ++r) {
        key.k[r][0] = k0;
        key.k[r][1] = k1;
        k0 += kPhiloxW0;
        k1 += kPhiloxW1;
    }
    return key;
}

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, const PhiloxKey& key) {
#pragma unroll
    for (int round = 0; round < 10; ++round) {
        const uint32_t hi0 = __umulhi(kPhiloxM0, c.x), lo0 = kPhiloxM0 * c.x;
        const uint32_t hi1 = __umulhi(kPhiloxM1, c.z), lo1 = kPhiloxM1 * c.z;
        c = make_uint4(hi1 ^ c.y ^ key.k[round][0], lo1, hi0 ^ c.w ^ key.k[round][1], lo0);
    }
    return c;
}

// 24 high bits -> (0, 1], exact in fp32.
__device__ __forceinline__ float unit_interval(uint32_t w) {
    return __uint2float_rn((w >> 8) + 1u) * 5.9604644775390625e-8f;  // 2^-24
}

__device__ __forceinline__ float sqrt_approx(float v) {
    float r;
    asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(v));
    return r;
}

// Four standard normals for coordinates 4q .. 4q+3 (Box-Muller on the two
// word pairs of one Philox block): z = sqrt(-2 ln u_a) (cos, sin)(2 pi u_b).
// The angle is taken as 2 pi u_b - pi, inside the range where the hardware
// sine/cosine are accurate to 2^-21.4, and the half turn is undone by the
// sign; the radius keeps an accurate logarithm (its argument can sit just
// below 1, where an approximate one loses all relative accuracy).
__device__ __forceinline__ float4 normal4(uint32_t q, uint32_t row, uint32_t step, uint32_t stream,
                                          const PhiloxKey& key) {
    const uint4 w = philox4x32_10(make_uint4(q, row, step, stream), key);
    const float r0 = sqrt_approx(-2.0f * logf(unit_interval(w.x)));
    const float r1 = sqrt_approx(-2.0f * logf(unit_interval(w.z)));
    constexpr float kTwoPi = 6.28318530717958647692f, kPi = 3.14159265358979323846f;
    float s0, c0, s1, c1;
    __sincosf(fmaf(unit_interval(w.y), kTwoPi, -kPi), &s0, &c0);
    __sincosf(fmaf(unit_interval(w.w), kTwoPi, -kPi), &s1, &c1);
    return make_float4(-r0 * c0, -r0 * s0, -r1 * c1, -r1 * s1);
}

// ------------------------------------------------------------ float4 helpers

__device__ __forceinline__ float4 add4(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float4 sub4(float4 a, float4 b) {
    return make_float4(a.x - b.x, a.y - b.y, a.z - b.z, a.w - b.w);
}
__device__ __forceinline__ float4 scale4(float4 a, float s) {
    return make_float4(a.x * s, a.y * s, a.z * s, a.w * s);
}
// Rounded product that the compiler may not fuse into a later add: the
// regenerated mu must round exactly like the stored one.
__device__ __forceinline__ float4 scale4_rn(float4 a, float s) {
    return make_float4(__fmul_rn(a.x, s), __fmul_rn(a.y, s), __fmul_rn(a.z, s), __fmul_rn(a.w, s));
}
__device__ __forceinline__ float4 fma4(float w, float4 z, float4 acc) {
    return make_float4(fmaf(w, z.x, acc.x), fmaf(w, z.y, acc.y), fmaf(w, z.z, acc.z), fmaf(w, z.w, acc.w));
}
// Loads read once per step: read-only path, no L1 allocation.
__device__ __forceinline__ float4 ld_stream(const float* p) {
    float4 v;
    asm("ld.global.nc.L1::no_allocate.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "l"(p));
    return v;
}
// A wide node's incoming messages are read again at its children's visits
// (program.h): keep them in L2 with evict-last priority until then.
__device__ __forceinline__ float4 ld_keep(const float* p) {
    float4 v;
    asm("{\n\t.reg .b64 pol;\n\t"
        "createpolicy.fractional.L2::evict_last.b64 pol, 1.0;\n\t"
        "ld.global.nc.L2::cache_hint.v4.f32 {%0, %1, %2, %3}, [%4], pol;\n\t}"
        : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
        : "l"(p));
    return v;
}
__device__ __forceinline__ void st_stream(float* p, float4 v) {
    __stcs(reinterpret_cast<float4*>(p), v);
}

// ------------------------------------------------- programmatic dependent launch

// relay_step launches the step kernel as a programmatic dependent of the
// counter kernel: the counter kernel lets it be scheduled at once, and the
// step kernel waits for the counter kernel's completion (and its writes)
// before its first read of the counters.  Launched the ordinary way, the
// wait returns immediately.
__device__ __forceinline__ void allow_dependent_launch() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void wait_for_prior_grid() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// ------------------------------------------------------------------ counters

// c^t_{i->j} = 1 + sum_{k in N(i)\j} c^{t-1}_{k->i}: the incoming edge from
// j is e ^ 1 for e = i -> j.  A lost message (Section 4.4) arrives as c = 0.
// For distributed mean estimation (Alg. 5) it also adds each worker's
// models-received count 1 + sum_j c^t_{j->i} to the running count s_i.
struct LostMask {
    uint32_t w[relaysum::kMaxE / 32 + 1];
    __host__ __device__ __forceinline__ bool operator()(int e) const { return (w[e >> 5] >> (e & 31)) & 1u; }
};

// c^t of directed edge e from c^{t-1}; a lost message carries no count.
__device__ __forceinline__ int32_t next_count(const Program& prog, const LostMask& lost, int has_lost,
                                              const int32_t* c_old, int e) {
    const NodeRec r = prog.node[prog.edge_src[e]];
    int32_t s = 1;
    for (int p = 0; p < r.deg; ++p) {
        const int in = prog.pos_in[r.pos_base + p];
        if (in != (e ^ 1)) s += c_old[in];
    }
    return (has_lost && lost(e)) ? 0 : s;
}

// The counters of NT handles (the tree windows of relay_step_windows, or one
// handle): CTA w updates window w's.
template <int NT>
struct CountWindows {
    Program prog[NT];
    LostMask lost[NT];
    int32_t has_lost[NT];
    int32_t* counts[NT];
    int64_t* dme_count[NT];  // Alg. 5's counts s_i, or null
};

template <int NT>
__global__ void relay_counts_kernel(const __grid_constant__ CountWindows<NT> cw) {
    allow_dependent_launch();
    __shared__ int32_t c_old[kMaxE];
    const int w = (NT == 1) ? 0 : static_cast<int>(blockIdx.x);
    const Program& prog = cw.prog[w];
    const LostMask& lost = cw.lost[w];
    const int has_lost = cw.has_lost[w];
    int32_t* const counts = cw.counts[w];
    int64_t* const dme_count = cw.dme_count[w];
    const int E = prog.E;
    for (int e = threadIdx.x; e < E; e += blockDim.x) c_old[e] = counts[e];
    __syncthreads();
    for (int e = threadIdx.x; e < E; e += blockDim.x) counts[e] = next_count(prog, lost, has_lost, c_old, e);
    if (dme_count) {  // Alg. 5: s_i += 1 + sum_j c^t_{j->i}
        __syncthreads();
        for (int i = threadIdx.x; i < prog.n; i += blockDim.x) {
            const NodeRec r = prog.node[i];
            int64_t nb = 1;
            for (int p = 0; p < r.deg; ++p) nb += counts[prog.pos_in[r.pos_base + p]];
            dme_count[i] += nb;
        }
    }
}

// The counters (and the mean-estimation counts) advanced by k steps, for
// relay_steps: one CTA of kCountsThreads >= n threads (thread i carries
// worker i's mean-estimation count), the counters of the two step parities
// in shared memory, one barrier per step.
constexpr int kCountsThreads = 256;
static_assert(kMaxN <= kCountsThreads, "relay_counts_steps_kernel gives each worker its own thread");

__global__ void __launch_bounds__(kCountsThreads)
relay_counts_steps_kernel(const __grid_constant__ Program prog,
                                          const __grid_constant__ LostMask lost, int has_lost, int32_t* counts,
                                          int64_t* dme_count, int k) {
    __shared__ int32_t c[2][kMaxE];
    const int E = prog.E;
    for (int e = threadIdx.x; e < E; e += blockDim.x) c[1][e] = counts[e];
    __syncthreads();
    int64_t received = 0;  // worker threadIdx.x: sum over the k steps of 1 + sum_j c^t_{j->i}
    for (int j = 0; j < k; ++j) {
        const int32_t* c_old = c[(j + 1) & 1];
        int32_t* c_new = c[j & 1];
        for (int e = threadIdx.x; e < E; e += blockDim.x) c_new[e] = next_count(prog, lost, has_lost, c_old, e);
        __syncthreads();
        if (dme_count && threadIdx.x < prog.n) {
            const NodeRec r = prog.node[threadIdx.x];
            int64_t nb = 1;
            for (int p = 0; p < r.deg; ++p) nb += c_new[prog.pos_in[r.pos_base + p]];
            received += nb;
        }
    }
    for (int e = threadIdx.x; e < E; e += blockDim.x) counts[e] = c[(k - 1) & 1][e];
    if (dme_count && threadIdx.x < prog.n) dme_count[threadIdx.x] += received;
}

// --------------------------------------------------------------- fused step

struct ModelArgs {
    float* x;
    const float* mu;
    const float* msg_in;
    float* msg_out;
    const int32_t* counts;
    int64_t ld_x;     // row stride (floats) of x and mu
    int64_t ld_m;     // row stride (floats) of the messages
    int64_t nquads;   // ceil(d / 4)
    uint32_t q0;      // absolute quad of local coordinate 0
    uint32_t step;
    float lr, sigma;
    int mode;         // 0: Alg. 1 rebuild, 1: robust rebuild
    int algo;         // 0 RelaySGD, 1 RelaySum/Grad, 2 mean estimation
    int has_lost;     // any bit of `lost` set
    int rsum;         // wide nodes read and write their received-sum rows (program.h)
    LostMask lost;    // messages lost in transit this step
    float* s1;        // optimiser state (momentum / Adam m), [n][ld_x]
    float* s2;        // Adam v, [n][ld_x]
    float beta1, beta2, eps;
    float adam_step;  // lr / (1 - beta1^{t+1})
    float adam_ibc2;  // 1 / sqrt(1 - beta2^{t+1})
    PhiloxKey key;    // noise key schedule
};

// A lost message reaches its receiver as zero (Section 4.4).
__device__ __forceinline__ float4 delivered(const ModelArgs& a, int e, float4 m) {
    return (a.has_lost && a.lost(e)) ? make_float4(0.f, 0.f, 0.f, 0.f) : m;
}

// Per-thread view of the shared-memory slots: slot s of this thread is
// base[s * stride]; a warp's 32 float4 of one slot are contiguous.
struct Slots {
    float4* base;
    int stride;
    __device__ __forceinline__ float4& operator[](int s) const { return base[s * stride]; }
};

// Row of wide node i's received sum in a message buffer (program.h).
__device__ __forceinline__ int64_t rsum_row(const Program& prog, int i) { return prog.E + prog.rsum_row[i]; }

// The message to the DFS parent joins the parent's accumulator (and, with
// received sums, a wide parent's running sum S_p^t); if this worker is the
// parent's last child, the parent's rebuild (and S_p^t) is complete.  WIDE:
// the tree has a node of degree > kRegDeg (the walk's wide-node paths are
// compiled only then).
template <bool WIDE>
__device__ __forceinline__ void to_parent(const Program& prog, const NodeRec& r, const ModelArgs& a, int64_t q,
                                          float4 out, const Slots& sl, const float* s_scale) {
    const float4 acc = add4(sl[r.parent_acc], out);
    if (r.fin_parent >= 0) {
        st_stream(a.x + r.fin_parent * a.ld_x + 4 * q, scale4(acc, s_scale[r.fin_parent]));
    } else {
        sl[r.parent_acc] = acc;
    }
    if (WIDE && a.rsum && (r.flags & relaysum::kRecvFromTotal)) {
        const int rs = prog.rsum_slot[r.parent];
        const float4 sum = add4(sl[rs], out);
        if (r.fin_parent >= 0) {
            st_stream(a.msg_out + rsum_row(prog, r.parent) * a.ld_m + 4 * q, sum);
        } else {
            sl[rs] = sum;
        }
    }
}

// Degree D <= kRegDeg: the D incoming messages live in registers; outgoing
// message s is prefix(s) + suffix(s+1) with prefix(s) = xh + m_0 + ... + m_{s-1}.
template <int D, bool WIDE>
__device__ __forceinline__ void visit_small(const Program& prog, const NodeRec& r, const ModelArgs& a,
                                            int64_t q, float4 xh, const Slots& sl,
                                            const float* s_scale) {
    float4 m[D];
#pragma unroll
    for (int s = 0; s < D; ++s) m[s] = ld_stream(a.msg_in + prog.pos_in[r.pos_base + s] * a.ld_m + 4 * q);
    float4 pre[D];
    pre[0] = xh;
#pragma unroll
    for (int s = 1; s < D; ++s) pre[s] = add4(pre[s - 1], m[s - 1]);
    float4 suf[D];
    suf[D - 1] = m[D - 1];
#pragma unroll
    for (int s = D - 2; s >= 0; --s) suf[s] = add4(m[s], suf[s + 1]);
#pragma unroll
    for (int s = 0; s < D; ++s) {
        const int e = prog.pos_out[r.pos_base + s];
        const float4 out = delivered(a, e, (s == D - 1) ? pre[s] : add4(pre[s], suf[s + 1]));
        st_stream(a.msg_out + e * a.ld_m + 4 * q, out);
        if (s == r.parent_pos) {
            to_parent<WIDE>(prog, r, a, q, out, sl, s_scale);
        } else {
            sl[prog.pos_slot[r.pos_base + s]] = out;
        }
    }
}

// Degree D > kRegDeg: T = xh + the sum of all incoming messages; the message
// to the parent is T minus the parent's incoming message, and T stays in a
// slot for the children (see program.h).  Without received sums one
// streaming pass reads the D incoming rows, over descending positions while
// the children are visited in ascending order, so the first children
// re-read the most recently read (L2-resident) rows.  With received sums,
// T = xh + S_i^{t-1} from the one sum row, and only the parent's incoming
// row is read here.
__device__ __noinline__ void visit_wide(const Program& prog, const NodeRec& r, const ModelArgs& a, int i,
                                        int64_t q, float4 xh, const Slots& sl,
                                        const float* s_scale) {
    const int D = r.deg;
    const int base = r.pos_base;
    float4 total = xh;
    float4 from_parent = make_float4(0.f, 0.f, 0.f, 0.f);
    if (a.rsum) {
        total = add4(xh, ld_stream(a.msg_in + rsum_row(prog, i) * a.ld_m + 4 * q));
        if (r.parent_pos >= 0) from_parent = ld_stream(a.msg_in + prog.pos_in[base + r.parent_pos] * a.ld_m + 4 * q);
    } else {
        for (int s = D - 1; s >= 0; --s) {
            const float4 m = ld_keep(a.msg_in + prog.pos_in[base + s] * a.ld_m + 4 * q);
            total = add4(total, m);
            if (s == r.parent_pos) from_parent = m;
        }
    }
    if (r.parent_pos >= 0) {
        const int e = prog.pos_out[base + r.parent_pos];
        const float4 out = delivered(a, e, sub4(total, from_parent));
        st_stream(a.msg_out + e * a.ld_m + 4 * q, out);
        to_parent<true>(prog, r, a, q, out, sl, s_scale);
    }
    sl[r.tot_slot] = total;
}

// The local optimiser's update u (Alg. 1's local step is x^{t+1/2} = x + u):
//   SGD:      u = -lr g
//   Nesterov: m = beta1 m + g;  u = -lr (g + beta1 m)          (state s1 = m)
//   Adam:     m = beta1 m + (1 - beta1) g;  v = beta2 v + (1 - beta2) g^2;
//             u = -adam_step m / (sqrt(v) adam_ibc2 + eps)     (s1 = m, s2 = v)
// The rule on the optimiser state (m, v) held in registers; adam_step and
// adam_ibc2 are the factors of this step.
template <int OPT>
__device__ __forceinline__ float4 update_rule(const ModelArgs& a, float adam_step, float adam_ibc2, float4 g,
                                              float4& m, float4& v) {
    if (OPT == 0) return scale4(g, -a.lr);
    if (OPT == 1) {
        m = make_float4(fmaf(a.beta1, m.x, g.x), fmaf(a.beta1, m.y, g.y), fmaf(a.beta1, m.z, g.z),
                        fmaf(a.beta1, m.w, g.w));
        return make_float4(-a.lr * fmaf(a.beta1, m.x, g.x), -a.lr * fmaf(a.beta1, m.y, g.y),
                           -a.lr * fmaf(a.beta1, m.z, g.z), -a.lr * fmaf(a.beta1, m.w, g.w));
    }
    const float c1 = 1.0f - a.beta1, c2 = 1.0f - a.beta2;
    m = make_float4(fmaf(a.beta1, m.x, c1 * g.x), fmaf(a.beta1, m.y, c1 * g.y), fmaf(a.beta1, m.z, c1 * g.z),
                    fmaf(a.beta1, m.w, c1 * g.w));
    v = make_float4(fmaf(a.beta2, v.x, c2 * g.x * g.x), fmaf(a.beta2, v.y, c2 * g.y * g.y),
                    fmaf(a.beta2, v.z, c2 * g.z * g.z), fmaf(a.beta2, v.w, c2 * g.w * g.w));
    auto upd = [&](float mm, float vv) { return -adam_step * mm / fmaf(sqrtf(vv), adam_ibc2, a.eps); };
    return make_float4(upd(m.x, v.x), upd(m.y, v.y), upd(m.z, v.z), upd(m.w, v.w));
}

// One step's update with the state read from and written back to HBM.
template <int OPT>
__device__ __forceinline__ float4 local_update(const ModelArgs& a, int i, int64_t q, float4 g) {
    float4 m = make_float4(0.f, 0.f, 0.f, 0.f), v = m;
    if (OPT == 0) return update_rule<OPT>(a, a.adam_step, a.adam_ibc2, g, m, v);
    float4* pm = reinterpret_cast<float4*>(a.s1 + i * a.ld_x + 4 * q);
    float4* pv = reinterpret_cast<float4*>(a.s2 + i * a.ld_x + 4 * q);
    m = *pm;
    if (OPT == 2) v = *pv;
    const float4 u = update_rule<OPT>(a, a.adam_step, a.adam_ibc2, g, m, v);
    __stcs(pm, m);
    if (OPT == 2) __stcs(pv, v);
    return u;
}

// mu_i for quad q: read, or regenerated exactly as relay_fill_mu_kernel
// writes it (same normals, same fma order), so both sources give the same bits.
template <int OBJ>
__device__ __forceinline__ float4 centre(const Objective& obj, const PhiloxKey& mu_key, const ModelArgs& a,
                                         int i, int64_t q, const float4* cen, int cen_stride) {
    if (OBJ == relaysum::kMuStored) return ld_stream(a.mu + i * a.ld_x + 4 * q);
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int j = obj.row_off[i]; j < obj.row_off[i + 1]; ++j) {
        const float4 z = (OBJ == relaysum::kMuPerRow)
                             ? normal4(a.q0 + static_cast<uint32_t>(q), static_cast<uint32_t>(obj.col[j]),
                                       0u, 1u, mu_key)
                             : cen[obj.col[j] * cen_stride];
        acc = fma4(obj.w[j], z, acc);
    }
    return scale4_rn(acc, obj.scale);
}

// Per-worker rebuild factors from this step's counters: x' = scale * acc
// with acc = fill * x + x^{t+1/2} + incoming messages.
//   mode 0: x' = acc / nbar (Alg. 1).  mode 1: x' = (acc + (n - nbar) x) / n
//   (robust rule), the fill term folded into the accumulator up front.
__device__ __forceinline__ void worker_factors(const ModelArgs& a, int n, int nbar, float& scale, float& fill) {
    if (a.algo == 1) {  // x' = x + (u + sum m) / n
        scale = 1.0f / static_cast<float>(n);
        fill = static_cast<float>(n);
    } else if (a.algo == 2) {  // y' = y + dhat + sum m
        scale = 1.0f;
        fill = 1.0f;
    } else if (a.mode == 0) {
        scale = 1.0f / static_cast<float>(nbar);
        fill = 0.0f;
    } else {
        scale = 1.0f / static_cast<float>(n);
        fill = static_cast<float>(n - nbar);
    }
}

__device__ __forceinline__ void rebuild_factors(const Program& prog, const ModelArgs& a, float* s_scale,
                                                float* s_fill) {
    const int n = prog.n;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        const NodeRec r = prog.node[i];
        int nbar = 1;
        for (int p = 0; p < r.deg; ++p) nbar += __ldg(a.counts + prog.pos_in[r.pos_base + p]);
        worker_factors(a, n, nbar, s_scale[i], s_fill[i]);
    }
}

// The relayed value of worker i at quad q: x^{t+1/2} = x + u (Alg. 1), the
// update u (Alg. 6) or the sample mu + sigma xi (Alg. 5), with
// g = (x - mu) + sigma xi and z the worker's noise normals.
// `update` maps g to u (and advances the optimiser state).
template <typename Update>
__device__ __forceinline__ float4 relayed_with(const ModelArgs& a, float4 xv, float4 mv, float4 z,
                                               Update update) {
    if (a.algo == 2)
        return make_float4(fmaf(a.sigma, z.x, mv.x), fmaf(a.sigma, z.y, mv.y), fmaf(a.sigma, z.z, mv.z),
                           fmaf(a.sigma, z.w, mv.w));
    const float4 g = make_float4(fmaf(a.sigma, z.x, xv.x - mv.x), fmaf(a.sigma, z.y, xv.y - mv.y),
                                 fmaf(a.sigma, z.z, xv.z - mv.z), fmaf(a.sigma, z.w, xv.w - mv.w));
    const float4 u = update(g);
    return (a.algo == 1) ? u : add4(xv, u);
}

template <int OPT>
__device__ __forceinline__ float4 relayed_value(const ModelArgs& a, int i, int64_t q, float4 xv, float4 mv,
                                                float4 z) {
    return relayed_with(a, xv, mv, z, [&](float4 g) { return local_update<OPT>(a, i, q, g); });
}

// The step of NT handles in one launch: one handle, or the tree windows of
// relay_step_windows (the double binary trees of Section 3: two trees over
// the same workers, each carrying its own columns of the models).  The
// grid's first `split` CTAs work on window 0, the rest on window 1.
template <int NT>
struct Windows {
    Program prog[NT];
    ModelArgs a[NT];
    int32_t split;
};

// The walk over one window's quads: CTA `cta` of `ctas` takes quads
// cta*blockDim + threadIdx, stepping by ctas*blockDim.  OBJ: where mu comes
// from (ObjectiveSource).  OPT: the local optimiser (0 SGD, 1 Nesterov
// momentum, 2 Adam).  WIDE: some node has more than kRegDeg neighbours;
// without one the wide-node paths are not compiled, and they cost the narrow
// trees nothing.
template <int OBJ, int OPT, bool WIDE>
__device__ __forceinline__ void walk(const Program& prog, const ModelArgs& a, const Objective& obj,
                                     const PhiloxKey& mu_key, int64_t cta, int64_t ctas, float4* slot_mem,
                                     float* s_scale, float* s_fill) {
    const int n = prog.n;
    wait_for_prior_grid();
    rebuild_factors(prog, a, s_scale, s_fill);
    __syncthreads();
    const Slots sl{slot_mem + threadIdx.x, static_cast<int>(blockDim.x)};
    float4* cen = slot_mem + prog.nslots * blockDim.x + threadIdx.x;  // OBJ == kMuCachedCentres
    const int64_t stride = ctas * blockDim.x;
    for (int64_t q = cta * blockDim.x + threadIdx.x; q < a.nquads; q += stride) {
        if (OBJ == relaysum::kMuCachedCentres) {
            for (int k = 0; k < obj.K; ++k)
                cen[k * blockDim.x] = normal4(a.q0 + static_cast<uint32_t>(q), static_cast<uint32_t>(k), 0u,
                                              1u, mu_key);
        }
        // x (and a stored mu) of the next node in the walk are loaded one visit
        // early, so their latency overlaps the current visit's arithmetic
        float4 xn = *reinterpret_cast<const float4*>(a.x + prog.order[0] * a.ld_x + 4 * q);
        float4 mn = (OBJ == relaysum::kMuStored) ? ld_stream(a.mu + prog.order[0] * a.ld_x + 4 * q)
                                                  : make_float4(0.f, 0.f, 0.f, 0.f);
        for (int v = 0; v < n; ++v) {
            const int i = prog.order[v];
            const NodeRec r = prog.node[i];
            const float4 xv = xn;
            const float4 mv = (OBJ == relaysum::kMuStored)
                                  ? mn : centre<OBJ>(obj, mu_key, a, i, q, cen, static_cast<int>(blockDim.x));
            if (v + 1 < n) {  // the next node is never finalised before its own visit
                const int inext = prog.order[v + 1];
                xn = *reinterpret_cast<const float4*>(a.x + inext * a.ld_x + 4 * q);
                if (OBJ == relaysum::kMuStored) mn = ld_stream(a.mu + inext * a.ld_x + 4 * q);
            }
            // a child of a wide node p forms its incoming message as
            // T_p - m^{t-1}_{i->p}; that row is loaded before the noise
            // arithmetic, whose latency it then overlaps (with received sums
            // this is the one read of m^{t-1}_{i->p})
            float4 back = make_float4(0.f, 0.f, 0.f, 0.f);
            if (WIDE && (r.flags & relaysum::kRecvFromTotal)) {
                const float* mp = a.msg_in + prog.pos_out[r.pos_base + r.parent_pos] * a.ld_m + 4 * q;
                back = a.rsum ? ld_stream(mp) : __ldg(reinterpret_cast<const float4*>(mp));
            }
            const float4 z = normal4(a.q0 + static_cast<uint32_t>(q), static_cast<uint32_t>(i),
                                     a.step, 0u, a.key);
            const float4 xh = relayed_value<OPT>(a, i, q, xv, mv, z);
            // the rebuild sum starts from fill_i x_i (robust rule: n - nbar_i;
            // Alg. 6: n; Alg. 5: 1; Alg. 1: nothing)
            float4 acc = xh;
            if (s_fill[i] != 0.0f) acc = add4(scale4(xv, s_fill[i]), xh);
            float4 recv = make_float4(0.f, 0.f, 0.f, 0.f);
            if (r.recv_slot >= 0) {
                recv = sl[r.recv_slot];
                if (WIDE && (r.flags & relaysum::kRecvFromTotal)) {  // m^t_{p->i} = T_p - m^{t-1}_{i->p}, written out here
                    const int e = prog.pos_in[r.pos_base + r.parent_pos];
                    recv = delivered(a, e, sub4(recv, back));
                    st_stream(a.msg_out + e * a.ld_m + 4 * q, recv);
                }
                acc = add4(acc, recv);
            }
            // a wide node's received sum S_i^t starts with its DFS parent's message
            if (WIDE && a.rsum && r.deg > kRegDeg) sl[prog.rsum_slot[i]] = add4(make_float4(0.f, 0.f, 0.f, 0.f), recv);
            switch (r.deg) {
                case 0: break;
                case 1: visit_small<1, WIDE>(prog, r, a, q, xh, sl, s_scale); break;
                case 2: visit_small<2, WIDE>(prog, r, a, q, xh, sl, s_scale); break;
                case 3: visit_small<3, WIDE>(prog, r, a, q, xh, sl, s_scale); break;
                case 4: visit_small<4, WIDE>(prog, r, a, q, xh, sl, s_scale); break;
                default:
                    if (WIDE) visit_wide(prog, r, a, i, q, xh, sl, s_scale);
                    break;
            }
            if (r.acc_slot < 0) {
                st_stream(a.x + i * a.ld_x + 4 * q, scale4(acc, s_scale[i]));
            } else {
                sl[r.acc_slot] = acc;
            }
        }
    }
}

// The step kernel over NT windows.  The walk is inlined once per window, so
// each copy reads its window's program and arguments at fixed parameter
// offsets (constant operands), as the one-window kernel does; the grid's
// first `split` CTAs take window 0.
// Resident CTAs of 128 threads per SM the walk's registers are budgeted for
// (0: no bound, the compiler's choice, 72 registers and 7 CTAs for the
// stored-centre walk).  The wide-node variant runs 8 CTAs with 64 registers:
// 6.17 -> 6.08 ms per step on the 64-worker star, while the same budget
// slowed every narrow tree (double16 +11 %, binary32 +4 %; same-box A/B).
template <bool WIDE>
constexpr int kWalkMinCtas = WIDE ? 8 : 0;

template <int OBJ, int OPT, int NT, bool WIDE>
__global__ void __launch_bounds__(128, kWalkMinCtas<WIDE>)
relay_models_kernel(const __grid_constant__ Windows<NT> win, const __grid_constant__ Objective obj,
                    const __grid_constant__ PhiloxKey mu_key) {
    extern __shared__ float4 slot_mem[];
    __shared__ float s_scale[kMaxN];
    __shared__ float s_fill[kMaxN];
    if (NT == 1) {
        walk<OBJ, OPT, WIDE>(win.prog[0], win.a[0], obj, mu_key, blockIdx.x, gridDim.x, slot_mem, s_scale, s_fill);
    } else if (static_cast<int>(blockIdx.x) < win.split) {
        walk<OBJ, OPT, WIDE>(win.prog[0], win.a[0], obj, mu_key, blockIdx.x, win.split, slot_mem, s_scale, s_fill);
    } else {
        walk<OBJ, OPT, WIDE>(win.prog[NT - 1], win.a[NT - 1], obj, mu_key, blockIdx.x - win.split,
                             gridDim.x - win.split, slot_mem, s_scale, s_fill);
    }
}

// ------------------------------------------------- node-parallel fused step

// For short vectors the walk leaves the GPU idle (one thread per quad walks
// all n workers in turn), so this form of the same step gives each
// (worker, quad) pair its own thread.  A CTA owns qb consecutive quads of
// every worker (threads worker-major: a worker's qb quads are contiguous).
// Phase 1: each thread forms x_i^{t+1/2} and worker i's outgoing messages
// with the walk's arithmetic (prefix + suffix at degree <= kRegDeg, the
// total minus the reverse message above it), writes them out and leaves
// them in shared memory.  Phase 2, after one barrier: each thread adds its
// worker's incoming messages in the walk's order (Program::rb_in) and
// writes the new model.  The results equal relay_models_kernel's bit for
// bit, and every array is still read and written once.

// Degree D <= kRegDeg: outgoing message s = prefix(s) + suffix(s+1).
template <int D>
__device__ __forceinline__ void node_small(const Program& prog, const NodeRec& r, const ModelArgs& a,
                                           int64_t q, float4 xh, float4* m_new, int qb) {
    float4 m[D];
#pragma unroll
    for (int s = 0; s < D; ++s) m[s] = ld_stream(a.msg_in + prog.pos_in[r.pos_base + s] * a.ld_m + 4 * q);
    float4 pre[D];
    pre[0] = xh;
#pragma unroll
    for (int s = 1; s < D; ++s) pre[s] = add4(pre[s - 1], m[s - 1]);
    float4 suf[D];
    suf[D - 1] = m[D - 1];
#pragma unroll
    for (int s = D - 2; s >= 0; --s) suf[s] = add4(m[s], suf[s + 1]);
#pragma unroll
    for (int s = 0; s < D; ++s) {
        const int e = prog.pos_out[r.pos_base + s];
        const float4 out = delivered(a, e, (s == D - 1) ? pre[s] : add4(pre[s], suf[s + 1]));
        st_stream(a.msg_out + e * a.ld_m + 4 * q, out);
        m_new[e * qb] = out;
    }
}

// Degree D > kRegDeg: T = x^{t+1/2} + the incoming messages summed over
// descending positions (with received sums: + the sum row S_i^{t-1}), then
// message s = T - (incoming message s), as in visit_wide and at the wide
// node's children.  The incoming messages wait in shared memory (rows of
// worker i's own incoming edges).
__device__ __noinline__ void node_wide(const Program& prog, const NodeRec& r, const ModelArgs& a, int i,
                                       int64_t q, float4 xh, float4* m_new, float4* m_old, int qb) {
    const int D = r.deg;
    const int base = r.pos_base;
    float4 total = xh;
    if (a.rsum) total = add4(xh, ld_stream(a.msg_in + rsum_row(prog, i) * a.ld_m + 4 * q));
    for (int s = D - 1; s >= 0; --s) {
        const int ein = prog.pos_in[base + s];
        const float4 m = ld_stream(a.msg_in + ein * a.ld_m + 4 * q);
        if (!a.rsum) total = add4(total, m);
        m_old[ein * qb] = m;
    }
    for (int s = 0; s < D; ++s) {
        const int e = prog.pos_out[base + s];
        const float4 out = delivered(a, e, sub4(total, m_old[prog.pos_in[base + s] * qb]));
        st_stream(a.msg_out + e * a.ld_m + 4 * q, out);
        m_new[e * qb] = out;
    }
}

// blockDim.x = qb * n <= 1024.  Dynamic shared memory: two [E][qb] float4
// message buffers used by alternate blocks, plus one more for the incoming
// messages of wide nodes when the tree has any.  With two buffers a block
// needs one barrier: a warp already in the next block's phase 1 writes the
// other buffer, and it can reach this buffer again only after every warp
// has passed the next block's barrier, i.e. finished reading this one.
template <int OBJ, int OPT>
__global__ void __launch_bounds__(1024)
relay_nodes_kernel(const __grid_constant__ Program prog, const __grid_constant__ Objective obj,
                   const __grid_constant__ PhiloxKey mu_key, const __grid_constant__ ModelArgs a, int qb) {
    extern __shared__ float4 node_mem[];
    __shared__ float s_scale[kMaxN];
    __shared__ float s_fill[kMaxN];
    // regenerated centres are formed per row (the walk's cached centres are
    // the same normals mixed in the same order)
    constexpr int kObj = (OBJ == relaysum::kMuStored) ? relaysum::kMuStored : relaysum::kMuPerRow;
    const int i = static_cast<int>(threadIdx.x) / qb;
    const int qi = static_cast<int>(threadIdx.x) - i * qb;
    float4* const buf0 = node_mem + qi;                     // [e * qb]: m^t on edge e (even blocks)
    float4* const buf1 = node_mem + prog.E * qb + qi;       // (odd blocks)
    float4* const m_old = node_mem + 2 * prog.E * qb + qi;  // [e * qb]: m^{t-1} (wide nodes)
    const NodeRec r = prog.node[i];
    const float* const xrow = a.x + i * a.ld_x;
    const float* const murow = (OBJ == relaysum::kMuStored) ? a.mu + i * a.ld_x : nullptr;
    const int64_t nblk = (a.nquads + qb - 1) / qb;
    const int64_t qstep = static_cast<int64_t>(gridDim.x) * qb;
    // x (and a stored mu) of this thread's next block are loaded one block
    // early, so their latency overlaps the barrier and the rebuild
    float4 xn = make_float4(0.f, 0.f, 0.f, 0.f), mn = xn;
    int64_t q = static_cast<int64_t>(blockIdx.x) * qb + qi;
    if (q < a.nquads) {
        xn = *reinterpret_cast<const float4*>(xrow + 4 * q);
        if (OBJ == relaysum::kMuStored) mn = ld_stream(murow + 4 * q);
    }
    // Phase 1 needs no counter: the first block's runs before the wait for the
    // counter kernel (programmatic dependent launch), overlapping it; only the
    // rebuild factors of phase 2 need the counters, which the counter kernel
    // writes (it writes nothing phase 1 reads).
    bool counted = false;
    int parity = 0;
    for (int64_t b = blockIdx.x; b < nblk; b += gridDim.x, q += qstep, parity ^= 1) {
        float4* const m_new = parity ? buf1 : buf0;
        const bool active = q < a.nquads;
        const float4 xv = xn, ms = mn;
        if (q + qstep < a.nquads) {
            xn = *reinterpret_cast<const float4*>(xrow + 4 * (q + qstep));
            if (OBJ == relaysum::kMuStored) mn = ld_stream(murow + 4 * (q + qstep));
        }
        float4 xh = make_float4(0.f, 0.f, 0.f, 0.f);
        if (active) {
            const float4 mv = (OBJ == relaysum::kMuStored) ? ms : centre<kObj>(obj, mu_key, a, i, q, nullptr, 0);
            const float4 z = normal4(a.q0 + static_cast<uint32_t>(q), static_cast<uint32_t>(i), a.step, 0u,
                                     a.key);
            xh = relayed_value<OPT>(a, i, q, xv, mv, z);
            switch (r.deg) {
                case 0: break;
                case 1: node_small<1>(prog, r, a, q, xh, m_new, qb); break;
                case 2: node_small<2>(prog, r, a, q, xh, m_new, qb); break;
                case 3: node_small<3>(prog, r, a, q, xh, m_new, qb); break;
                case 4: node_small<4>(prog, r, a, q, xh, m_new, qb); break;
                default: node_wide(prog, r, a, i, q, xh, m_new, m_old, qb); break;
            }
        }
        if (!counted) {
            wait_for_prior_grid();
            rebuild_factors(prog, a, s_scale, s_fill);
            counted = true;
        }
        __syncthreads();  // also publishes the factors
        if (active) {
            // the rebuild sum starts from fill_i x_i + x^{t+1/2}, as in the walk
            float4 acc = xh;
            if (s_fill[i] != 0.0f) acc = add4(scale4(xv, s_fill[i]), xh);
            if (a.rsum && r.deg > kRegDeg) {  // and the wide node's received sum S_i^t, in the same order
                float4 sum = make_float4(0.f, 0.f, 0.f, 0.f);
                for (int k = 0; k < r.deg; ++k) {
                    const float4 m = m_new[prog.rb_in[r.pos_base + k] * qb];
                    acc = add4(acc, m);
                    sum = add4(sum, m);
                }
                st_stream(a.msg_out + rsum_row(prog, i) * a.ld_m + 4 * q, sum);
            } else {
                for (int k = 0; k < r.deg; ++k) acc = add4(acc, m_new[prog.rb_in[r.pos_base + k] * qb]);
            }
            st_stream(a.x + i * a.ld_x + 4 * q, scale4(acc, s_scale[i]));
        }
    }
}

// ------------------------------------------------ several steps per launch

// relay_steps: k consecutive steps in one launch, in the node-parallel
// layout.  Every coordinate evolves on its own (the counters are the same
// for all of them), so a CTA carries its qb quads of every worker through
// all k steps without hearing from another CTA: models, centres and
// optimiser state stay in registers, the messages of the step just taken
// in shared memory, and the CTA advances its own copy of the counters.  HBM
// is read once (x, mu, the optimiser state, m^{t0-1}) and written once (x,
// the state, and the messages of the last two steps, which k relay_step
// calls leave in the two buffers).  Each step is the node kernel's
// arithmetic in the node kernel's order, so the result equals k relay_step
// calls bit for bit.
constexpr int kMaxFusedSteps = 64;  // steps per launch (Adam's per-step factors ride in the parameters)

struct FusedSteps {
    int32_t k;                        // steps in this launch, 1 .. kMaxFusedSteps
    float* msg[2];                    // step t0 + j reads msg[j & 1] and writes msg[(j + 1) & 1]
    float adam_step[kMaxFusedSteps];  // Adam's factors of step t0 + j
    float adam_ibc2[kMaxFusedSteps];
};

// Outgoing messages of worker i from its incoming ones in shared memory
// (`prev`, this thread's column), with node_small's / node_wide's arithmetic.
// They go to `cur`, and to HBM at `out` (row e at out + e * ld_m) unless null.
template <int D>
__device__ __forceinline__ void fused_small(const Program& prog, const NodeRec& r, const ModelArgs& a, float4 xh,
                                            const float4* prev, float4* cur, int qb, float* out,
                                            uint32_t lost_bits) {
    float4 m[D];
#pragma unroll
    for (int s = 0; s < D; ++s) m[s] = prev[prog.pos_in[r.pos_base + s] * qb];
    float4 pre[D];
    pre[0] = xh;
#pragma unroll
    for (int s = 1; s < D; ++s) pre[s] = add4(pre[s - 1], m[s - 1]);
    float4 suf[D];
    suf[D - 1] = m[D - 1];
#pragma unroll
    for (int s = D - 2; s >= 0; --s) suf[s] = add4(m[s], suf[s + 1]);
#pragma unroll
    for (int s = 0; s < D; ++s) {
        const int e = prog.pos_out[r.pos_base + s];
        const float4 o = ((lost_bits >> s) & 1u) ? make_float4(0.f, 0.f, 0.f, 0.f)
                                                 : ((s == D - 1) ? pre[s] : add4(pre[s], suf[s + 1]));
        cur[e * qb] = o;
        if (out) st_stream(out + e * a.ld_m, o);
    }
}

// The rebuild sum: acc plus the incoming messages of step j in rb_in order.
template <int D>
__device__ __forceinline__ float4 fused_rebuild(const Program& prog, const NodeRec& r, const float4* cur, int qb,
                                                float4 acc) {
#pragma unroll
    for (int k = 0; k < D; ++k) acc = add4(acc, cur[prog.rb_in[r.pos_base + k] * qb]);
    return acc;
}

__device__ __noinline__ void fused_wide(const Program& prog, const NodeRec& r, const ModelArgs& a, float4 xh,
                                        const float4* prev, float4* cur, int qb, float* out) {
    const int D = r.deg;
    const int base = r.pos_base;
    float4 total = xh;
    for (int s = D - 1; s >= 0; --s) total = add4(total, prev[prog.pos_in[base + s] * qb]);
    for (int s = 0; s < D; ++s) {
        const int e = prog.pos_out[base + s];
        const float4 o = delivered(a, e, sub4(total, prev[prog.pos_in[base + s] * qb]));
        cur[e * qb] = o;
        if (out) st_stream(out + e * a.ld_m, o);
    }
}

// blockDim.x = qb * n <= 1024, threads worker-major as in relay_nodes_kernel.
// Dynamic shared memory: two [E][qb] float4 message buffers, buffer j & 1
// holding the messages of step t0 + j (buffer 1 starts with m^{t0-1}), then
// the rebuild factors (scale, fill) of every worker and step, [k][n] float2.
// The counters, hence the factors, are the same for every quad: the CTA
// advances them through the k steps once, before its first quads.  One
// barrier per step: a thread can write a buffer again only two steps later,
// after every thread has passed the barrier between, i.e. finished reading it.
template <int OBJ, int OPT>
__global__ void __launch_bounds__(1024)
relay_fused_steps_kernel(const __grid_constant__ Program prog, const __grid_constant__ Objective obj,
                         const __grid_constant__ PhiloxKey mu_key, const __grid_constant__ ModelArgs a,
                         const __grid_constant__ FusedSteps fs, int qb) {
    extern __shared__ float4 fused_mem[];
    __shared__ int32_t c_mem[2][kMaxE];  // counters of the step parities
    constexpr int kObj = (OBJ == relaysum::kMuStored) ? relaysum::kMuStored : relaysum::kMuPerRow;
    const int tid = static_cast<int>(threadIdx.x);
    const int i = tid / qb;
    const int qi = tid - i * qb;
    const int n = prog.n;
    const int E = prog.E;
    const NodeRec r = prog.node[i];
    const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
    float2* const factors = reinterpret_cast<float2*>(fused_mem + 2 * E * qb);  // [j * n + i]
    // bit s: the message to this worker's neighbour s is lost (narrow nodes)
    uint32_t lost_bits = 0;
    if (a.has_lost && r.deg <= kRegDeg)
        for (int s = 0; s < r.deg; ++s) lost_bits |= (a.lost(prog.pos_out[r.pos_base + s]) ? 1u : 0u) << s;
    for (int e = tid; e < E; e += blockDim.x) c_mem[1][e] = a.counts[e];  // c^{t0-1}
    __syncthreads();
    for (int j = 0; j < fs.k; ++j) {
        const int32_t* const c_old = c_mem[(j + 1) & 1];
        int32_t* const c_new = c_mem[j & 1];
        for (int e = tid; e < E; e += blockDim.x) c_new[e] = next_count(prog, a.lost, a.has_lost, c_old, e);
        __syncthreads();
        for (int w = tid; w < n; w += blockDim.x) {
            const NodeRec rw = prog.node[w];
            int nbar = 1;
            for (int p = 0; p < rw.deg; ++p) nbar += c_new[prog.pos_in[rw.pos_base + p]];
            float scale, fill;
            worker_factors(a, n, nbar, scale, fill);
            factors[j * n + w] = make_float2(scale, fill);
        }
    }
    const int64_t nblk = (a.nquads + qb - 1) / qb;
    for (int64_t b = blockIdx.x; b < nblk; b += gridDim.x) {
        const int64_t q = b * qb + qi;
        const bool active = q < a.nquads;
        // m^{t0-1} of this CTA's quads (coalesced rows of qb quads) into buffer 1
        for (int idx = tid; idx < E * qb; idx += blockDim.x) {
            const int e = idx / qb;
            const int64_t qg = b * qb + (idx - e * qb);
            fused_mem[E * qb + idx] = qg < a.nquads ? ld_stream(a.msg_in + e * a.ld_m + 4 * qg) : zero;
        }
        float4 xv = zero, mv = zero, m1 = zero, m2 = zero;
        if (active) {
            xv = *reinterpret_cast<const float4*>(a.x + i * a.ld_x + 4 * q);
            mv = (OBJ == relaysum::kMuStored) ? ld_stream(a.mu + i * a.ld_x + 4 * q)
                                               : centre<kObj>(obj, mu_key, a, i, q, nullptr, 0);
            if (OPT >= 1) m1 = *reinterpret_cast<const float4*>(a.s1 + i * a.ld_x + 4 * q);
            if (OPT == 2) m2 = *reinterpret_cast<const float4*>(a.s2 + i * a.ld_x + 4 * q);
        }
        __syncthreads();
        for (int j = 0; j < fs.k; ++j) {
            float4* const cur = fused_mem + (j & 1) * E * qb + qi;
            const float4* const prev = fused_mem + ((j + 1) & 1) * E * qb + qi;
            float4 xh = zero;
            if (active) {
                const float4 z = normal4(a.q0 + static_cast<uint32_t>(q), static_cast<uint32_t>(i),
                                         a.step + static_cast<uint32_t>(j), 0u, a.key);
                const float st = fs.adam_step[j], ib = fs.adam_ibc2[j];
                xh = relayed_with(a, xv, mv, z, [&](float4 g) { return update_rule<OPT>(a, st, ib, g, m1, m2); });
                float* const out = (E > 0 && j + 2 >= fs.k) ? fs.msg[(j + 1) & 1] + 4 * q : nullptr;
                switch (r.deg) {
                    case 0: break;
                    case 1: fused_small<1>(prog, r, a, xh, prev, cur, qb, out, lost_bits); break;
                    case 2: fused_small<2>(prog, r, a, xh, prev, cur, qb, out, lost_bits); break;
                    case 3: fused_small<3>(prog, r, a, xh, prev, cur, qb, out, lost_bits); break;
                    case 4: fused_small<4>(prog, r, a, xh, prev, cur, qb, out, lost_bits); break;
                    default: fused_wide(prog, r, a, xh, prev, cur, qb, out); break;
                }
            }
            __syncthreads();
            if (active) {
                const float2 f = factors[j * n + i];  // (scale, fill)
                float4 acc = xh;
                if (f.y != 0.0f) acc = add4(scale4(xv, f.y), xh);
                switch (r.deg) {
                    case 0: break;
                    case 1: acc = fused_rebuild<1>(prog, r, cur, qb, acc); break;
                    case 2: acc = fused_rebuild<2>(prog, r, cur, qb, acc); break;
                    case 3: acc = fused_rebuild<3>(prog, r, cur, qb, acc); break;
                    case 4: acc = fused_rebuild<4>(prog, r, cur, qb, acc); break;
                    default:
                        for (int k = 0; k < r.deg; ++k) acc = add4(acc, cur[prog.rb_in[r.pos_base + k] * qb]);
                        break;
                }
                xv = scale4(acc, f.x);
            }
        }
        if (active) {
            st_stream(a.x + i * a.ld_x + 4 * q, xv);
            if (OPT >= 1) st_stream(a.s1 + i * a.ld_x + 4 * q, m1);
            if (OPT == 2) st_stream(a.s2 + i * a.ld_x + 4 * q, m2);
        }
        __syncthreads();  // the next block refills buffer 1
    }
}

// --------------------------------------------------------------------- init

// rows: message rows to zero (E, plus the received-sum rows when they are on).
__global__ void relay_init_kernel(float* x, float* msg_a, float* msg_b, int n, int rows, int64_t ld_x,
                                  int64_t ld_m, int64_t nquads, int64_t d, uint32_t q0, float x0_std,
                                  const __grid_constant__ PhiloxKey key) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < nquads; q += stride) {
        const int64_t c = 4 * q;
        const float4 z = normal4(q0 + static_cast<uint32_t>(q), 0u, 0u, 2u, key);
        const float4 v = make_float4(x0_std * z.x, c + 1 < d ? x0_std * z.y : 0.f,
                                     c + 2 < d ? x0_std * z.z : 0.f, c + 3 < d ? x0_std * z.w : 0.f);
        for (int i = 0; i < n; ++i) *reinterpret_cast<float4*>(x + i * ld_x + c) = v;
        const float4 zero = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int e = 0; e < rows; ++e) {
            *reinterpret_cast<float4*>(msg_a + e * ld_m + c) = zero;
            if (msg_b) *reinterpret_cast<float4*>(msg_b + e * ld_m + c) = zero;
        }
    }
}

__global__ void relay_fill_mu_kernel(float* mu, const float* mix, int n, int K, int64_t ld_x, int64_t nquads,
                                     int64_t d, uint32_t q0, float scale, const __grid_constant__ PhiloxKey key) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < nquads; q += stride) {
        const int64_t c = 4 * q;
        for (int i = 0; i < n; ++i) {
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int k = 0; k < K; ++k) {
                const float w = __ldg(mix + static_cast<int64_t>(i) * K + k);
                if (w != 0.0f) {  // a zero weight adds exactly nothing
                    const float4 z = normal4(q0 + static_cast<uint32_t>(q), static_cast<uint32_t>(k), 0u, 1u, key);
                    acc = fma4(w, z, acc);
                }
            }
            const float4 sv = scale4_rn(acc, scale);
            *reinterpret_cast<float4*>(mu + i * ld_x + c) =
                make_float4(sv.x, c + 1 < d ? sv.y : 0.f, c + 2 < d ? sv.z : 0.f, c + 3 < d ? sv.w : 0.f);
        }
    }
}

// ------------------------------------------------------------------ metrics

// Consensus distance and distance to the optimum (the quantities of the
// paper's analysis, Section 4): per coordinate c, with xbar = mean_i x_i and
// mubar = mean_i mu_i,
//   xi   += sum_i (x_i - xbar)^2        dist += (xbar - mubar)^2
// Pass 1: each block reduces its share of the coordinates (grid-stride,
// fixed order) into partials[2 blockIdx]; pass 2 sums the partials in a
// fixed order, so the result is deterministic.  Within a coordinate the
// sums over the workers run in fp32 pairs (below) and only the coordinate's
// totals in double: the GB300's fp64 rate is a small fraction of its fp32
// rate, and per-worker fp64 arithmetic made the metrics fp64-bound.
constexpr int kMetricsThreads = 256;
constexpr int kMetricsMaxBlocks = 1024;

// A running fp32 sum kept as the unevaluated pair s + c (Neumaier's
// compensated summation): c gathers every addition's exact rounding error,
// so the pair carries about twice fp32's precision.  The _rn intrinsics
// keep the compiler from contracting or reordering the error terms.
struct PairSum {
    float s = 0.0f, c = 0.0f;
    __device__ __forceinline__ void add(float v) {
        const float t = __fadd_rn(s, v);
        const float e = (fabsf(s) >= fabsf(v)) ? __fadd_rn(__fsub_rn(s, t), v) : __fadd_rn(__fsub_rn(v, t), s);
        c = __fadd_rn(c, e);
        s = t;
    }
    __device__ __forceinline__ double value() const { return static_cast<double>(s) + static_cast<double>(c); }
};

// The exact rounding error of a + b, given s = fl(a + b) (Knuth's TwoSum).
__device__ __forceinline__ float sum_error(float a, float b, float s) {
    const float bb = __fsub_rn(s, a);
    return __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
}

__device__ __forceinline__ double block_sum(double v, double* red) {
    for (int o = 16; o > 0; o >>= 1) v += __shfl_down_sync(0xffffffffu, v, o);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    __syncthreads();
    if (lane == 0) red[warp] = v;
    __syncthreads();
    double s = 0.0;
    if (threadIdx.x == 0)
        for (int w = 0; w < static_cast<int>(blockDim.x >> 5); ++w) s += red[w];
    return s;  // valid in thread 0
}

template <int OBJ>
__global__ void __launch_bounds__(kMetricsThreads)
relay_metrics_kernel(const __grid_constant__ Objective obj, const __grid_constant__ PhiloxKey mu_key,
                     const __grid_constant__ ModelArgs a, int n, int64_t d, double* partials) {
    __shared__ double red[kMetricsThreads / 32];
    double xi = 0.0, dist = 0.0;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    const double inv_n = 1.0 / n;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < a.nquads; q += stride) {
        PairSum xs[4], ms[4];
        for (int i = 0; i < n; ++i) {
            const float4 xv = *reinterpret_cast<const float4*>(a.x + i * a.ld_x + 4 * q);
            const float4 mv = centre<OBJ>(obj, mu_key, a, i, q, nullptr, 0);
            xs[0].add(xv.x); xs[1].add(xv.y); xs[2].add(xv.z); xs[3].add(xv.w);
            ms[0].add(mv.x); ms[1].add(mv.y); ms[2].add(mv.z); ms[3].add(mv.w);
        }
        // xbar as the fp32 pair hi + lo
        float hi[4], lo[4];
        double xb[4];
        for (int k = 0; k < 4; ++k) {
            xb[k] = xs[k].value() * inv_n;
            hi[k] = static_cast<float>(xb[k]);
            lo[k] = static_cast<float>(xb[k] - static_cast<double>(hi[k]));
        }
        // sum_i (x_i - xbar)^2: x_i - hi exactly as t + its rounding error,
        // less lo; t^2 exactly as p + its fma remainder
        PairSum sq[4];
        float sq_lo[4] = {0.f, 0.f, 0.f, 0.f};
        for (int i = 0; i < n; ++i) {
            const float4 xv = *reinterpret_cast<const float4*>(a.x + i * a.ld_x + 4 * q);
            const float xk[4] = {xv.x, xv.y, xv.z, xv.w};
            for (int k = 0; k < 4; ++k) {
                const float t = __fsub_rn(xk[k], hi[k]);
                const float dl = __fsub_rn(sum_error(xk[k], -hi[k], t), lo[k]);
                const float p = __fmul_rn(t, t);
                const float pe = __fmaf_rn(t, t, -p);
                sq[k].add(p);
                sq_lo[k] = __fadd_rn(sq_lo[k], __fmaf_rn(__fmul_rn(2.0f, t), dl, pe));
            }
        }
        for (int k = 0; k < 4; ++k)
            if (4 * q + k < d) {
                xi += sq[k].value() + static_cast<double>(sq_lo[k]);
                const double e = xb[k] - ms[k].value() * inv_n;
                dist += e * e;
            }
    }
    const double bxi = block_sum(xi, red);
    const double bdist = block_sum(dist, red);
    if (threadIdx.x == 0) {
        partials[2 * blockIdx.x] = bxi;
        partials[2 * blockIdx.x + 1] = bdist;
    }
}

__global__ void relay_metrics_finish_kernel(const double* partials, int blocks, double scale_xi,
                                            double scale_dist, double* out) {
    __shared__ double red[kMetricsThreads / 32];
    double xi = 0.0, dist = 0.0;
    for (int b = threadIdx.x; b < blocks; b += blockDim.x) {
        xi += partials[2 * b];
        dist += partials[2 * b + 1];
    }
    const double sxi = block_sum(xi, red);
    const double sdist = block_sum(dist, red);
    if (threadIdx.x == 0) {
        out[0] = sxi * scale_xi;
        out[1] = sdist * scale_dist;
    }
}

// ------------------------------------------------------------- host helpers

constexpr int kMaxDevices = 64;
// dynamic shared memory cap: 227 KB per CTA minus the static scale/fill tables
constexpr int kMaxSmem = 224 * 1024;

int device_sms(int* dev_out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return -1;
    static std::atomic<int> sms_cache[kMaxDevices];
    int sms = (dev < kMaxDevices) ? sms_cache[dev].load() : 0;
    if (sms <= 0) {
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return -1;
        if (dev < kMaxDevices) sms_cache[dev].store(sms);
    }
    *dev_out = dev;
    return sms;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlap(const void* a, int64_t abytes, const void* b, int64_t bbytes) {
    if (abytes <= 0 || bbytes <= 0) return false;
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
    return a0 < b0 + static_cast<uintptr_t>(bbytes) && b0 < a0 + static_cast<uintptr_t>(abytes);
}

int launch_status() {
    return cudaGetLastError() == cudaSuccess ? RELAY_OK : RELAY_ECUDA;
}

// Launches a step kernel; `after_counts` makes it a programmatic dependent of
// the counter kernel just enqueued on the same stream (relay_step only).
template <typename... Params, typename... Args>
int launch_step_kernel(void (*kernel)(Params...), int grid, int threads, size_t smem, cudaStream_t stream,
                       bool after_counts, Args... args) {
    if (!after_counts) {
        kernel<<<grid, threads, smem, stream>>>(args...);
        return launch_status();
    }
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(static_cast<unsigned>(threads));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kernel, args...) != cudaSuccess) return RELAY_ECUDA;
    return launch_status();
}

// AUTO picks the node-parallel kernel below this many worker-quads (n times
// the quads) when no worker has more than kRegDeg neighbours.  Measured on
// one GB300 (whole step, L2 flushed, n = 8 to 64): the node kernel is ahead
// below about 2^21 worker-quads on chains, binary trees and the torus tree
// and even or behind above; on a star one thread carries the hub's edges
// while its CTA waits, so the walk stays faster there.
constexpr int64_t kNodesBelowWorkerQuads = int64_t(1) << 21;

// Threads per CTA for the fused kernel: 128, fewer when the slots would not
// fit in shared memory.
int models_threads(int nslots) {
    int t = 128;
    while (t > 32 && static_cast<int64_t>(nslots) * t * 16 > kMaxSmem) t -= 32;
    return t;
}

// Opts `Kernel` in to the dynamic shared memory it may use (kMaxSmem, less
// when its static shared memory and kMaxSmem would pass the device's per-CTA
// limit) once per device, and returns its resident CTAs per SM for
// (threads, smem).  Both are cached per device (queried once, not per step:
// steps may be captured into CUDA graphs); each kernel instantiation has its
// own cache.  0 on a CUDA error, which is cleared so that it is not reported
// again by a later launch.
template <auto Kernel>
int resident_ctas(int dev, int threads, size_t smem) {
    static std::atomic<bool> smem_set[kMaxDevices];
    if (dev >= kMaxDevices || !smem_set[dev].load()) {
        cudaFuncAttributes fa;
        int optin = 0;
        if (cudaFuncGetAttributes(&fa, Kernel) != cudaSuccess ||
            cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        const int room = optin - static_cast<int>(fa.sharedSizeBytes);
        if (room <= 0 ||
            cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 room < kMaxSmem ? room : kMaxSmem) != cudaSuccess) {
            (void)cudaGetLastError();
            return 0;
        }
        if (dev < kMaxDevices) smem_set[dev].store(true);
    }
    static std::atomic<int64_t> occ_cache[kMaxDevices];
    const int64_t key = static_cast<int64_t>(smem) * 1024 + threads;
    const int64_t cached = dev < kMaxDevices ? occ_cache[dev].load() : 0;
    if (cached != 0 && (cached >> 8) == key) return static_cast<int>(cached & 0xFF);
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, Kernel, threads, smem) != cudaSuccess || per_sm <= 0) {
        (void)cudaGetLastError();
        return 0;
    }
    if (dev < kMaxDevices) occ_cache[dev].store((key << 8) | (per_sm & 0xFF));
    return per_sm;
}

// The walk over NT handles' windows in one launch (NT = 1: one handle).  The
// handles share the objective source and the local optimiser (the caller
// checks); threads and shared memory are sized for the larger program, and
// the CTAs are split between the windows in proportion to their quads.
template <int OBJ, int OPT, int NT, bool WIDE>
int launch_models(const relay_handle* const* hs, const ModelArgs* as, cudaStream_t stream, bool after_counts) {
    int dev = 0;
    const int sms = device_sms(&dev);
    if (sms <= 0) return RELAY_ECUDA;
    int per_thread = 0;
    for (int k = 0; k < NT; ++k)
        per_thread = std::max(per_thread, hs[k]->prog.nslots + (OBJ == relaysum::kMuCachedCentres ? hs[k]->obj.K : 0));
    const int threads = models_threads(per_thread);
    const size_t smem = static_cast<size_t>(per_thread) * threads * 16;
    if (smem > static_cast<size_t>(kMaxSmem)) return RELAY_EUNSUPPORTED;
    const int per_sm = resident_ctas<relay_models_kernel<OBJ, OPT, NT, WIDE>>(dev, threads, smem);
    if (per_sm <= 0) return RELAY_ECUDA;
    const int64_t cap = static_cast<int64_t>(sms) * per_sm;
    int64_t want[NT], total = 0, nq = 0;
    for (int k = 0; k < NT; ++k) {
        want[k] = (as[k].nquads + threads - 1) / threads;
        total += want[k];
        nq += as[k].nquads;
    }
    Windows<NT> win;
    for (int k = 0; k < NT; ++k) {
        win.prog[k] = hs[k]->prog;
        win.a[k] = as[k];
    }
    int64_t grid = total < cap ? total : cap;
    win.split = 0;
    if (NT == 2) {
        int64_t split = want[0];
        if (total > cap) {  // CTAs in proportion to the quads, at least one per window
            split = (cap * as[0].nquads + nq / 2) / nq;
            split = std::min(std::max<int64_t>(split, 1), cap - 1);
        }
        win.split = static_cast<int32_t>(split);
    }
    const PhiloxKey mu_key =
        philox_key(static_cast<uint64_t>(hs[0]->obj.k0) | (static_cast<uint64_t>(hs[0]->obj.k1) << 32));
    return launch_step_kernel(relay_models_kernel<OBJ, OPT, NT, WIDE>, static_cast<int>(grid), threads, smem, stream,
                              after_counts, win, hs[0]->obj, mu_key);
}

// Quads per CTA of the node-parallel kernel, threads = qb * n <= 1024: a
// whole warp per worker up to n = 16 (every per-worker table read is then
// warp-uniform), half a warp up to 64, then 8 and 4 quads.
int nodes_qb(int n) { return n <= 16 ? 32 : n <= 64 ? 16 : n <= 128 ? 8 : 4; }

template <int OBJ, int OPT>
int launch_nodes(const relay_handle* h, const ModelArgs& a, cudaStream_t stream, bool after_counts) {
    int dev = 0;
    const int sms = device_sms(&dev);
    if (sms <= 0) return RELAY_ECUDA;
    const int qb = nodes_qb(h->prog.n);
    const int threads = qb * h->prog.n;
    bool wide = false;
    for (int i = 0; i < h->prog.n; ++i) wide = wide || h->prog.node[i].deg > kRegDeg;
    const size_t smem = static_cast<size_t>(wide ? 3 : 2) * h->prog.E * qb * 16;
    if (smem > static_cast<size_t>(kMaxSmem)) return RELAY_EUNSUPPORTED;
    const int per_sm = resident_ctas<relay_nodes_kernel<OBJ, OPT>>(dev, threads, smem);
    if (per_sm <= 0) return RELAY_ECUDA;
    const int64_t want = (a.nquads + qb - 1) / qb;
    const int64_t cap = static_cast<int64_t>(sms) * per_sm;
    const int grid = static_cast<int>(want < cap ? want : cap);
    const PhiloxKey mu_key = philox_key(static_cast<uint64_t>(h->obj.k0) | (static_cast<uint64_t>(h->obj.k1) << 32));
    return launch_step_kernel(relay_nodes_kernel<OBJ, OPT>, grid, threads, smem, stream, after_counts, h->prog,
                              h->obj, mu_key, a, qb);
}

// AUTO: the walk keeps every array's traffic at one pass with one thread
// per quad; below about one resident wave of those threads the GPU idles,
// and the node-parallel form (n threads per quad) is used instead.
bool use_nodes(const relay_handle* h) {
    if (h->kernel == RELAY_KERNEL_NODES) return true;
    if (h->kernel == RELAY_KERNEL_WALK) return false;
    if (h->nquads * h->prog.n >= kNodesBelowWorkerQuads) return false;
    for (int i = 0; i < h->prog.n; ++i)
        if (h->prog.node[i].deg > kRegDeg) return false;
    return true;
}

// Whether a tree has a node of degree > kRegDeg (the walk's WIDE variant).
bool has_wide(const relay_handle* h) {
    for (int i = 0; i < h->prog.n; ++i)
        if (h->prog.node[i].deg > kRegDeg) return true;
    return false;
}

template <int OPT, int NT, bool WIDE>
int launch_walk_src(const relay_handle* const* hs, const ModelArgs* as, cudaStream_t stream, bool after_counts) {
    switch (hs[0]->obj.source) {
        case relaysum::kMuStored: return launch_models<relaysum::kMuStored, OPT, NT, WIDE>(hs, as, stream, after_counts);
        case relaysum::kMuPerRow: return launch_models<relaysum::kMuPerRow, OPT, NT, WIDE>(hs, as, stream, after_counts);
        default: return launch_models<relaysum::kMuCachedCentres, OPT, NT, WIDE>(hs, as, stream, after_counts);
    }
}

// One handle: the WIDE variant when its tree has a wide node.  Several
// windows (relay_step_windows) launch together only when none has one.
template <int OPT, int NT>
int launch_walk_obj(const relay_handle* const* hs, const ModelArgs* as, cudaStream_t stream, bool after_counts) {
    if (NT == 1 && has_wide(hs[0])) return launch_walk_src<OPT, 1, true>(hs, as, stream, after_counts);
    return launch_walk_src<OPT, NT, false>(hs, as, stream, after_counts);
}

template <int OPT>
int launch_models_obj(const relay_handle* h, const ModelArgs& a, cudaStream_t stream, bool after_counts) {
    if (use_nodes(h)) {
        if (h->obj.source == relaysum::kMuStored)
            return launch_nodes<relaysum::kMuStored, OPT>(h, a, stream, after_counts);
        return launch_nodes<relaysum::kMuPerRow, OPT>(h, a, stream, after_counts);
    }
    return launch_walk_obj<OPT, 1>(&h, &a, stream, after_counts);
}

// Quads per CTA of relay_fused_steps_kernel: nodes_qb, halved (down to 4)
// while that leaves fewer CTAs than SMs, so short vectors still spread over
// the whole GPU.
int fused_qb(int n, int64_t nquads, int sms) {
    int qb = nodes_qb(n);
    while (qb > 4 && (nquads + qb - 1) / qb < sms) qb /= 2;
    return qb;
}

template <int OBJ, int OPT>
int launch_fused(const relay_handle* h, const ModelArgs& a, const FusedSteps& fs, cudaStream_t stream) {
    int dev = 0;
    const int sms = device_sms(&dev);
    if (sms <= 0) return RELAY_ECUDA;
    const int qb = fused_qb(h->prog.n, a.nquads, sms);
    const int threads = qb * h->prog.n;
    const size_t smem = static_cast<size_t>(2) * h->prog.E * qb * 16 + static_cast<size_t>(fs.k) * h->prog.n * 8;
    if (smem > static_cast<size_t>(kMaxSmem)) return RELAY_EUNSUPPORTED;
    const int per_sm = resident_ctas<relay_fused_steps_kernel<OBJ, OPT>>(dev, threads, smem);
    if (per_sm <= 0) return RELAY_ECUDA;
    const int64_t want = (a.nquads + qb - 1) / qb;
    const int64_t cap = static_cast<int64_t>(sms) * per_sm;
    const int grid = static_cast<int>(want < cap ? want : cap);
    const PhiloxKey mu_key = philox_key(static_cast<uint64_t>(h->obj.k0) | (static_cast<uint64_t>(h->obj.k1) << 32));
    relay_fused_steps_kernel<OBJ, OPT><<<grid, threads, smem, stream>>>(h->prog, h->obj, mu_key, a, fs, qb);
    return launch_status();
}

// relay_steps takes the multi-step kernel unless the walk is forced or, under
// AUTO, a worker has more than kRegDeg neighbours: its threads then carry
// all its edges at every step while the rest of the CTA waits at the
// barrier (a 64-worker star measured 3.7x slower than one relay_step per
// step).  Measured on one GB300 with every degree <= kRegDeg, from 8 workers
// and d = 4096 to 32 workers and d = 1.1e8, the multi-step kernel was ahead
// everywhere (1.2x to 1.8x).
bool use_fused(const relay_handle* h) {
    if (h->prog.nwide > 0) return false;  // received-sum rows are kept by the per-step kernels only
    if (h->kernel == RELAY_KERNEL_NODES) return true;
    if (h->kernel == RELAY_KERNEL_WALK) return false;
    for (int i = 0; i < h->prog.n; ++i)
        if (h->prog.node[i].deg > kRegDeg) return false;
    return true;
}

template <int OPT>
int launch_fused_obj(const relay_handle* h, const ModelArgs& a, const FusedSteps& fs, cudaStream_t stream) {
    if (h->obj.source == relaysum::kMuStored) return launch_fused<relaysum::kMuStored, OPT>(h, a, fs, stream);
    return launch_fused<relaysum::kMuPerRow, OPT>(h, a, fs, stream);
}

// Rows of a message buffer: E, plus one received-sum row per wide node when
// received sums are on.
int message_rows(const relay_handle* h) { return h->prog.E + h->prog.nwide; }

// Argument checks shared by relay_step_models and relay_step.
int check_step_args(const relay_handle* h, const float* x, const float* msg_in, const float* msg_out,
                    const int32_t* counts, float lr, int64_t step) {
    if (!h || !h->has_objective || !std::isfinite(lr)) return RELAY_EINVAL;
    if (step < 0 || step >= (int64_t(1) << 32)) return RELAY_EINVAL;
    const int E = h->prog.E;
    const int rows = message_rows(h);
    if (E > 0 && !counts) return RELAY_EINVAL;
    if (h->d == 0) return RELAY_OK;  // counters only
    if (E > 0 && (!msg_in || !msg_out || msg_in == msg_out)) return RELAY_EINVAL;
    if (!x || !aligned16(x) || (E > 0 && (!aligned16(msg_in) || !aligned16(msg_out))))
        return RELAY_EINVAL;
    // exact byte spans of the strided arrays (windows of wider arrays may sit side by side)
    const int64_t xb = ((h->prog.n - 1) * h->ld_x + 4 * h->nquads) * 4;
    const int64_t mb = rows > 0 ? ((rows - 1) * h->ld_m + 4 * h->nquads) * 4 : 0;
    if (overlap(x, xb, msg_in, mb) || overlap(x, xb, msg_out, mb) || overlap(msg_in, mb, msg_out, mb))
        return RELAY_EINVAL;
    for (const float* st : {static_cast<const float*>(h->s1), static_cast<const float*>(h->s2)})
        if (st && (overlap(st, xb, x, xb) || overlap(st, xb, msg_in, mb) || overlap(st, xb, msg_out, mb)))
            return RELAY_EINVAL;
    return RELAY_OK;
}

int grid_for(int64_t items, int threads) {
    int dev = 0;
    const int sms = device_sms(&dev);
    const int64_t want = (items + threads - 1) / threads;
    const int64_t cap = static_cast<int64_t>(sms > 0 ? sms : 1) * 8;
    return static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
}

// Window k of a counter launch: handle h's program, lost mask and arrays.
template <int NT>
void count_window(const relay_handle* h, int32_t* counts, CountWindows<NT>& cw, int k) {
    cw.prog[k] = h->prog;
    std::memcpy(cw.lost[k].w, h->lost, sizeof(cw.lost[k].w));
    cw.has_lost[k] = h->has_lost ? 1 : 0;
    cw.counts[k] = counts;
    cw.dme_count[k] = h->algo == RELAY_ALGO_DME ? h->dme_count : nullptr;
}

}  // namespace

// ====================================================================== ABI

extern "C" {

int relay_create(relay_handle** out, int32_t n, int64_t d, const int32_t* edges, int32_t n_edges) {
    if (out == nullptr) return RELAY_EINVAL;
    *out = nullptr;
    if (d < 0) return RELAY_EINVAL;
    const int64_t ld = (d + 31) / 32 * 32;
    if (ld / 4 >= (int64_t(1) << 32)) return RELAY_EINVAL;
    relay_handle* h = new (std::nothrow) relay_handle;
    if (h == nullptr) return RELAY_ENOMEM;
    int rc = RELAY_OK;
    try {
        rc = relaysum::build_program(n, edges, n_edges, &h->prog);
    } catch (...) {
        rc = RELAY_ENOMEM;
    }
    if (rc != RELAY_OK) {
        delete h;
        return rc;
    }
    h->d = d;
    h->ld = ld;
    h->ld_x = ld;
    h->ld_m = ld;
    h->nquads = (d + 3) / 4;
    *out = h;
    return RELAY_OK;
}

void relay_destroy(relay_handle* h) { delete h; }

int64_t relay_ld(const relay_handle* h) { return h ? h->ld : RELAY_EINVAL; }

int32_t relay_num_edges(const relay_handle* h) { return h ? h->prog.E : RELAY_EINVAL; }

int relay_edges(const relay_handle* h, int32_t* src, int32_t* dst) {
    if (!h || (h->prog.E > 0 && (!src || !dst))) return RELAY_EINVAL;
    for (int e = 0; e < h->prog.E; ++e) {
        src[e] = h->prog.edge_src[e];
        dst[e] = h->prog.edge_dst[e];
    }
    return RELAY_OK;
}

int relay_set_strides(relay_handle* h, int64_t ld_x, int64_t ld_msg) {
    if (!h || ld_x < 4 * h->nquads || ld_msg < 4 * h->nquads || (ld_x & 3) || (ld_msg & 3)) return RELAY_EINVAL;
    h->ld_x = ld_x;
    h->ld_m = ld_msg;
    return RELAY_OK;
}

int relay_set_local_optimizer(relay_handle* h, int32_t kind, float beta1, float beta2, float eps,
                              float* state1, float* state2) {
    if (!h || kind < RELAY_OPT_SGD || kind > RELAY_OPT_ADAM) return RELAY_EINVAL;
    if (!std::isfinite(beta1) || !std::isfinite(beta2) || !std::isfinite(eps)) return RELAY_EINVAL;
    if (kind == RELAY_OPT_NESTEROV && (beta1 < 0.0f || beta1 >= 1.0f)) return RELAY_EINVAL;
    if (kind == RELAY_OPT_ADAM &&
        (beta1 < 0.0f || beta1 >= 1.0f || beta2 < 0.0f || beta2 >= 1.0f || !(eps > 0.0f)))
        return RELAY_EINVAL;
    if (h->d > 0 && kind >= RELAY_OPT_NESTEROV && (!state1 || !aligned16(state1))) return RELAY_EINVAL;
    if (h->d > 0 && kind == RELAY_OPT_ADAM && (!state2 || !aligned16(state2) || state2 == state1))
        return RELAY_EINVAL;
    h->opt = kind;
    h->beta1 = beta1;
    h->beta2 = beta2;
    h->eps = eps;
    h->s1 = kind >= RELAY_OPT_NESTEROV ? state1 : nullptr;
    h->s2 = kind == RELAY_OPT_ADAM ? state2 : nullptr;
    return RELAY_OK;
}

int relay_set_algorithm(relay_handle* h, int32_t algo, int64_t* dme_count) {
    if (!h || algo < RELAY_ALGO_RELAYSGD || algo > RELAY_ALGO_DME) return RELAY_EINVAL;
    if (algo == RELAY_ALGO_DME && !dme_count) return RELAY_EINVAL;
    h->algo = algo;
    h->dme_count = algo == RELAY_ALGO_DME ? dme_count : nullptr;
    return RELAY_OK;
}

int relay_set_lost_messages(relay_handle* h, const uint8_t* lost) {
    if (!h) return RELAY_EINVAL;
    std::memset(h->lost, 0, sizeof(h->lost));
    h->has_lost = false;
    if (!lost) return RELAY_OK;
    for (int e = 0; e < h->prog.E; ++e)
        if (lost[e]) {
            h->lost[e >> 5] |= 1u << (e & 31);
            h->has_lost = true;
        }
    return RELAY_OK;
}

int relay_set_rebuild_mode(relay_handle* h, int32_t mode) {
    if (!h || (mode != 0 && mode != 1)) return RELAY_EINVAL;
    h->mode = mode;
    return RELAY_OK;
}

int relay_set_kernel(relay_handle* h, int32_t kernel) {
    if (!h || kernel < RELAY_KERNEL_AUTO || kernel > RELAY_KERNEL_NODES) return RELAY_EINVAL;
    h->kernel = kernel;
    return RELAY_OK;
}

int relay_set_received_sums(relay_handle* h, int32_t enable) {
    if (!h || (enable != 0 && enable != 1)) return RELAY_EINVAL;
    if ((enable != 0) == h->rsum) return RELAY_OK;
    // rebuild the visit program from the handle's own edge list (edge 2u is
    // the u-th pair as given)
    const int n = h->prog.n;
    int32_t edges[2 * (kMaxN - 1)];
    for (int u = 0; u < n - 1; ++u) {
        edges[2 * u] = h->prog.edge_src[2 * u];
        edges[2 * u + 1] = h->prog.edge_dst[2 * u];
    }
    Program* p = new (std::nothrow) Program;
    if (!p) return RELAY_ENOMEM;
    int rc = RELAY_OK;
    try {
        rc = relaysum::build_program(n, edges, n - 1, p, enable != 0);
    } catch (...) {
        rc = RELAY_ENOMEM;
    }
    if (rc == RELAY_OK) {
        h->prog = *p;
        h->rsum = enable != 0;
    }
    delete p;
    return rc;
}

int32_t relay_message_rows(const relay_handle* h) { return h ? message_rows(h) : RELAY_EINVAL; }

int relay_get_kernel(const relay_handle* h) {
    if (!h) return RELAY_EINVAL;
    return use_nodes(h) ? RELAY_KERNEL_NODES : RELAY_KERNEL_WALK;
}

int relay_set_coord_offset(relay_handle* h, int64_t c0) {
    if (!h || c0 < 0 || (c0 & 3) != 0) return RELAY_EINVAL;
    if ((c0 + h->ld) / 4 >= (int64_t(1) << 32)) return RELAY_EINVAL;
    h->c0 = c0;
    return RELAY_OK;
}

int relay_set_objective(relay_handle* h, const float* mu, float sigma) {
    if (!h || !std::isfinite(sigma) || sigma < 0.0f) return RELAY_EINVAL;
    if (h->d > 0 && (!mu || !aligned16(mu))) return RELAY_EINVAL;
    h->mu = mu;
    h->sigma = sigma;
    h->obj.source = relaysum::kMuStored;
    h->has_objective = true;
    return RELAY_OK;
}

// The non-zeros of a host mixture matrix mix [n][K] into an Objective.
static int mixture(const relay_handle* h, const float* mix, int32_t K, float mu_scale, Objective* o, int* nnz_out) {
    if (K > 32767) return RELAY_EUNSUPPORTED;
    const int n = h->prog.n;
    std::memset(o, 0, sizeof(*o));
    int nnz = 0;
    for (int i = 0; i < n; ++i) {
        o->row_off[i] = static_cast<int16_t>(nnz);
        for (int k = 0; k < K; ++k) {
            const float w = mix[static_cast<int64_t>(i) * K + k];
            if (!std::isfinite(w)) return RELAY_EINVAL;
            if (w == 0.0f) continue;
            if (nnz >= relaysum::kMaxMixNnz) return RELAY_EUNSUPPORTED;
            o->col[nnz] = static_cast<int16_t>(k);
            o->w[nnz] = w;
            ++nnz;
        }
    }
    o->row_off[n] = static_cast<int16_t>(nnz);
    o->K = K;
    o->scale = mu_scale;
    *nnz_out = nnz;
    return RELAY_OK;
}

int relay_set_objective_generated(relay_handle* h, const float* mix, int32_t K, float mu_scale,
                                  uint64_t mu_seed, float sigma) {
    if (!h || K < 0 || (K > 0 && !mix) || !std::isfinite(mu_scale) || !std::isfinite(sigma) ||
        sigma < 0.0f)
        return RELAY_EINVAL;
    Objective o;
    int nnz = 0;
    const int rc = mixture(h, mix, K, mu_scale, &o, &nnz);
    if (rc != RELAY_OK) return rc;
    o.k0 = static_cast<uint32_t>(mu_seed);
    o.k1 = static_cast<uint32_t>(mu_seed >> 32);
    // one Philox block per non-zero, or K per quad when that is fewer
    o.source = (K <= relaysum::kMaxCachedCentres && K < nnz) ? relaysum::kMuCachedCentres
                                                              : relaysum::kMuPerRow;
    h->obj = o;
    h->mu = nullptr;
    h->sigma = sigma;
    h->has_objective = true;
    return RELAY_OK;
}

int relay_fill_objective(relay_handle* h, float* mu, const float* mix, int32_t K, float mu_scale,
                         uint64_t mu_seed, relay_stream_t stream) {
    if (!h || K < 0 || !std::isfinite(mu_scale)) return RELAY_EINVAL;
    if (h->d == 0) return RELAY_OK;
    if (!mu || !aligned16(mu) || (K > 0 && !mix)) return RELAY_EINVAL;
    const int threads = 256;
    relay_fill_mu_kernel<<<grid_for(h->nquads, threads), threads, 0, stream>>>(
        mu, mix, h->prog.n, K, h->ld_x, h->nquads, h->d, static_cast<uint32_t>(h->c0 / 4), mu_scale,
        philox_key(mu_seed));
    return launch_status();
}

int relay_init(relay_handle* h, float* x, float* msg_a, float* msg_b, int32_t* counts, float x0_std,
               uint64_t seed, relay_stream_t stream) {
    if (!h || !std::isfinite(x0_std)) return RELAY_EINVAL;
    const int E = h->prog.E;
    if (E > 0 && !counts) return RELAY_EINVAL;
    if (h->d > 0 && (!x || !aligned16(x) || (E > 0 && (!msg_a || !aligned16(msg_a))) ||
                     (msg_b && !aligned16(msg_b))))
        return RELAY_EINVAL;
    if (E > 0 && cudaMemsetAsync(counts, 0, sizeof(int32_t) * E, stream) != cudaSuccess) return RELAY_ECUDA;
    if (h->dme_count &&
        cudaMemsetAsync(h->dme_count, 0, sizeof(int64_t) * h->prog.n, stream) != cudaSuccess)
        return RELAY_ECUDA;
    if (h->d == 0) return RELAY_OK;
    // optimiser state starts at zero (momentum buffer, Adam moments)
    for (float* st : {h->s1, h->s2})
        if (st && cudaMemset2DAsync(st, static_cast<size_t>(h->ld_x) * 4, 0, static_cast<size_t>(4 * h->nquads) * 4,
                                    static_cast<size_t>(h->prog.n), stream) != cudaSuccess)
            return RELAY_ECUDA;
    const int threads = 256;
    relay_init_kernel<<<grid_for(h->nquads, threads), threads, 0, stream>>>(
        x, E > 0 ? msg_a : nullptr, E > 0 ? msg_b : nullptr, h->prog.n, message_rows(h), h->ld_x, h->ld_m, h->nquads,
        h->d, static_cast<uint32_t>(h->c0 / 4), x0_std, philox_key(seed));
    return launch_status();
}

int relay_step_counts(relay_handle* h, int32_t* counts, relay_stream_t stream) {
    if (!h) return RELAY_EINVAL;
    if (h->prog.E == 0 && h->algo != RELAY_ALGO_DME) return RELAY_OK;
    if (!counts && h->prog.E > 0) return RELAY_EINVAL;
    CountWindows<1> cw;
    count_window(h, counts, cw, 0);
    relay_counts_kernel<1><<<1, 256, 0, stream>>>(cw);
    return launch_status();
}

// Adam's bias-corrected factors of step t (k = t + 1), in double.
static void adam_factors(const relay_handle* h, float lr, int64_t step, float* adam_step, float* adam_ibc2) {
    *adam_step = 0.0f;
    *adam_ibc2 = 0.0f;
    if (h->opt != 2) return;
    const double k = static_cast<double>(step) + 1.0;
    *adam_step = static_cast<float>(lr / (1.0 - std::pow(static_cast<double>(h->beta1), k)));
    *adam_ibc2 = static_cast<float>(1.0 / std::sqrt(1.0 - std::pow(static_cast<double>(h->beta2), k)));
}

// The step kernels' arguments for step `step` (checked by check_step_args).
static ModelArgs model_args(const relay_handle* h, float* x, const float* msg_in, float* msg_out,
                            const int32_t* counts, float lr, uint64_t seed, int64_t step) {
    ModelArgs a;
    a.x = x;
    a.mu = h->mu;
    a.msg_in = msg_in;
    a.msg_out = msg_out;
    a.counts = counts;
    a.ld_x = h->ld_x;
    a.ld_m = h->ld_m;
    a.nquads = h->nquads;
    a.q0 = static_cast<uint32_t>(h->c0 / 4);
    a.step = static_cast<uint32_t>(step);
    a.key = philox_key(seed);
    a.lr = lr;
    a.sigma = h->sigma;
    a.mode = h->mode;
    a.algo = h->algo;
    a.has_lost = h->has_lost ? 1 : 0;
    a.rsum = h->prog.nwide > 0 ? 1 : 0;
    std::memcpy(a.lost.w, h->lost, sizeof(a.lost.w));
    a.s1 = h->s1;
    a.s2 = h->s2;
    a.beta1 = h->beta1;
    a.beta2 = h->beta2;
    a.eps = h->eps;
    adam_factors(h, lr, step, &a.adam_step, &a.adam_ibc2);
    return a;
}

// The step kernel's launch; `after_counts`: relay_step's counter kernel was
// just enqueued on `stream`, so the step may start as its programmatic
// dependent.
static int step_models(relay_handle* h, float* x, const float* msg_in, float* msg_out, const int32_t* counts,
                       float lr, uint64_t seed, int64_t step, relay_stream_t stream, bool after_counts) {
    const int rc = check_step_args(h, x, msg_in, msg_out, counts, lr, step);
    if (rc != RELAY_OK) return rc;
    if (h->d == 0) return RELAY_OK;
    const ModelArgs a = model_args(h, x, msg_in, msg_out, counts, lr, seed, step);
    switch (h->opt) {
        case 0: return launch_models_obj<0>(h, a, stream, after_counts);
        case 1: return launch_models_obj<1>(h, a, stream, after_counts);
        default: return launch_models_obj<2>(h, a, stream, after_counts);
    }
}

int relay_step_models(relay_handle* h, float* x, const float* msg_in, float* msg_out,
                      const int32_t* counts, float lr, uint64_t seed, int64_t step,
                      relay_stream_t stream) {
    return step_models(h, x, msg_in, msg_out, counts, lr, seed, step, stream, false);
}

int relay_step(relay_handle* h, float* x, const float* msg_in, float* msg_out, int32_t* counts, float lr,
               uint64_t seed, int64_t step, relay_stream_t stream) {
    // every check of relay_step_models runs before the counter launch, so a
    // rejected step leaves the counters untouched
    int rc = check_step_args(h, x, msg_in, msg_out, counts, lr, step);
    if (rc != RELAY_OK) return rc;
    // relay_step_counts launches only when there are counters to update
    const bool counted = h->prog.E > 0 || h->algo == RELAY_ALGO_DME;
    rc = relay_step_counts(h, counts, stream);
    if (rc != RELAY_OK) return rc;
    return step_models(h, x, msg_in, msg_out, counts, lr, seed, step, stream, counted);
}

// relay_step_windows runs the windows in one launch when both take the walk,
// neither tree has a node of degree > kRegDeg (double binary trees have
// degree <= 3), and they share the objective (its source; the mixture too
// when regenerated) and the local optimiser; otherwise it issues one
// relay_step per window.
static bool one_launch(const relay_handle* a, const relay_handle* b) {
    if (a->d == 0 || b->d == 0 || use_nodes(a) || use_nodes(b) || has_wide(a) || has_wide(b)) return false;
    if (a->opt != b->opt || a->obj.source != b->obj.source) return false;
    return a->obj.source == relaysum::kMuStored || std::memcmp(&a->obj, &b->obj, sizeof(Objective)) == 0;
}

int relay_step_windows(relay_handle* const* h, int32_t count, float* const* x, const float* const* msg_in,
                       float* const* msg_out, int32_t* const* counts, float lr, uint64_t seed, int64_t step,
                       relay_stream_t stream) {
    if (!h || !x || !msg_in || !msg_out || !counts || count < 1 || count > RELAY_MAX_WINDOWS) return RELAY_EINVAL;
    for (int k = 0; k < count; ++k) {
        if (!h[k]) return RELAY_EINVAL;
        for (int j = 0; j < k; ++j)
            if (h[j] == h[k]) return RELAY_EINVAL;
        const int rc = check_step_args(h[k], x[k], msg_in[k], msg_out[k], counts[k], lr, step);
        if (rc != RELAY_OK) return rc;
    }
    if (count == 1 || !one_launch(h[0], h[1])) {
        for (int k = 0; k < count; ++k) {
            const int rc = relay_step(h[k], x[k], msg_in[k], msg_out[k], counts[k], lr, seed, step, stream);
            if (rc != RELAY_OK) return rc;
        }
        return RELAY_OK;
    }
    // the counters of both windows (one CTA each), then the step kernel as
    // its programmatic dependent
    bool counted = false;
    CountWindows<2> cw;
    for (int k = 0; k < 2; ++k) {
        count_window(h[k], counts[k], cw, k);
        counted = counted || h[k]->prog.E > 0 || h[k]->algo == RELAY_ALGO_DME;
    }
    if (counted) {
        relay_counts_kernel<2><<<2, 256, 0, stream>>>(cw);
        const int rc = launch_status();
        if (rc != RELAY_OK) return rc;
    }
    const ModelArgs as[2] = {model_args(h[0], x[0], msg_in[0], msg_out[0], counts[0], lr, seed, step),
                             model_args(h[1], x[1], msg_in[1], msg_out[1], counts[1], lr, seed, step)};
    const relay_handle* const hs[2] = {h[0], h[1]};
    switch (h[0]->opt) {
        case 0: return launch_walk_obj<0, 2>(hs, as, stream, counted);
        case 1: return launch_walk_obj<1, 2>(hs, as, stream, counted);
        default: return launch_walk_obj<2, 2>(hs, as, stream, counted);
    }
}

int relay_get_steps_kernel(const relay_handle* h) {
    if (!h) return RELAY_EINVAL;
    return use_fused(h) ? RELAY_KERNEL_FUSED : relay_get_kernel(h);
}

int relay_steps(relay_handle* h, float* x, float* msg_a, float* msg_b, int32_t* counts, float lr, uint64_t seed,
                int64_t t0, int64_t k, relay_stream_t stream) {
    int rc = check_step_args(h, x, msg_a, msg_b, counts, lr, t0);
    if (rc != RELAY_OK) return rc;
    if (k < 0 || k > (int64_t(1) << 32) - t0) return RELAY_EINVAL;  // step counters stay below 2^32
    float* const buf[2] = {msg_a, msg_b};
    if (!use_fused(h)) {  // a wide node would hold its CTA at every step: one relay_step per step
        for (int64_t j = 0; j < k; ++j) {
            rc = relay_step(h, x, buf[j & 1], buf[(j + 1) & 1], counts, lr, seed, t0 + j, stream);
            if (rc != RELAY_OK) return rc;
        }
        return RELAY_OK;
    }
    const bool counted = h->prog.E > 0 || h->algo == RELAY_ALGO_DME;
    LostMask lost;
    std::memcpy(lost.w, h->lost, sizeof(lost.w));
    for (int64_t done = 0; done < k;) {
        const int kc = static_cast<int>(k - done < kMaxFusedSteps ? k - done : kMaxFusedSteps);
        const int par = static_cast<int>(done & 1);  // step t0 + done reads buf[par]
        if (h->d > 0) {
            const ModelArgs a = model_args(h, x, buf[par], buf[par ^ 1], counts, lr, seed, t0 + done);
            FusedSteps fs;
            fs.k = kc;
            fs.msg[0] = buf[par];
            fs.msg[1] = buf[par ^ 1];
            for (int j = 0; j < kMaxFusedSteps; ++j)
                adam_factors(h, lr, t0 + done + (j < kc ? j : 0), &fs.adam_step[j], &fs.adam_ibc2[j]);
            switch (h->opt) {
                case 0: rc = launch_fused_obj<0>(h, a, fs, stream); break;
                case 1: rc = launch_fused_obj<1>(h, a, fs, stream); break;
                default: rc = launch_fused_obj<2>(h, a, fs, stream); break;
            }
            if (rc != RELAY_OK) return rc;
        }
        // the counters advance after the models kernel, which read them
        if (counted) {
            relay_counts_steps_kernel<<<1, kCountsThreads, 0, stream>>>(h->prog, lost, h->has_lost ? 1 : 0, counts,
                                                             h->algo == RELAY_ALGO_DME ? h->dme_count : nullptr, kc);
            rc = launch_status();
            if (rc != RELAY_OK) return rc;
        }
        done += kc;
    }
    return RELAY_OK;
}

int relay_nbar(const relay_handle* h, const int32_t* counts_host, int32_t* nbar_host) {
    if (!h || !nbar_host || (h->prog.E > 0 && !counts_host)) return RELAY_EINVAL;
    for (int i = 0; i < h->prog.n; ++i) {
        const NodeRec& r = h->prog.node[i];
        int32_t s = 1;
        for (int p = 0; p < r.deg; ++p) s += counts_host[h->prog.pos_in[r.pos_base + p]];
        nbar_host[i] = s;
    }
    return RELAY_OK;
}

int relay_program(const relay_handle* h, int32_t* nslots, int32_t* order, int32_t* node_rec,
                  int32_t* pos_rec) {
    if (!h) return RELAY_EINVAL;
    const Program& p = h->prog;
    if (nslots) *nslots = p.nslots;
    for (int i = 0; i < p.n; ++i) {
        if (order) order[i] = p.order[i];
        if (node_rec) {
            const NodeRec& r = p.node[i];
            const int32_t v[12] = {r.deg,        r.pos_base,   r.parent_pos, r.recv_slot, r.acc_slot,
                                   r.parent_acc, r.fin_parent, r.parent,     r.tot_slot,  r.flags,
                                   p.rsum_slot[i], p.rsum_row[i]};
            std::memcpy(node_rec + 12 * i, v, sizeof(v));
        }
    }
    if (pos_rec)
        for (int e = 0; e < p.E; ++e) {
            pos_rec[4 * e] = p.pos_in[e];
            pos_rec[4 * e + 1] = p.pos_out[e];
            pos_rec[4 * e + 2] = p.pos_slot[e];
            pos_rec[4 * e + 3] = p.rb_in[e];
        }
    return RELAY_OK;
}

int64_t relay_metrics_workspace(const relay_handle* h) {
    if (!h) return RELAY_EINVAL;
    const int64_t blocks = (h->nquads + kMetricsThreads - 1) / kMetricsThreads;
    return 2 * std::max<int64_t>(1, std::min<int64_t>(blocks, kMetricsMaxBlocks));
}

int relay_metrics(relay_handle* h, const float* x, double* workspace, double* out, relay_stream_t stream) {
    if (!h || !h->has_objective || !out || !workspace) return RELAY_EINVAL;
    if (h->d > 0 && (!x || !aligned16(x))) return RELAY_EINVAL;
    const int blocks = static_cast<int>(relay_metrics_workspace(h) / 2);
    ModelArgs a;
    std::memset(&a, 0, sizeof(a));
    a.x = const_cast<float*>(x);
    a.mu = h->mu;
    a.ld_x = h->ld_x;
    a.nquads = h->nquads;
    a.q0 = static_cast<uint32_t>(h->c0 / 4);
    const PhiloxKey mu_key = philox_key(static_cast<uint64_t>(h->obj.k0) | (static_cast<uint64_t>(h->obj.k1) << 32));
    const int n = h->prog.n;
    switch (h->obj.source) {
        case relaysum::kMuStored:
            relay_metrics_kernel<relaysum::kMuStored><<<blocks, kMetricsThreads, 0, stream>>>(
                h->obj, mu_key, a, n, h->d, workspace);
            break;
        default:  // cached centres are regenerated per row here
            relay_metrics_kernel<relaysum::kMuPerRow><<<blocks, kMetricsThreads, 0, stream>>>(
                h->obj, mu_key, a, n, h->d, workspace);
            break;
    }
    const double denom = h->d > 0 ? static_cast<double>(h->d) : 1.0;
    relay_metrics_finish_kernel<<<1, kMetricsThreads, 0, stream>>>(workspace, blocks, 1.0 / (n * denom),
                                                                   1.0 / denom, out);
    return launch_status();
}

// ------------------------------------------- allocation-free metrics variant

// Scratch for relay_metrics_static: the per-block partial sums of the metrics
// reduction, in a file-scope device array instead of a caller workspace.
// Every GPU that loads the library holds it (16 KB) until the process exits.
constexpr int kStaticMetricsDoubles = 2 * kMetricsMaxBlocks;
static __device__ __align__(256) double g_metrics_scratch[kStaticMetricsDoubles];

namespace {
// The array's device address, looked up once per device with that device
// current.  (In host code the array's name is only a host-side stand-in.)
std::atomic<double*> g_metrics_scratch_addr[kMaxDevices];

double* metrics_scratch_address(int dev) {
    double* p = dev < kMaxDevices ? g_metrics_scratch_addr[dev].load() : nullptr;
    if (p) return p;
    if (cudaGetSymbolAddress(reinterpret_cast<void**>(&p), g_metrics_scratch) != cudaSuccess || !p)
        return nullptr;
    if (dev < kMaxDevices) g_metrics_scratch_addr[dev].store(p);
    return p;
}
}  // namespace

int relay_metrics_static(relay_handle* h, const float* x, double* out, relay_stream_t stream) {
    if (!h) return RELAY_EINVAL;
    if (relay_metrics_workspace(h) > kStaticMetricsDoubles) return RELAY_EUNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return RELAY_ECUDA;
    double* scratch = metrics_scratch_address(dev);
    if (!scratch) return RELAY_ECUDA;
    // pass 1 overwrites every partial that pass 2 reads: nothing to clear
    return relay_metrics(h, x, scratch, out, stream);
}

const char* relay_error_string(int status) {
    switch (status) {
        case RELAY_OK: return "ok";
        case RELAY_EINVAL: return "invalid argument";
        case RELAY_ENOTTREE: return "edge list is not a tree";
        case RELAY_ECUDA: return "CUDA launch or runtime error";
        case RELAY_ENOMEM: return "host allocation failed";
        case RELAY_EUNSUPPORTED: return "unsupported size";
        default: return "unknown status";
    }
}

}  // extern "C"
