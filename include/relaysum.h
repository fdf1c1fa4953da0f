/*
 * relaysum.h -- C ABI of the GB300 RelaySum step library (librelaysum.so).
 *
 * One RelaySGD iteration (Vogels et al., "RelaySum for Decentralized Deep
 * Learning on Heterogeneous Data", arXiv 2110.04175, Algorithm 1) for n
 * virtual workers of a spanning tree, all resident on one GPU:
 *
 *   local step     x_i^{t+1/2} = x_i^t - lr * ((x_i^t - mu_i) + sigma * xi_i^t)
 *   relay message  m_{i->j}^t  = x_i^{t+1/2} + sum_{k in N(i)\j} m_{k->i}^{t-1}
 *   counter        c_{i->j}^t  = 1 + sum_{k in N(i)\j} c_{k->i}^{t-1}
 *   models seen    nbar_i      = 1 + sum_{j in N(i)} c_{j->i}^t
 *   rebuild        mode 0 (Alg. 1):  x_i^{t+1} = (x_i^{t+1/2} + sum_j m_{j->i}^t) / nbar_i
 *                  mode 1 (robust rule of Section 4.4):
 *                      x_i^{t+1} = (x_i^{t+1/2} + sum_j m_{j->i}^t + (n - nbar_i) x_i^t) / n
 *
 * The objective is the synthetic heterogeneous quadratic f_i = 1/2||x - mu_i||^2
 * with Philox4x32-10 gradient noise xi (the appendix "Independence of
 * heterogeneity" adds random normal noise to each gradient update).
 *
 * Conventions shared by every call:
 *   - Layout.  x and mu are fp32 [n][ld], messages fp32 [E][ld] with
 *     E = 2(n-1) (more rows with received sums: relay_message_rows),
 *     counters int32 [E]; ld = relay_ld(h) >= d is the padded
 *     row stride (a multiple of 32 floats; relay_set_strides sets others).
 *     The kernels touch columns [0, 4 ceil(d/4)) of each row only; init
 *     zeroes the ragged columns [d, 4 ceil(d/4)), whose values after a step
 *     are unspecified, and never reads or writes columns beyond.
 *     Undirected edge u of the edge list gives directed edges 2u
 *     (edges[2u] -> edges[2u+1]) and 2u+1 (the reverse).
 *   - Ownership.  The caller allocates and owns every device buffer; a
 *     handle owns only its host-side tables.  No call allocates device
 *     memory, and no call synchronises: device work is enqueued on `stream`
 *     (a cudaStream_t; NULL is the legacy default stream) of the current
 *     device.
 *   - Errors.  Every int-returning call returns RELAY_OK (0) or a negative
 *     status; arguments are checked before anything is enqueued, and a
 *     rejected call leaves every buffer untouched.  RELAY_ECUDA reports a
 *     failed launch (cudaGetLastError); no C++ exception crosses the ABI.
 *   - Handles.  A handle's settings (offset, strides, objective, optimiser,
 *     lost messages, ...) are copied into each launch's arguments when a
 *     call enqueues work, so they may be changed between calls without
 *     waiting for the GPU.  A handle is not safe for concurrent use from
 *     several host threads; distinct handles are independent.
 *   - Random numbers.  Philox4x32-10 (Salmon et al., SC'11) with key
 *     (seed lo32, seed hi32) and counter (q, row, step, stream) where q is
 *     the ABSOLUTE coordinate quad (c0 + c) / 4; stream 0 = gradient noise
 *     of worker `row` at `step`, 1 = Gaussian centre `row`, 2 = the shared
 *     initial model.  Words (0,1) and (2,3) become two Box-Muller pairs
 *     for coordinates 4q, 4q+1 and 4q+2, 4q+3, via u = ((w >> 8) + 1) 2^-24.
 */
#ifndef RELAYSUM_H
#define RELAYSUM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RELAY_OK 0
#define RELAY_EINVAL (-1)        /* bad argument (null pointer, range, aliasing) */
#define RELAY_ENOTTREE (-2)      /* the edge list is not a tree on 0..n-1        */
#define RELAY_ECUDA (-3)         /* a CUDA launch or runtime call failed         */
#define RELAY_ENOMEM (-4)        /* host allocation failed                       */
#define RELAY_EUNSUPPORTED (-5)  /* n > RELAY_MAX_N, or a size beyond the limits */

#define RELAY_MAX_N 256          /* workers per handle                            */

typedef struct relay_handle relay_handle;
typedef struct CUstream_st *relay_stream_t; /* identical to cudaStream_t */

/* Creates a handle for n >= 1 workers with d >= 0 parameters each on the
 * tree given by n_edges = n - 1 undirected pairs `edges` (host, int32
 * [n_edges][2], ids in 0..n-1).  Validates that the pairs form a tree
 * (Section 3 "Setup": no self loops; Alg. 1 runs on a tree) and builds the
 * per-node visit program of the fused kernel.  Host work only: no CUDA call.
 * Errors: RELAY_EINVAL (out == NULL, d < 0, d with (d+31)/4 >= 2^32 quads),
 * RELAY_ENOTTREE, RELAY_EUNSUPPORTED (n > RELAY_MAX_N), RELAY_ENOMEM. */
int relay_create(relay_handle **out, int32_t n, int64_t d, const int32_t *edges,
                 int32_t n_edges);

/* Releases a handle (NULL is allowed).  Device buffers are the caller's. */
void relay_destroy(relay_handle *h);

/* Padded row stride in floats: d rounded up to a multiple of 32. */
int64_t relay_ld(const relay_handle *h);

/* Number of directed edges E = 2(n-1) (rows of a message buffer). */
int32_t relay_num_edges(const relay_handle *h);

/* Directed edge table: src[e] -> dst[e] for e < E (host int32 [E] each).
 * Edge 2u is edges[u][0] -> edges[u][1], edge 2u+1 its reverse. */
int relay_edges(const relay_handle *h, int32_t *src, int32_t *dst);

/* Row strides (floats) of x / mu and of the message buffers, for a handle
 * working on a column window of wider arrays (for example the two trees of
 * a double binary tree, each owning half the coordinates of one model
 * array).  Each must be a multiple of 4 and >= 4 ceil(d / 4); pointers
 * passed to later calls must stay 16-byte aligned.  Default: relay_ld(h). */
int relay_set_strides(relay_handle *h, int64_t ld_x, int64_t ld_msg);

#define RELAY_OPT_SGD 0       /* x^{t+1/2} = x^t - lr g                                  */
#define RELAY_OPT_NESTEROV 1  /* m = beta1 m + g; x^{t+1/2} = x^t - lr (g + beta1 m)     */
#define RELAY_OPT_ADAM 2      /* PyTorch's Adam (no weight decay), bias-corrected at t+1 */

/* Local optimiser of Alg. 1's local step (appendix "RelaySGD with
 * momentum", "RelaySGD with Adam"; all state is local to each worker).
 * state1 (Nesterov: m; Adam: first moment) and state2 (Adam: second moment)
 * are caller-owned device fp32 [n][ld_x] arrays with the stride of x,
 * read and written by every step; relay_init zeroes them.  Nesterov needs
 * 0 <= beta1 < 1; Adam 0 <= beta1, beta2 < 1 and eps > 0.  Default SGD. */
int relay_set_local_optimizer(relay_handle *h, int32_t kind, float beta1, float beta2, float eps,
                              float *state1, float *state2);

#define RELAY_ALGO_RELAYSGD 0  /* Algorithm 1: x' = rebuild of x^{t+1/2} and the messages      */
#define RELAY_ALGO_GRAD 1      /* Algorithm 6: relay the update u; x' = x + (u + sum m) / n    */
#define RELAY_ALGO_DME 2       /* Algorithm 5: relay samples mu + sigma xi; x holds y += ...  */

/* Which algorithm runs on the relay (appendix "RelaySum for distributed mean
 * estimation", "Alternative optimizer based on RelaySum").  For RELAY_ALGO_DME
 * x holds the running sums y_i, the samples are mu_i + sigma xi_i^t (the
 * objective's centres and noise), and dme_count (device int64 [n], zeroed by
 * relay_init) accumulates s_i += 1 + sum_j c^t_{j->i} at every step; the
 * estimate of worker i is y_i / s_i.  RELAY_ALGO_GRAD needs no counters (they
 * are still maintained).  Default RELAY_ALGO_RELAYSGD. */
int relay_set_algorithm(relay_handle *h, int32_t algo, int64_t *dme_count);

/* Messages lost in transit (Section 4.4, "Robustness to unreliable
 * communication"): host uint8 [E], non-zero = the message sent on that
 * directed edge by every later step never arrives, so its receiver reads
 * m = 0 and c = 0 (and relays those).  NULL clears.  The mask is copied into
 * the launch arguments of each step: change it between steps freely. */
int relay_set_lost_messages(relay_handle *h, const uint8_t *lost);

/* Rebuild rule: 0 = Algorithm 1 (divide by nbar), 1 = robust rule of
 * Section 4.4 (fill the n - nbar missing models with x_i^t, divide by n).
 * The default is 1. */
int relay_set_rebuild_mode(relay_handle *h, int32_t mode);

/* Which kernel runs the fused step (an implementation choice: the paper's
 * Algorithm 1 fixes only what is computed).  RELAY_KERNEL_WALK: one thread
 * per quad of coordinates walks every worker of the tree in turn.
 * RELAY_KERNEL_NODES: one thread per (worker, quad), the new messages meeting
 * in shared memory; it uses n times more threads, which pays off when d is
 * short.  Both form every sum in the same order, so their results are
 * identical bit for bit.  RELAY_KERNEL_AUTO (the default) takes NODES when
 * n * ceil(d/4) < 2^21 and no worker has more than 4 neighbours (where it
 * measured faster), WALK otherwise.  Errors: RELAY_EINVAL for another value. */
#define RELAY_KERNEL_AUTO 0
#define RELAY_KERNEL_WALK 1
#define RELAY_KERNEL_NODES 2
int relay_set_kernel(relay_handle *h, int32_t kernel);

/* The kernel the next step of this handle launches: RELAY_KERNEL_WALK or
 * RELAY_KERNEL_NODES (RELAY_KERNEL_AUTO resolved), or RELAY_EINVAL. */
int relay_get_kernel(const relay_handle *h);

/* Received sums (an implementation choice; Algorithm 1 fixes only what is
 * computed).  A worker i with more than 4 neighbours ("wide", such as a
 * star's hub) sends every neighbour j the message x_i^{t+1/2} + S_i^{t-1} -
 * m^{t-1}_{j->i}, where S_i^{t-1} = sum_k m^{t-1}_{k->i} is the sum of the
 * messages it received at step t-1 -- the sum Alg. 1's rebuild line formed
 * in that step.  With enable = 1 every message buffer carries, after its E
 * message rows, one row per wide node (in ascending worker id) holding that
 * sum for the messages in the buffer: relay_step reads S_i^{t-1} from
 * msg_in's row and writes S_i^t to msg_out's, so each incoming message row
 * is read once per step instead of twice.  Buffers then have
 * relay_message_rows(h) rows; relay_init zeroes them all, and msg_in must
 * be a buffer that relay_init or a relay_step of this handle wrote (or one
 * whose sum rows the caller keeps equal to the sums of its message rows).
 * The models and messages agree with the default path within rounding (the
 * same sums, summed in another order) and the counters are identical.
 * Rebuilds the handle's visit program (host work only).  Default 0.
 * Errors: RELAY_EINVAL unless enable is 0 or 1; RELAY_EUNSUPPORTED if the
 * walk would need more than 127 slots. */
int relay_set_received_sums(relay_handle *h, int32_t enable);

/* Rows of a message buffer: E, plus one per wide node when received sums
 * are on (relay_set_received_sums); RELAY_EINVAL for a NULL handle. */
int32_t relay_message_rows(const relay_handle *h);

/* Absolute index of this handle's first coordinate within a longer model
 * vector (c0 >= 0, a multiple of 4): the noise of local coordinate c is
 * that of coordinate c0 + c, so a vector split into slices -- across GPUs,
 * or for spot checks -- reproduces the unsplit run exactly.  Default 0. */
int relay_set_coord_offset(relay_handle *h, int64_t c0);

/* Binds the objective used by every later step: mu is a caller-owned device
 * fp32 [n][ld] array of quadratic centres (read, never written; it must stay
 * valid while steps using it run), sigma >= 0 the gradient-noise std. */
int relay_set_objective(relay_handle *h, const float *mu, float sigma);

/* Binds the same objective without a mu array: the fused kernel regenerates
 * mu_i(c) = mu_scale * sum_k mix[i][k] N_k(c) on the fly (Gaussian centres
 * N_k from Philox stream 1, row k), bit-identical to what
 * relay_fill_objective writes, so a step reads 4 n d fewer bytes.  mix is a
 * HOST fp32 [n][K] matrix, copied (its non-zeros) into the handle; sigma >= 0
 * the gradient-noise std.  RELAY_EUNSUPPORTED if mix has more than 1024
 * non-zeros. */
int relay_set_objective_generated(relay_handle *h, const float *mix, int32_t K, float mu_scale,
                                  uint64_t mu_seed, float sigma);

/* Fills mu (device fp32 [n][ld]) with mu_i(c) = mu_scale * sum_k
 * mix[i][k] N_k(c): K Gaussian centres N_k (Philox stream 1, row k) mixed by
 * the device fp32 [n][K] matrix `mix` (identity for one centre per worker,
 * Dirichlet rows for a mixture). */
int relay_fill_objective(relay_handle *h, float *mu, const float *mix, int32_t K,
                         float mu_scale, uint64_t mu_seed, relay_stream_t stream);

/* Initial state of Algorithm 1: x_i^0 = x0_std * N(c) for every worker (one
 * shared draw, Philox stream 2), m^{-1} = 0 in msg_a (and in msg_b unless it
 * is NULL), c^{-1} = 0.  x: device [n][ld]; msg_a, msg_b: device [E][ld];
 * counts: device int32 [E]. */
int relay_init(relay_handle *h, float *x, float *msg_a, float *msg_b, int32_t *counts,
               float x0_std, uint64_t seed, relay_stream_t stream);

/* Counter update of Alg. 1 in place: counts c^{t-1} -> c^t (int32 [E]).
 * Integer, bit-exact.  One 1-CTA launch. */
int relay_step_counts(relay_handle *h, int32_t *counts, relay_stream_t stream);

/* The per-coordinate part of iteration t in one fused pass over d: local
 * step, every outgoing relay message and the rebuild, for all workers.
 * counts must already hold c^t (relay_step_counts ran first); they give
 * nbar.  x: device [n][ld] in/out (x^t -> x^{t+1}); msg_in: [E][ld] m^{t-1}
 * (read only); msg_out: [E][ld] m^t (written); msg_in != msg_out, and
 * neither may overlap x.  lr finite; step in [0, 2^32) is the noise
 * counter.  RELAY_EINVAL also when no objective is bound. */
int relay_step_models(relay_handle *h, float *x, const float *msg_in, float *msg_out,
                       const int32_t *counts, float lr, uint64_t seed, int64_t step,
                       relay_stream_t stream);

/* One full RelaySGD iteration t: relay_step_counts, then
 * relay_step_models, enqueued back to back on `stream`.  The step kernel is
 * launched as a programmatic dependent of the counter kernel: it may be
 * scheduled while the counter kernel runs and waits for it before reading
 * the counters (relay_step_models called alone is an ordinary launch).  The
 * caller swaps msg_in and msg_out before the next step (double-buffered
 * messages). */
int relay_step(relay_handle *h, float *x, const float *msg_in, float *msg_out,
               int32_t *counts, float lr, uint64_t seed, int64_t step,
               relay_stream_t stream);

/* One RelaySGD iteration t of `count` (1 or 2) handles that split the
 * coordinates of the same workers into windows -- the double binary trees of
 * Section 3 ("Spanning trees"): two trees over the n workers, each carrying
 * half of every model's coordinates, so every worker sends and receives two
 * half-size messages per step.  The result is that of relay_step(h[k],
 * x[k], msg_in[k], msg_out[k], counts[k], lr, seed, step, stream) for
 * k = 0 .. count-1, bit for bit.  When both handles take the walk kernel and
 * share the objective (the same source; the same mixture when regenerated)
 * and the local optimiser, their counters are updated by one launch and
 * their steps by one launch of the step kernel, whose CTAs split between the
 * windows; otherwise the relay_step calls are issued one after the other.
 * h, x, msg_in, msg_out, counts: host arrays of `count` entries, each
 * entry as relay_step takes it (a window's x is usually a column offset
 * into one model array, with relay_set_strides giving the full row
 * stride; the caller keeps the windows' columns disjoint).  Errors: those of
 * relay_step for any window, checked for every window before anything is
 * enqueued, and RELAY_EINVAL for count outside [1, RELAY_MAX_WINDOWS], a
 * NULL array or the same handle twice. */
#define RELAY_MAX_WINDOWS 2
int relay_step_windows(relay_handle *const *h, int32_t count, float *const *x,
                       const float *const *msg_in, float *const *msg_out, int32_t *const *counts,
                       float lr, uint64_t seed, int64_t step, relay_stream_t stream);

/* k consecutive iterations t0, t0+1, ..., t0+k-1 of Algorithm 1 (k >= 0),
 * equal bit for bit to k relay_step calls that alternate the two message
 * buffers: iteration t0+j reads msg_a if j is even (msg_b if odd) and writes
 * the other.  On entry msg_a holds m^{t0-1}; on return the buffer written
 * last holds m^{t0+k-1} (msg_b if k is odd, msg_a if even), the other one
 * m^{t0+k-2} (k >= 2), counts hold c^{t0+k-1}, and x, the optimiser state
 * and the mean-estimation counts have advanced k steps.  The lost-message
 * mask in force applies to every one of the k steps.  Every coordinate
 * evolves on its own, so the steps run without a round trip through HBM:
 * each CTA keeps its quads' models and optimiser state in registers and
 * their messages in shared memory for up to 64 steps per launch (then a
 * 1-CTA launch advances the counters).  That multi-step kernel is taken under
 * RELAY_KERNEL_NODES, and under RELAY_KERNEL_AUTO when no worker has more
 * than 4 neighbours; otherwise (RELAY_KERNEL_WALK, or a wide node such as a
 * star's hub, whose threads would hold their CTA at every step) relay_steps
 * enqueues k relay_step calls.  Arguments and errors as relay_step
 * (x, msg_a, msg_b, counts, lr, seed; t0 the noise counter of the first
 * step), plus RELAY_EINVAL when k < 0 or t0 + k > 2^32.  The buffers are
 * caller-owned device memory; nothing is allocated. */
int relay_steps(relay_handle *h, float *x, float *msg_a, float *msg_b, int32_t *counts,
                float lr, uint64_t seed, int64_t t0, int64_t k, relay_stream_t stream);

/* ---- State in host memory --------------------------------------------
 *
 * A state larger than the GPU, or owned by the host, can stay in page-locked
 * host memory: x [n][ld_x], the message buffers [relay_message_rows][ld_msg]
 * and the counters [E], in the same layout as on the device (the handle's
 * strides), allocated with cudaHostAlloc / cudaMallocHost or registered
 * with cudaHostRegister.  A step streams the coordinates through the GPU in
 * chunks of `chunk` coordinates: each chunk's x and message rows are copied
 * in, stepped by the fused kernel at the chunk's absolute coordinate offset,
 * and copied back, with the copies in both directions and the kernels
 * overlapped on the plan's own streams.  Every coordinate of Algorithm 1
 * evolves on its own and the noise is keyed by the absolute coordinate, so
 * the result equals relay_step on the resident state bit for bit.  The
 * handle must use regenerated centres (relay_set_objective_generated) and
 * the SGD local step: a device mu array or optimiser state has no place in
 * a host-state step (RELAY_EUNSUPPORTED otherwise).
 *
 * Copies: only the message rows a step reads go in -- every row except
 * those arriving at a leaf, whose one outgoing message excludes its one
 * incoming one -- and the same rows come back (the state the next step
 * needs), unless the plan was created with RELAY_HOST_FULL_OUTPUT, which
 * copies every row of m^t back, as relay_step writes it.  The rows not
 * copied back keep whatever the host buffer held.  x and the counters are
 * copied both ways.  msg_in may equal msg_out: each chunk is read before it
 * is written, and chunks do not overlap.
 *
 * Ordering: a step starts after the work already enqueued on `stream` and
 * `stream` waits for all of it, so the host arrays may be read after
 * cudaStreamSynchronize(stream); consecutive steps on the same stream are
 * ordered.  The plan's streams and events are created by
 * relay_host_plan_create; relay_step_host and relay_steps_host allocate
 * nothing and issue one cudaMemcpy2DAsync per array and run of rows per
 * chunk.  A plan and its staging serve one step at a time. */
typedef struct relay_host_plan relay_host_plan;
#define RELAY_HOST_FULL_OUTPUT 1

/* Device staging bytes relay_host_plan_create needs for `buffers` (2..8)
 * staging sets of one chunk (chunk a positive multiple of 32 coordinates;
 * capped at d rounded up to 32): (n + 2 rows) * chunk floats per set, plus
 * the counters.  RELAY_EINVAL for bad arguments. */
int64_t relay_host_staging_bytes(const relay_handle *h, int64_t chunk, int32_t buffers);

/* Creates a plan for handle h on the current device: `staging` is
 * caller-owned device memory (256-byte aligned, at least
 * relay_host_staging_bytes) that the plan uses until destroyed; flags 0 or
 * RELAY_HOST_FULL_OUTPUT.  Creates three non-blocking streams and the
 * events that order them.  The plan reads h's settings at every step: keep
 * h alive while the plan is in use.  Errors: RELAY_EINVAL, RELAY_ENOMEM,
 * RELAY_ECUDA. */
int relay_host_plan_create(relay_host_plan **out, relay_handle *h, int64_t chunk, int32_t buffers,
                           void *staging, int64_t staging_bytes, int32_t flags);

/* Releases the plan's streams and events (NULL allowed); the staging memory
 * is the caller's. */
void relay_host_plan_destroy(relay_host_plan *p);

/* Bytes one relay_step_host copies host-to-device and device-to-host. */
int relay_host_bytes(const relay_host_plan *p, int64_t *h2d, int64_t *d2h);

/* relay_step on a state in host memory (see above): x (in/out), msg_in =
 * m^{t-1}, msg_out <- m^t, counts c^{t-1} -> c^t, all page-locked host
 * arrays; lr, seed and step as relay_step.  Errors: RELAY_EINVAL (NULL or
 * pageable host array, another device than the plan's, step out of range,
 * no objective), RELAY_EUNSUPPORTED (a stored mu or an optimiser with
 * state), RELAY_ECUDA. */
int relay_step_host(relay_host_plan *p, float *x, const float *msg_in, float *msg_out, int32_t *counts,
                    float lr, uint64_t seed, int64_t step, relay_stream_t stream);

/* k steps t0 .. t0+k-1 per chunk visit (relay_steps on each chunk), so the
 * state crosses the host link once per k steps: x, msg_in = m^{t0-1} and
 * counts c^{t0-1} go in, x, msg_out <- m^{t0+k-1} and c^{t0+k-1} come back
 * (the intermediate messages stay on the device).  Every chunk starts from
 * the same host counters.  The result equals k relay_step_host calls on x,
 * the counters and m^{t0+k-1}.  RELAY_EUNSUPPORTED for mean estimation
 * (its counts would advance once per chunk); otherwise as relay_step_host. */
int relay_steps_host(relay_host_plan *p, float *x, const float *msg_in, float *msg_out, int32_t *counts,
                     float lr, uint64_t seed, int64_t t0, int64_t k, relay_stream_t stream);

/* The path relay_steps takes on this handle: RELAY_KERNEL_FUSED (several
 * steps per launch), else the per-step kernel of relay_get_kernel; or
 * RELAY_EINVAL. */
#define RELAY_KERNEL_FUSED 3
int relay_get_steps_kernel(const relay_handle *h);

/* nbar_i = 1 + sum of the counters arriving at i, from host counters
 * (int32 [E]) into nbar_host (int32 [n]).  Host arithmetic only. */
int relay_nbar(const relay_handle *h, const int32_t *counts_host, int32_t *nbar_host);

/* Introspection of the fused kernel's visit program (for tests and tools):
 * number of shared-memory accumulator slots per thread, the visit order
 * (int32 [n]), per node 12 ints {deg, pos_base, parent_pos, recv_slot,
 * acc_slot, parent_acc, fin_parent, parent, tot_slot, flags, rsum_slot,
 * rsum_row} (int32 [n][12]; flags bit 0: recv_slot holds the parent's
 * total; the last two are -1 unless the node is wide and received sums are
 * on: the slot of its running sum and its sum row, message row
 * E + rsum_row) and per position 4 ints
 * {in_edge, out_edge, slot, rebuild_in_edge} (int32 [E][4]; the last lists
 * each worker's incoming edges in the order its rebuild adds them); any
 * output pointer may be NULL. */
int relay_program(const relay_handle *h, int32_t *nslots, int32_t *order, int32_t *node_rec,
                  int32_t *pos_rec);

/* Convergence metrics of the current models x (device [n][ld_x]): out[0] =
 * the consensus distance 1/(n d) sum_i ||x_i - xbar||^2, out[1] = the
 * distance of the average model to the optimum ||xbar - mubar||^2 / d, where
 * xbar, mubar are the worker averages (the quantities of Section 4's
 * analysis; mubar is the optimum of f = 1/n sum_i f_i).  out: device double
 * [2]; workspace: device double [relay_metrics_workspace(h)], caller-owned
 * scratch for per-block partial sums, overwritten by every call.  Reduced in
 * double in a fixed order: deterministic.  Needs a bound objective. */
int64_t relay_metrics_workspace(const relay_handle *h);
int relay_metrics(relay_handle *h, const float *x, double *workspace, double *out,
                  relay_stream_t stream);

/* relay_metrics without a workspace argument, for callers that cannot
 * allocate device memory: code that runs while a CUDA graph is being
 * captured in global mode (where cudaMalloc is refused), or a host that
 * hands all device memory to its own pool and gives a plug-in none.  The
 * per-block partial sums go to a scratch array of 2 x 1024 doubles (16 KB)
 * built into the library, which every GPU that loads the library holds until
 * the process exits; nothing is allocated, and each call overwrites every
 * partial it reads, so no state carries over between calls.  The first call
 * on a device looks the array's address up (cudaGetSymbolAddress) with that
 * device current, so make it before any stream capture.  The caller still
 * passes x and out (device double [2]).  All calls share the one array:
 * calls whose work overlaps on the GPU (different streams, or different
 * host threads) race, so order them.  RELAY_EUNSUPPORTED if the reduction
 * would need more than 1024 partial blocks (it never does: the block count
 * is capped there).  The paper has no counterpart: this is a library
 * convenience. */
int relay_metrics_static(relay_handle *h, const float *x, double *out, relay_stream_t stream);

/* Static description of a status code. */
const char *relay_error_string(int status);

#ifdef __cplusplus
}
#endif

#endif /* RELAYSUM_H */
