// host_step.cpp -- RelaySGD steps on a state held in host memory.
//
// The models, messages and counters of Algorithm 1 may live in the host's
// (pinned) memory, for a state larger than the GPU or owned by the host.  A
// step then streams the coordinates through the GPU in chunks: every
// coordinate of the method evolves on its own and the noise is keyed by the
// absolute coordinate, so a chunk stepped by relay_step_models on a handle
// whose coordinate offset is the chunk's position gives exactly the bits of a
// step on the whole resident vector.  The counters are per edge, not per
// coordinate: they are stepped once, before the chunks.
//
// Per chunk c (staging set b = c mod B): the copy-in stream brings x and the
// message rows the step reads into set b, the compute stream runs the step
// kernel on them, and the copy-out stream writes x and the new message rows
// back, so both copy directions and the kernels overlap.  Each set is reused
// only after its previous chunk has been copied out.  All copies are
// cudaMemcpy2DAsync / cudaMemcpyAsync calls on page-locked host memory, one
// per array and contiguous run of rows; the plan's streams and events are
// created once, with the plan, and a step allocates nothing.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <new>
#include <utility>
#include <vector>

#include "handle.h"
#include "program.h"
#include "relaysum.h"

namespace {

constexpr int kMaxBuffers = 8;

// rows [lo, hi) of a message buffer
using RowRun = std::pair<int, int>;

std::vector<RowRun> runs_of(const std::vector<char>& take) {
    std::vector<RowRun> out;
    for (int e = 0; e < static_cast<int>(take.size()); ++e) {
        if (!take[e]) continue;
        if (!out.empty() && out.back().second == e) {
            out.back().second = e + 1;
        } else {
            out.emplace_back(e, e + 1);
        }
    }
    return out;
}

bool pinned_host(const void* p) {
    cudaPointerAttributes attr;
    if (cudaPointerGetAttributes(&attr, p) != cudaSuccess) {
        (void)cudaGetLastError();
        return false;
    }
    return attr.type == cudaMemoryTypeHost;
}

}  // namespace

struct relay_host_plan {
    relay_handle* h = nullptr;   // the caller's handle: its settings are read at every step
    relay_handle* hc = nullptr;  // the chunk handles: full width, and the ragged last chunk
    relay_handle* hl = nullptr;
    int64_t cw = 0, nchunks = 0, last_w = 0;
    int nbuf = 0, flags = 0, n = 0, E = 0, rows = 0, dev = 0;
    std::vector<RowRun> in_runs, out_runs;  // message rows copied in / out
    float* xb[kMaxBuffers] = {};
    float* mib[kMaxBuffers] = {};
    float* mob[kMaxBuffers] = {};
    int32_t* counts_d = nullptr;
    cudaStream_t s_in = nullptr, s_out = nullptr, s_comp = nullptr;
    cudaEvent_t in_done[kMaxBuffers] = {}, comp_done[kMaxBuffers] = {}, out_done[kMaxBuffers] = {};
    cudaEvent_t start = nullptr, comp_end = nullptr, out_end = nullptr;
};

namespace {

int64_t staging_bytes(int n, int rows, int E, int64_t cw, int nbuf) {
    const int64_t set = (static_cast<int64_t>(n) + 2 * static_cast<int64_t>(rows)) * cw * 4;
    return nbuf * set + (static_cast<int64_t>(E) * 4 + 255) / 256 * 256;
}

void destroy(relay_host_plan* p) {
    if (!p) return;
    for (int b = 0; b < kMaxBuffers; ++b)
        for (cudaEvent_t ev : {p->in_done[b], p->comp_done[b], p->out_done[b]})
            if (ev) cudaEventDestroy(ev);
    for (cudaEvent_t ev : {p->start, p->comp_end, p->out_end})
        if (ev) cudaEventDestroy(ev);
    for (cudaStream_t s : {p->s_in, p->s_out, p->s_comp})
        if (s) cudaStreamDestroy(s);
    delete p->hc;
    delete p->hl;
    delete p;
}

// The chunk handles take the caller's current settings, with the chunk's
// width, strides and coordinate offset.
void refresh(relay_host_plan* p) {
    *p->hc = *p->h;
    p->hc->ld = p->hc->ld_x = p->hc->ld_m = p->cw;
    *p->hl = *p->hc;
    p->hc->d = std::min<int64_t>(p->cw, p->h->d);
    p->hc->nquads = (p->hc->d + 3) / 4;
    p->hl->d = p->last_w;
    p->hl->nquads = (p->last_w + 3) / 4;
}

relay_handle* chunk_handle(relay_host_plan* p, int64_t c) {
    relay_handle* hc = (c == p->nchunks - 1) ? p->hl : p->hc;
    hc->c0 = p->h->c0 + c * p->cw;
    return hc;
}

int cuda(cudaError_t e) { return e == cudaSuccess ? RELAY_OK : RELAY_ECUDA; }

// Copies rows of chunk c between the host array (row stride ld floats) and
// a staging array (row stride cw floats), `bytes` per row.
int copy_rows(float* dst, int64_t dpitch, const float* src, int64_t spitch, int64_t bytes, int rows,
              cudaMemcpyKind kind, cudaStream_t s) {
    if (rows <= 0 || bytes <= 0) return RELAY_OK;
    return cuda(cudaMemcpy2DAsync(dst, dpitch * 4, src, spitch * 4, bytes, rows, kind, s));
}

// Arguments shared by relay_step_host and relay_steps_host.
int check_host_args(relay_host_plan* p, const float* x, const float* msg_in, const float* msg_out,
                    const int32_t* counts, float lr) {
    if (!p || !p->h) return RELAY_EINVAL;
    const relay_handle* h = p->h;
    if (!h->has_objective || !std::isfinite(lr)) return RELAY_EINVAL;
    // device-resident inputs have no place in a host-state step
    if (h->obj.source == relaysum::kMuStored || h->opt != RELAY_OPT_SGD) return RELAY_EUNSUPPORTED;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev != p->dev) return RELAY_EINVAL;
    if (p->E > 0 && !counts) return RELAY_EINVAL;
    if (h->d == 0) return RELAY_OK;
    if (!x || (p->E > 0 && (!msg_in || !msg_out))) return RELAY_EINVAL;
    for (const void* q : {static_cast<const void*>(x), static_cast<const void*>(msg_in),
                          static_cast<const void*>(msg_out), static_cast<const void*>(counts)})
        if (q && !pinned_host(q)) return RELAY_EINVAL;
    return RELAY_OK;
}

// Enqueues the copy-in of chunk c into set b (x and the message rows of
// `msg`) on the copy-in stream.
int chunk_in(relay_host_plan* p, int64_t c, int b, const float* x, const float* msg) {
    const relay_handle* h = p->h;
    const int64_t w = (c == p->nchunks - 1) ? p->last_w : p->cw;
    const int64_t bytes = 4 * ((w + 3) / 4 * 4);  // the kernels touch whole quads
    int rc = cuda(cudaStreamWaitEvent(p->s_in, p->out_done[b], 0));
    if (rc == RELAY_OK) rc = copy_rows(p->xb[b], p->cw, x + c * p->cw, h->ld_x, bytes, p->n, cudaMemcpyHostToDevice, p->s_in);
    for (const RowRun& r : p->in_runs) {
        if (rc != RELAY_OK) break;
        rc = copy_rows(p->mib[b] + r.first * p->cw, p->cw, msg + r.first * h->ld_m + c * p->cw, h->ld_m, bytes,
                       r.second - r.first, cudaMemcpyHostToDevice, p->s_in);
    }
    if (rc == RELAY_OK) rc = cuda(cudaEventRecord(p->in_done[b], p->s_in));
    return rc;
}

// Enqueues the copy-out of chunk c from set b (x and the message rows of the
// staging array `mdev`) once the compute stream has finished with it.
int chunk_out(relay_host_plan* p, int64_t c, int b, float* x, float* msg, const float* mdev) {
    const relay_handle* h = p->h;
    const int64_t w = (c == p->nchunks - 1) ? p->last_w : p->cw;
    const int64_t bytes = 4 * ((w + 3) / 4 * 4);
    int rc = cuda(cudaEventRecord(p->comp_done[b], p->s_comp));
    if (rc == RELAY_OK) rc = cuda(cudaStreamWaitEvent(p->s_out, p->comp_done[b], 0));
    if (rc == RELAY_OK) rc = copy_rows(x + c * p->cw, h->ld_x, p->xb[b], p->cw, bytes, p->n, cudaMemcpyDeviceToHost, p->s_out);
    for (const RowRun& r : p->out_runs) {
        if (rc != RELAY_OK) break;
        rc = copy_rows(msg + r.first * h->ld_m + c * p->cw, h->ld_m, mdev + r.first * p->cw, p->cw, bytes,
                       r.second - r.first, cudaMemcpyDeviceToHost, p->s_out);
    }
    if (rc == RELAY_OK) rc = cuda(cudaEventRecord(p->out_done[b], p->s_out));
    return rc;
}

// The caller's stream waits for everything the step enqueued.
int join(relay_host_plan* p, cudaStream_t stream) {
    int rc = cuda(cudaEventRecord(p->comp_end, p->s_comp));
    if (rc == RELAY_OK) rc = cuda(cudaEventRecord(p->out_end, p->s_out));
    if (rc == RELAY_OK) rc = cuda(cudaStreamWaitEvent(stream, p->comp_end, 0));
    if (rc == RELAY_OK) rc = cuda(cudaStreamWaitEvent(stream, p->out_end, 0));
    return rc;
}

// The plan's streams start after the work already on the caller's stream.
int fork(relay_host_plan* p, cudaStream_t stream) {
    int rc = cuda(cudaEventRecord(p->start, stream));
    for (cudaStream_t s : {p->s_in, p->s_comp, p->s_out})
        if (rc == RELAY_OK) rc = cuda(cudaStreamWaitEvent(s, p->start, 0));
    return rc;
}

}  // namespace

extern "C" {

int64_t relay_host_staging_bytes(const relay_handle* h, int64_t chunk, int32_t buffers) {
    if (!h || chunk <= 0 || (chunk & 31) || buffers < 2 || buffers > kMaxBuffers) return RELAY_EINVAL;
    const int64_t cw = std::min<int64_t>(chunk, std::max<int64_t>(32, (h->d + 31) / 32 * 32));
    return staging_bytes(h->prog.n, h->prog.E + h->prog.nwide, h->prog.E, cw, buffers);
}

int relay_host_plan_create(relay_host_plan** out, relay_handle* h, int64_t chunk, int32_t buffers, void* staging,
                           int64_t bytes, int32_t flags) {
    if (!out) return RELAY_EINVAL;
    *out = nullptr;
    const int64_t need = relay_host_staging_bytes(h, chunk, buffers);
    if (need < 0) return static_cast<int>(need);
    if ((flags & ~RELAY_HOST_FULL_OUTPUT) != 0) return RELAY_EINVAL;
    if (!staging || (reinterpret_cast<uintptr_t>(staging) & 255) || bytes < need) return RELAY_EINVAL;
    relay_host_plan* p = new (std::nothrow) relay_host_plan;
    if (!p) return RELAY_ENOMEM;
    p->h = h;
    p->hc = new (std::nothrow) relay_handle;
    p->hl = new (std::nothrow) relay_handle;
    if (!p->hc || !p->hl) {
        destroy(p);
        return RELAY_ENOMEM;
    }
    p->cw = std::min<int64_t>(chunk, std::max<int64_t>(32, (h->d + 31) / 32 * 32));
    p->nchunks = std::max<int64_t>(1, (h->d + p->cw - 1) / p->cw);
    p->last_w = h->d - (p->nchunks - 1) * p->cw;
    p->nbuf = buffers;
    p->flags = flags;
    p->n = h->prog.n;
    p->E = h->prog.E;
    p->rows = h->prog.E + h->prog.nwide;
    // rows a step reads: every message row but those arriving at a leaf (a
    // leaf's only outgoing message excludes its only incoming one), and every
    // received-sum row; the copy-out takes the same rows (the state a later
    // step needs), or every row with RELAY_HOST_FULL_OUTPUT
    try {
        std::vector<char> read(p->rows, 1);
        for (int i = 0; i < p->n; ++i)
            if (h->prog.node[i].deg == 1) read[h->prog.pos_in[h->prog.node[i].pos_base]] = 0;
        p->in_runs = runs_of(read);
        p->out_runs = (flags & RELAY_HOST_FULL_OUTPUT) ? runs_of(std::vector<char>(p->rows, 1)) : p->in_runs;
    } catch (...) {
        destroy(p);
        return RELAY_ENOMEM;
    }
    char* base = static_cast<char*>(staging);
    const int64_t set = (static_cast<int64_t>(p->n) + 2 * static_cast<int64_t>(p->rows)) * p->cw * 4;
    for (int b = 0; b < buffers; ++b) {
        p->xb[b] = reinterpret_cast<float*>(base + b * set);
        p->mib[b] = p->xb[b] + static_cast<int64_t>(p->n) * p->cw;
        p->mob[b] = p->mib[b] + static_cast<int64_t>(p->rows) * p->cw;
    }
    p->counts_d = reinterpret_cast<int32_t*>(base + buffers * set);
    int rc = cuda(cudaGetDevice(&p->dev));
    for (cudaStream_t* s : {&p->s_in, &p->s_out, &p->s_comp})
        if (rc == RELAY_OK) rc = cuda(cudaStreamCreateWithFlags(s, cudaStreamNonBlocking));
    for (int b = 0; b < buffers && rc == RELAY_OK; ++b)
        for (cudaEvent_t* ev : {&p->in_done[b], &p->comp_done[b], &p->out_done[b]})
            if (rc == RELAY_OK) rc = cuda(cudaEventCreateWithFlags(ev, cudaEventDisableTiming));
    for (cudaEvent_t* ev : {&p->start, &p->comp_end, &p->out_end})
        if (rc == RELAY_OK) rc = cuda(cudaEventCreateWithFlags(ev, cudaEventDisableTiming));
    if (rc != RELAY_OK) {
        destroy(p);
        return rc;
    }
    *out = p;
    return RELAY_OK;
}

void relay_host_plan_destroy(relay_host_plan* p) { destroy(p); }

int relay_host_bytes(const relay_host_plan* p, int64_t* h2d, int64_t* d2h) {
    if (!p || !h2d || !d2h) return RELAY_EINVAL;
    int64_t cols = 0;  // copied columns of a row, over all chunks (whole quads)
    for (int64_t c = 0; c < p->nchunks; ++c) cols += ((c == p->nchunks - 1 ? p->last_w : p->cw) + 3) / 4 * 4;
    if (p->h->d == 0) cols = 0;
    auto rows_of = [](const std::vector<RowRun>& runs) {
        int64_t r = 0;
        for (const RowRun& x : runs) r += x.second - x.first;
        return r;
    };
    *h2d = 4 * (cols * (p->n + rows_of(p->in_runs)) + p->E);
    *d2h = 4 * (cols * (p->n + rows_of(p->out_runs)) + p->E);
    return RELAY_OK;
}

int relay_step_host(relay_host_plan* p, float* x, const float* msg_in, float* msg_out, int32_t* counts, float lr,
                    uint64_t seed, int64_t step, relay_stream_t stream) {
    int rc = check_host_args(p, x, msg_in, msg_out, counts, lr);
    if (rc != RELAY_OK) return rc;
    if (step < 0 || step >= (int64_t(1) << 32)) return RELAY_EINVAL;
    refresh(p);
    rc = fork(p, stream);
    // the counters, once per step: c^{t-1} in, c^t computed and copied back;
    // the step kernels below read the device copy
    const bool counted = p->E > 0 || p->h->algo == RELAY_ALGO_DME;
    if (rc == RELAY_OK && p->E > 0)
        rc = cuda(cudaMemcpyAsync(p->counts_d, counts, 4 * p->E, cudaMemcpyHostToDevice, p->s_comp));
    if (rc == RELAY_OK && counted) rc = relay_step_counts(p->hc, p->counts_d, p->s_comp);
    if (rc == RELAY_OK && p->E > 0)
        rc = cuda(cudaMemcpyAsync(counts, p->counts_d, 4 * p->E, cudaMemcpyDeviceToHost, p->s_comp));
    for (int64_t c = 0; c < p->nchunks && rc == RELAY_OK && p->h->d > 0; ++c) {
        const int b = static_cast<int>(c % p->nbuf);
        rc = chunk_in(p, c, b, x, msg_in);
        if (rc == RELAY_OK) rc = cuda(cudaStreamWaitEvent(p->s_comp, p->in_done[b], 0));
        if (rc == RELAY_OK)
            rc = relay_step_models(chunk_handle(p, c), p->xb[b], p->mib[b], p->mob[b], p->counts_d, lr, seed, step,
                                   p->s_comp);
        if (rc == RELAY_OK) rc = chunk_out(p, c, b, x, msg_out, p->mob[b]);
    }
    if (rc == RELAY_OK) rc = join(p, stream);
    return rc;
}

int relay_steps_host(relay_host_plan* p, float* x, const float* msg_in, float* msg_out, int32_t* counts, float lr,
                     uint64_t seed, int64_t t0, int64_t k, relay_stream_t stream) {
    int rc = check_host_args(p, x, msg_in, msg_out, counts, lr);
    if (rc != RELAY_OK) return rc;
    if (p->h->algo == RELAY_ALGO_DME) return RELAY_EUNSUPPORTED;  // its counts would advance once per chunk
    if (t0 < 0 || k < 0 || t0 >= (int64_t(1) << 32) || k > (int64_t(1) << 32) - t0) return RELAY_EINVAL;
    if (k == 0) return RELAY_OK;
    refresh(p);
    rc = fork(p, stream);
    for (int64_t c = 0; c < p->nchunks && rc == RELAY_OK; ++c) {
        const int b = static_cast<int>(c % p->nbuf);
        if (p->h->d > 0) rc = chunk_in(p, c, b, x, msg_in);
        if (rc == RELAY_OK && p->h->d > 0) rc = cuda(cudaStreamWaitEvent(p->s_comp, p->in_done[b], 0));
        // every chunk starts from the same c^{t0-1}
        if (rc == RELAY_OK && p->E > 0)
            rc = cuda(cudaMemcpyAsync(p->counts_d, counts, 4 * p->E, cudaMemcpyHostToDevice, p->s_comp));
        if (rc == RELAY_OK)
            rc = relay_steps(chunk_handle(p, c), p->xb[b], p->mib[b], p->mob[b], p->counts_d, lr, seed, t0, k,
                             p->s_comp);
        // step t0+k-1 wrote the staging array of parity k
        if (rc == RELAY_OK && p->h->d > 0) rc = chunk_out(p, c, b, x, msg_out, (k & 1) ? p->mob[b] : p->mib[b]);
    }
    if (rc == RELAY_OK && p->E > 0)
        rc = cuda(cudaMemcpyAsync(counts, p->counts_d, 4 * p->E, cudaMemcpyDeviceToHost, p->s_comp));
    if (rc == RELAY_OK) rc = join(p, stream);
    return rc;
}

}  // extern "C"
