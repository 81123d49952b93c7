// rc_api.cu -- the C ABI of librc.so (declared and documented in include/rc.h):
// context set-up, argument checks, host-buffer staging, and the five ways a
// step's decision reaches the next step (Sections 7.1 and 8.1 of the paper):
// host round trip, CUDA-graph WHILE node, persistent kernel, fixed nested
// device graph, and the no-decision floor.
#include <cuda_runtime.h>
#include <stdint.h>

#include <chrono>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>
#include <algorithm>
#include <vector>

#include "rc.h"
#include "rc_internal.h"

namespace {

struct Buf {
    void *p = nullptr;
    size_t cap = 0;
};

// What a cached graph was built for; a graph is reused only for equal keys.
struct GraphKey {
    const void *state, *outcome, *payload, *idx, *decisions, *effects, *state_log;
    uint32_t n_sets, K, n_steps, extra;
    uint64_t seq_hash;
    bool operator==(const GraphKey &o) const { return std::memcmp(this, &o, sizeof(*this)) == 0; }
};

struct CachedGraph {
    bool valid = false;
    GraphKey key{};
    cudaGraph_t g = nullptr;
    cudaGraphExec_t e = nullptr;
    void reset() {
        if (e) cudaGraphExecDestroy(e);
        if (g) cudaGraphDestroy(g);
        e = nullptr;
        g = nullptr;
        valid = false;
    }
};

struct NestedGraphs {
    bool valid = false;
    GraphKey key{};
    cudaGraph_t child[2] = {nullptr, nullptr}, outer[2] = {nullptr, nullptr};
    cudaGraphExec_t child_e[2] = {nullptr, nullptr}, outer_e[2] = {nullptr, nullptr};
    void reset() {
        for (int b = 0; b < 2; ++b) {
            if (outer_e[b]) cudaGraphExecDestroy(outer_e[b]);
            if (outer[b]) cudaGraphDestroy(outer[b]);
            if (child_e[b]) cudaGraphExecDestroy(child_e[b]);
            if (child[b]) cudaGraphDestroy(child[b]);
            outer_e[b] = nullptr;
            outer[b] = nullptr;
            child_e[b] = nullptr;
            child[b] = nullptr;
        }
        valid = false;
    }
};

}  // namespace

struct rc_ctx {
    int device = 0;
    int num_sms = 0;
    int coop = 0;
    cudaStream_t stream = nullptr;
    uint32_t S = 0, SB = 0, P = 0, max_K = 0, tab_stride = 0;
    uint64_t n_sessions = 0;
    uint8_t *d_tables = nullptr;
    rc::DevBlock *dev = nullptr;
    uint32_t *h_pinned = nullptr;  // [0] decision flag copy, [1..3] error words
    uint64_t host_wait_ns = 60ull * 1000000000ull;
    uint64_t dev_wait_ns = 2ull * 1000000000ull;
    std::string err;
    Buf st_outcome, st_payload, st_idx, st_dec, st_eff, st_log;
    CachedGraph cond, floor;
    NestedGraphs nested;
    cudaEvent_t ev_start = nullptr, ev_stop = nullptr;
    cudaStream_t copy_stream = nullptr;  // host -> device copies of a chain run in pieces
    cudaStream_t out_stream = nullptr;   // device -> host copies of a chain run in pieces
    std::vector<cudaEvent_t> pipe_ev;    // per piece: inputs copied, piece done
    double last_ms = 0.0;
    uint32_t last_launches = 0;
    bool no_tma = false;   // RC_NO_TMA=1 in the environment selects the plain grid kernel
    bool no_pipe = false;   // RC_NO_PIPE=1 selects the plain single-CTA kernel
    bool no_link = false;   // RC_NO_LINK=1 turns off the linked single-CTA kernels
    bool no_prod = false;   // RC_NO_PROD=1 keeps the linked kernel without a producer warp
    bool no_pair = false;   // RC_NO_PAIR=1 turns off the single-CTA chain keying two steps per barrier
    bool no_pieces = false; // RC_NO_PIECES=1 stages host-memory events whole (no pieces)
    bool no_grid_link = false;  // RC_NO_GRID_LINK=1 turns off the grid chain split by links
    bool grid_pair = false;     // RC_GRID_PAIR=1 takes the grid chain keying two steps per barrier (measured slower)
    bool no_cluster = false;    // RC_NO_CLUSTER=1 turns off the cluster chain (512 < K <= 8192)
    bool use_split = false;  // RC_SPLIT=1 selects the split-phase chain (slower on GB300 so far)
    bool use_owned = false;  // RC_OWNED=1 selects the session-owned chain
    Buf route_buf;           // session-owned chain: routed member lists
    Buf link_buf;            // linked single-CTA chain: n_sets * K link words
    Buf marks;              // split-phase cohort marks (3 * n_sessions words)
    long long *trace = nullptr;
    uint64_t trace_entries = 0;
};

namespace {

int fail(rc_ctx *c, int code, const char *fmt, ...) {
    if (c) {
        char buf[512];
        va_list ap;
        va_start(ap, fmt);
        std::vsnprintf(buf, sizeof(buf), fmt, ap);
        va_end(ap);
        c->err = buf;
    }
    return code;
}

int cuda_fail(rc_ctx *c, cudaError_t e, const char *what) {
    return fail(c, RC_E_CUDA, "%s: %s (%d)", what, cudaGetErrorString(e), static_cast<int>(e));
}

#define RC_CUDA(c, expr)                                      \
    do {                                                      \
        cudaError_t e_ = (expr);                              \
        if (e_ != cudaSuccess) return cuda_fail((c), e_, #expr); \
    } while (0)

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// true when the pointer is ordinary host memory (pageable or pinned), false
// for memory the device addresses directly (device or managed).
bool is_host_ptr(const void *p) {
    cudaPointerAttributes at;
    cudaError_t e = cudaPointerGetAttributes(&at, p);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return true;
    }
    return !(at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged);
}

int ensure(rc_ctx *c, Buf &b, size_t bytes) {
    if (b.cap >= bytes) return RC_OK;
    if (b.p) cudaFree(b.p);
    b.p = nullptr;
    b.cap = 0;
    size_t want = bytes < 256 ? 256 : bytes;
    cudaError_t e = cudaMalloc(&b.p, want);
    if (e != cudaSuccess) {
        cudaGetLastError();
        return fail(c, RC_E_NOMEM, "staging allocation of %zu bytes failed", want);
    }
    b.cap = want;
    return RC_OK;
}

int wait_stream(rc_ctx *c) {
    const auto t0 = std::chrono::steady_clock::now();
    for (uint32_t i = 0;; ++i) {
        cudaError_t e = cudaStreamQuery(c->stream);
        if (e == cudaSuccess) return RC_OK;
        if (e != cudaErrorNotReady) return cuda_fail(c, e, "cudaStreamQuery");
        if ((i & 1023u) == 1023u) {
            const auto dt = std::chrono::steady_clock::now() - t0;
            if (static_cast<uint64_t>(std::chrono::duration_cast<std::chrono::nanoseconds>(dt).count()) >
                c->host_wait_ns)
                return fail(c, RC_E_TIMEOUT, "host wait on the context stream exceeded %llu ns",
                            static_cast<unsigned long long>(c->host_wait_ns));
        }
    }
}

// Copies the latched device error words to the host, waits, and turns a
// latched error into a return code (clearing it on the device).
int finish(rc_ctx *c) {
    RC_CUDA(c, cudaMemcpyAsync(c->h_pinned + 1, &c->dev->err, 3 * sizeof(uint32_t), cudaMemcpyDeviceToHost,
                               c->stream));
    int rc = wait_stream(c);
    if (rc != RC_OK) return rc;
    const uint32_t code = c->h_pinned[1];
    if (code == 0) return RC_OK;
    const uint32_t step = c->h_pinned[2], member = c->h_pinned[3];
    RC_CUDA(c, cudaMemsetAsync(&c->dev->err, 0, 3 * sizeof(uint32_t), c->stream));
    RC_CUDA(c, cudaMemsetAsync(&c->dev->abort, 0, sizeof(uint32_t), c->stream));
    rc = wait_stream(c);
    if (rc != RC_OK) return rc;
    const char *what = code == rc::DEV_E_STATE   ? "state >= S or outcome >= 8"
                       : code == rc::DEV_E_INDEX ? "session index >= n_sessions"
                       : code == rc::DEV_E_TIMEOUT ? "device wait limit reached"
                                                   : "device error";
    return fail(c, -static_cast<int>(code), "%s (step %u, member %u)", what, step, member);
}

struct Resolved {
    rc::StepArgs a{};
    bool host_dec = false, host_eff = false, host_log = false;
    bool host_out = false, host_pay = false, host_idx = false;  // inputs not yet copied (defer_inputs)
    uint32_t *user_dec = nullptr;
    void *user_eff = nullptr, *user_log = nullptr;
    const rc_events *user_ev = nullptr;
};

int check_events(rc_ctx *c, const rc_events *ev, uint32_t K) {
    if (!ev) return fail(c, RC_E_INVAL, "events is NULL");
    if (K > c->max_K) return fail(c, RC_E_INVAL, "K = %u exceeds max_K = %u", K, c->max_K);
    if (ev->payload_bytes != c->P)
        return fail(c, RC_E_INVAL, "payload_bytes %u differs from the context's %u", ev->payload_bytes, c->P);
    if (K > 0 && (!ev->outcome || !ev->payload)) return fail(c, RC_E_INVAL, "outcome or payload is NULL");
    if (!aligned16(ev->outcome) || !aligned16(ev->payload) || !aligned16(ev->session_idx))
        return fail(c, RC_E_INVAL, "event buffers must start on 16-byte boundaries");
    return RC_OK;
}

// Fills the kernel arguments; event and output buffers in host memory are
// staged through device buffers (inputs copied now, or by the caller when
// defer_inputs; outputs after the work).
int resolve(rc_ctx *c, void *state, const rc_events *ev, uint32_t K, uint32_t n_steps, uint32_t *dec,
            void *eff, void *slog, bool dec_is_input, Resolved *r, bool defer_inputs = false) {
    int rc = check_events(c, ev, K);
    if (rc != RC_OK) return rc;
    if (!state || !aligned16(state)) return fail(c, RC_E_INVAL, "state must be a 16-byte aligned device pointer");
    if (is_host_ptr(state)) return fail(c, RC_E_INVAL, "state must be device memory");
    if (!aligned16(dec) || !aligned16(eff) || !aligned16(slog))
        return fail(c, RC_E_INVAL, "output buffers must start on 16-byte boundaries");
    const uint32_t n_sets = ev->n_sets ? ev->n_sets : 1u;
    rc::StepArgs &a = r->a;
    a.state = static_cast<uint8_t *>(state);
    a.n_sessions = c->n_sessions;
    a.n_sets = n_sets;
    a.K = K;
    a.tables = c->d_tables;
    a.S = c->S;
    a.tab_stride = c->tab_stride;
    a.n_steps = n_steps;
    a.dev = c->dev;
    a.h_while = 0;
    a.trace = (c->trace && c->trace_entries >= 16ull * n_steps) ? c->trace : nullptr;
    const size_t n_ev = static_cast<size_t>(n_sets) * K;
    a.outcome = ev->outcome;
    a.payload = ev->payload;
    a.idx = ev->session_idx;
    r->user_ev = ev;
    if (K > 0) {
        if (is_host_ptr(ev->outcome)) {
            if ((rc = ensure(c, c->st_outcome, n_ev * 4)) != RC_OK) return rc;
            if (!defer_inputs)
                RC_CUDA(c, cudaMemcpyAsync(c->st_outcome.p, ev->outcome, n_ev * 4, cudaMemcpyHostToDevice,
                                           c->stream));
            a.outcome = static_cast<const uint32_t *>(c->st_outcome.p);
            r->host_out = defer_inputs;
        }
        if (is_host_ptr(ev->payload)) {
            if ((rc = ensure(c, c->st_payload, n_ev * c->P)) != RC_OK) return rc;
            if (!defer_inputs)
                RC_CUDA(c, cudaMemcpyAsync(c->st_payload.p, ev->payload, n_ev * c->P, cudaMemcpyHostToDevice,
                                           c->stream));
            a.payload = static_cast<const uint8_t *>(c->st_payload.p);
            r->host_pay = defer_inputs;
        }
        if (ev->session_idx && is_host_ptr(ev->session_idx)) {
            if ((rc = ensure(c, c->st_idx, n_ev * 4)) != RC_OK) return rc;
            if (!defer_inputs)
                RC_CUDA(c, cudaMemcpyAsync(c->st_idx.p, ev->session_idx, n_ev * 4, cudaMemcpyHostToDevice,
                                           c->stream));
            a.idx = static_cast<const uint32_t *>(c->st_idx.p);
            r->host_idx = defer_inputs;
        }
    }
    r->user_dec = dec;
    r->user_eff = eff;
    r->user_log = slog;
    a.decisions = dec;
    a.effects = static_cast<uint8_t *>(eff);
    a.state_log = static_cast<uint8_t *>(slog);
    if (dec && !dec_is_input && is_host_ptr(dec)) {
        if ((rc = ensure(c, c->st_dec, static_cast<size_t>(n_steps) * 4)) != RC_OK) return rc;
        a.decisions = static_cast<uint32_t *>(c->st_dec.p);
        r->host_dec = true;
    }
    if (eff && is_host_ptr(eff)) {
        if ((rc = ensure(c, c->st_eff, static_cast<size_t>(n_steps) * K * 16)) != RC_OK) return rc;
        a.effects = static_cast<uint8_t *>(c->st_eff.p);
        r->host_eff = true;
    }
    if (slog && is_host_ptr(slog)) {
        if ((rc = ensure(c, c->st_log, static_cast<size_t>(n_steps) * K * c->SB)) != RC_OK) return rc;
        a.state_log = static_cast<uint8_t *>(c->st_log.p);
        r->host_log = true;
    }
    return RC_OK;
}

int copy_back(rc_ctx *c, const Resolved &r, uint32_t n_steps) {
    const uint32_t K = r.a.K;
    if (r.host_dec)
        RC_CUDA(c, cudaMemcpyAsync(r.user_dec, r.a.decisions, static_cast<size_t>(n_steps) * 4,
                                   cudaMemcpyDeviceToHost, c->stream));
    if (r.host_eff)
        RC_CUDA(c, cudaMemcpyAsync(r.user_eff, r.a.effects, static_cast<size_t>(n_steps) * K * 16,
                                   cudaMemcpyDeviceToHost, c->stream));
    if (r.host_log)
        RC_CUDA(c, cudaMemcpyAsync(r.user_log, r.a.state_log, static_cast<size_t>(n_steps) * K * c->SB,
                                   cudaMemcpyDeviceToHost, c->stream));
    return RC_OK;
}

GraphKey key_of(const rc::StepArgs &a, uint32_t extra, uint64_t seq_hash) {
    GraphKey k;
    std::memset(&k, 0, sizeof(k));
    k.state = a.state;
    k.outcome = a.outcome;
    k.payload = a.payload;
    k.idx = a.idx;
    k.decisions = a.decisions;
    k.effects = a.effects;
    k.state_log = a.state_log;
    k.n_sets = a.n_sets;
    k.K = a.K;
    k.n_steps = a.n_steps;
    k.extra = extra;
    k.seq_hash = seq_hash;
    return k;
}

int add_step_node(rc_ctx *c, cudaGraph_t g, const cudaGraphNode_t *dep, size_t ndep, const rc::StepArgs &a,
                  int step, int sel, uint32_t epi, bool decide, cudaGraphNode_t *out) {
    rc::StepArgs aa = a;
    void *args[] = {&aa, &step, &sel, &epi};
    cudaKernelNodeParams kp;
    std::memset(&kp, 0, sizeof(kp));
    kp.func = const_cast<void *>(rc::step_kernel(c->SB, c->P, decide));
    kp.gridDim = rc::step_grid(a.K);
    kp.blockDim = rc::step_block(a.K);
    kp.sharedMemBytes = 0;
    kp.kernelParams = args;
    RC_CUDA(c, cudaGraphAddKernelNode(out, g, dep, ndep, &kp));
    return RC_OK;
}

// ---- host round trip --------------------------------------------------------
int run_host_rt(rc_ctx *c, const rc::StepArgs &a) {
    uint32_t sel = 0;
    for (uint32_t n = 0; n < a.n_steps; ++n) {
        // step 0 takes the flag left in device memory; later steps take the
        // value the host just read back
        RC_CUDA(c, rc::launch_step(a, c->SB, c->P, static_cast<int>(n), n == 0 ? -1 : static_cast<int>(sel),
                                   rc::EPI_NONE, true, c->stream));
        RC_CUDA(c, cudaMemcpyAsync(c->h_pinned, &c->dev->sel, sizeof(uint32_t), cudaMemcpyDeviceToHost, c->stream));
        int rc = wait_stream(c);
        if (rc != RC_OK) return rc;
        sel = c->h_pinned[0] & 1u;
    }
    return RC_OK;
}

// ---- device resident: CUDA-graph WHILE node --------------------------------
int build_cond(rc_ctx *c, const rc::StepArgs &a0) {
    c->cond.reset();
    cudaGraph_t g = nullptr;
    RC_CUDA(c, cudaGraphCreate(&g, 0));
    c->cond.g = g;
    cudaGraphConditionalHandle h;
    RC_CUDA(c, cudaGraphConditionalHandleCreate(&h, g, 1u, cudaGraphCondAssignDefault));
    cudaGraphNodeParams cp = {};
    cp.type = cudaGraphNodeTypeConditional;
    cp.conditional.handle = h;
    cp.conditional.type = cudaGraphCondTypeWhile;
    cp.conditional.size = 1;
    cudaGraphNode_t wn;
    RC_CUDA(c, cudaGraphAddNode(&wn, g, nullptr, nullptr, 0, &cp));
    cudaGraph_t body = cp.conditional.phGraph_out[0];
    rc::StepArgs a = a0;
    a.h_while = h;
    cudaGraphNode_t kn;
    int rc = add_step_node(c, body, nullptr, 0, a, -1, -1, rc::EPI_SET_WHILE, true, &kn);
    if (rc != RC_OK) return rc;
    RC_CUDA(c, cudaGraphInstantiate(&c->cond.e, g, 0));
    RC_CUDA(c, cudaGraphUpload(c->cond.e, c->stream));
    c->cond.key = key_of(a0, 1, 0);
    c->cond.valid = true;
    return RC_OK;
}

int run_cond(rc_ctx *c, const rc::StepArgs &a) {
    if (!(c->cond.valid && c->cond.key == key_of(a, 1, 0))) {
        int rc = build_cond(c, a);
        if (rc != RC_OK) return rc;
    }
    RC_CUDA(c, cudaMemsetAsync(&c->dev->step, 0, sizeof(uint32_t), c->stream));
    RC_CUDA(c, cudaGraphLaunch(c->cond.e, c->stream));
    return RC_OK;
}

// ---- device resident: persistent kernel ------------------------------------
constexpr uint32_t kPairMinSteps = 64;

int run_persist(rc_ctx *c, const rc::StepArgs &a) {
    if (a.idx && c->use_owned && c->coop && static_cast<uint64_t>(a.n_sets) * a.K < (1ull << 31) - 1024u) {
        int grid = 0;
        uint32_t threads = 0;
        size_t smem = 0;
        alignas(8) unsigned char shape[32];
        if (rc::chain_owned_plan(c->SB, c->P, a.K, c->n_sessions, c->tab_stride, &grid, &threads, &smem, shape)) {
            const size_t nev = static_cast<size_t>(a.n_sets) * a.K;
            const size_t words = (nev * 12 + static_cast<size_t>(a.n_sets) * (grid + 1) * 4 + 255u) & ~size_t(255);
            int rc = ensure(c, c->route_buf, words + nev * c->P);
            if (rc != RC_OK) return rc;
            uint32_t *pm = static_cast<uint32_t *>(c->route_buf.p);
            uint32_t *ps = pm + nev, *po = ps + nev, *off = po + nev;
            uint8_t *pay_routed = static_cast<uint8_t *>(c->route_buf.p) + words;
            RC_CUDA(c, cudaMemsetAsync(c->dev->slot4, 0, sizeof(c->dev->slot4), c->stream));
            RC_CUDA(c, cudaMemsetAsync(&c->dev->abort, 0, sizeof(uint32_t), c->stream));
            c->last_launches = 3;  // routing pass, payload in routed order, chain
            RC_CUDA(c, rc::launch_route(a, shape, pm, ps, po, off, c->stream));
            RC_CUDA(c, rc::launch_permute_payload(a, c->P, shape, pm, off, pay_routed, c->stream));
            RC_CUDA(c, rc::launch_chain_owned(a, c->SB, c->P, grid, threads, smem, shape, pm, ps, po, off,
                                              pay_routed, c->stream));
            RC_CUDA(c, cudaMemsetAsync(&c->dev->skip_arrival, 0, sizeof(uint32_t), c->stream));
            return RC_OK;
        }
    }
    if (a.idx && c->use_split) {
        int grid = 0;
        uint32_t threads = 0;
        size_t smem = 0;
        alignas(8) unsigned char shape[32];
        if (rc::chain_split_plan(c->SB, c->P, a.K, c->tab_stride, &grid, &threads, &smem, shape)) {
            if (grid > 1 && !c->coop) return fail(c, RC_E_UNSUPPORTED, "device lacks cooperative launch");
            int rc = ensure(c, c->marks, 3ull * c->n_sessions * sizeof(uint32_t));
            if (rc != RC_OK) return rc;
            RC_CUDA(c, cudaMemsetAsync(c->marks.p, 0xff, 3ull * c->n_sessions * sizeof(uint32_t), c->stream));
            RC_CUDA(c, cudaMemsetAsync(c->dev->slot, 0, sizeof(c->dev->slot), c->stream));
            RC_CUDA(c, cudaMemsetAsync(&c->dev->abort, 0, sizeof(uint32_t), c->stream));
            RC_CUDA(c, rc::launch_chain_split(a, c->SB, c->P, grid, threads, smem, shape,
                                              static_cast<uint32_t *>(c->marks.p), c->stream));
            RC_CUDA(c, cudaMemsetAsync(&c->dev->skip_arrival, 0, sizeof(uint32_t), c->stream));
            return RC_OK;
        }
    }
    // the two-step chain pays a heavier start (eight-cohort link pass, larger
    // prologue: about 5 to 7 us); it is taken for chains of kPairMinSteps or more
    if (a.idx && !c->no_pair && !c->no_pipe && !c->no_link && !c->no_prod && a.n_steps >= kPairMinSteps) {
        size_t smem = 0;
        alignas(8) unsigned char shape[16];
        if (rc::chain_cta_pair_plan(c->SB, c->P, a.K, c->S, c->n_sessions, c->tab_stride, &smem, shape)) {
            int rc = ensure(c, c->link_buf, static_cast<size_t>(a.n_sets) * a.K * sizeof(uint32_t));
            if (rc != RC_OK) return rc;
            uint32_t *lnk = static_cast<uint32_t *>(c->link_buf.p);
            c->last_launches = 2;  // link pass + chain
            RC_CUDA(c, rc::launch_link_pair(a, lnk, c->stream));
            RC_CUDA(c, rc::launch_chain_cta_pair(a, c->SB, c->P, smem, shape, lnk, c->stream));
            return RC_OK;
        }
    }
    if (a.idx && !c->no_pipe && !c->no_link) {
        size_t smem = 0;
        alignas(8) unsigned char shape[16];
        if (rc::chain_cta_link_plan(c->SB, c->P, a.K, c->n_sessions, c->tab_stride, !c->no_prod, &smem, shape)) {
            int rc = ensure(c, c->link_buf, static_cast<size_t>(a.n_sets) * a.K * sizeof(uint32_t));
            if (rc != RC_OK) return rc;
            uint32_t *lnk = static_cast<uint32_t *>(c->link_buf.p);
            c->last_launches = 2;  // link pass + chain
            RC_CUDA(c, rc::launch_link(a, lnk, c->stream));
            RC_CUDA(c, rc::launch_chain_cta_link(a, c->SB, c->P, smem, shape, lnk, c->stream));
            return RC_OK;
        }
    }
    if (a.K <= 1024u) {
        bool launched = false;
        if (!c->no_pipe) RC_CUDA(c, rc::launch_chain_cta_fast(a, c->SB, c->P, c->stream, &launched, !c->no_pair));
        if (launched) return RC_OK;
        if (a.K <= 512u) {
            RC_CUDA(c, rc::launch_chain_cta(a, c->SB, c->P, c->stream));
            return RC_OK;
        }
    }
    if (!c->no_cluster) {
        uint32_t cluster = 0, threads = 0;
        if (rc::chain_cluster_plan(c->SB, c->P, a.K, &cluster, &threads)) {
            RC_CUDA(c, rc::launch_chain_cluster(a, c->SB, c->P, cluster, threads, c->stream));
            return RC_OK;
        }
    }
    if (!c->coop) return fail(c, RC_E_UNSUPPORTED, "device lacks cooperative launch");
    RC_CUDA(c, cudaMemsetAsync(c->dev->slot, 0, sizeof(c->dev->slot), c->stream));
    RC_CUDA(c, cudaMemsetAsync(&c->dev->abort, 0, sizeof(uint32_t), c->stream));
    if (a.idx && c->grid_pair) {
        int grid = 0;
        uint32_t threads = 0;
        size_t smem = 0, scratch = 0;
        alignas(8) unsigned char shape[48];
        if (rc::chain_grid_pair_plan(c->SB, c->P, a.K, c->n_sessions, a.n_sets, c->tab_stride, &grid, &threads, &smem,
                                     shape, &scratch)) {
            int rc = ensure(c, c->link_buf, scratch);
            if (rc != RC_OK) return rc;
            c->last_launches = 3;  // position and link passes, chain
            RC_CUDA(c, rc::launch_chain_grid_pair(a, c->SB, c->P, grid, threads, smem, shape, c->link_buf.p, c->stream));
            RC_CUDA(c, cudaMemsetAsync(&c->dev->skip_arrival, 0, sizeof(uint32_t), c->stream));
            return RC_OK;
        }
    }
    if (a.idx && !c->no_grid_link) {
        int grid = 0;
        uint32_t threads = 0;
        size_t smem = 0, scratch = 0;
        alignas(8) unsigned char shape[48];
        if (rc::chain_grid_link_plan(c->SB, c->P, a.K, c->n_sessions, a.n_sets, c->tab_stride, &grid, &threads, &smem,
                                     shape, &scratch)) {
            int rc = ensure(c, c->link_buf, scratch);
            if (rc != RC_OK) return rc;
            c->last_launches = 3;  // mark + flag passes, chain
            RC_CUDA(c, rc::launch_chain_grid_link(a, c->SB, c->P, grid, threads, smem, shape, c->link_buf.p, c->stream));
            RC_CUDA(c, cudaMemsetAsync(&c->dev->skip_arrival, 0, sizeof(uint32_t), c->stream));
            return RC_OK;
        }
    }
    int grid = 0;
    uint32_t threads = 0;
    size_t smem = 0;
    alignas(8) unsigned char shape[32];
    if (!c->no_tma && rc::chain_grid_tma_plan(c->SB, c->P, a.K, c->tab_stride, &grid, &threads, &smem, shape)) {
        RC_CUDA(c, rc::launch_chain_grid_tma(a, c->SB, c->P, grid, threads, smem, shape, c->stream));
    } else {
        RC_CUDA(c, rc::chain_grid_size(c->SB, c->P, a.K, &grid));
        RC_CUDA(c, rc::launch_chain_grid(a, c->SB, c->P, grid, c->stream));
    }
    // the test hook arms one launch only
    RC_CUDA(c, cudaMemsetAsync(&c->dev->skip_arrival, 0, sizeof(uint32_t), c->stream));
    return RC_OK;
}

// ---- fixed nested device graph (negative control) --------------------------
int build_nested(rc_ctx *c, const rc::StepArgs &a) {
    c->nested.reset();
    for (int b = 0; b < 2; ++b) {
        RC_CUDA(c, cudaGraphCreate(&c->nested.child[b], 0));
        cudaGraphNode_t kn;
        int rc = add_step_node(c, c->nested.child[b], nullptr, 0, a, -1, b, rc::EPI_NONE, true, &kn);
        if (rc != RC_OK) return rc;
        RC_CUDA(c, cudaGraphInstantiate(&c->nested.child_e[b], c->nested.child[b],
                                        cudaGraphInstantiateFlagDeviceLaunch));
        RC_CUDA(c, cudaGraphUpload(c->nested.child_e[b], c->stream));
        RC_CUDA(c, cudaGraphCreate(&c->nested.outer[b], 0));
        cudaGraphExec_t child = c->nested.child_e[b];
        rc::DevBlock *dev = c->dev;
        void *args[] = {&child, &dev};
        cudaKernelNodeParams kp;
        std::memset(&kp, 0, sizeof(kp));
        kp.func = const_cast<void *>(rc::launcher_kernel());
        kp.gridDim = dim3(1);
        kp.blockDim = dim3(1);
        kp.kernelParams = args;
        cudaGraphNode_t ln;
        RC_CUDA(c, cudaGraphAddKernelNode(&ln, c->nested.outer[b], nullptr, 0, &kp));
        RC_CUDA(c, cudaGraphInstantiate(&c->nested.outer_e[b], c->nested.outer[b], 0));
        RC_CUDA(c, cudaGraphUpload(c->nested.outer_e[b], c->stream));
    }
    c->nested.key = key_of(a, 3, 0);
    c->nested.valid = true;
    return RC_OK;
}

// ---- persistent chain with host-memory events, in pieces -----------------
// The steps run as consecutive persistent launches over pieces of the event
// sets (64 steps first, then four times the previous, up to 1,024): one copy
// stream brings in every piece's events in order, another takes out each
// piece's decisions, effects and state log once it is done, both while later
// pieces run.  Each launch starts from the decision and the state the
// previous one left, so the cohort sequence is the one of a single launch;
// a link that would reach into the previous piece counts as absent and that
// record is gathered from HBM, where the previous launch stored it.  Errors
// report the step of the whole chain (dev->step_base).
constexpr uint32_t kPieceFirst = 64, kPieceGrow = 4, kPieceMax = 1024, kPieceSlots = 1024;  // at most slots pieces

bool pieces_apply(const Resolved &r, rc_mechanism mech) {
    const rc::StepArgs &a = r.a;
    return mech == RC_MECH_RESIDENT_PERSIST && a.K > 0 && a.n_steps >= 2u * kPieceFirst &&
           a.n_sets == a.n_steps && (r.host_out || r.host_pay || r.host_idx);
}

int run_persist_pieces(rc_ctx *c, const Resolved &r) {
    const rc::StepArgs &a0 = r.a;
    const uint32_t n = a0.n_steps, K = a0.K;
    const rc_events *ev = r.user_ev;
    uint32_t cap = kPieceMax;  // at most kPieceSlots - 8 pieces
    if ((n + cap - 1u) / cap > kPieceSlots - 8u) cap = (n + kPieceSlots - 9u) / (kPieceSlots - 8u);
    std::vector<std::pair<uint32_t, uint32_t>> pieces;  // (first step, steps)
    for (uint32_t first = 0, size = std::min(kPieceFirst, cap); first < n; first += pieces.back().second) {
        pieces.emplace_back(first, std::min(size, n - first));
        size = std::min(size * kPieceGrow, cap);
    }
    while (c->pipe_ev.size() < 2 * pieces.size() + 2) {
        cudaEvent_t e;
        RC_CUDA(c, cudaEventCreateWithFlags(&e, cudaEventDisableTiming));
        c->pipe_ev.push_back(e);
    }
    const cudaEvent_t start = c->pipe_ev[0], tail = c->pipe_ev[1];
    // no copy of this call may overtake the work already queued on the context stream
    RC_CUDA(c, cudaEventRecord(start, c->stream));
    RC_CUDA(c, cudaStreamWaitEvent(c->copy_stream, start, 0));
    RC_CUDA(c, cudaStreamWaitEvent(c->out_stream, start, 0));
    for (size_t k = 0; k < pieces.size(); ++k) {
        const size_t e0 = static_cast<size_t>(pieces[k].first) * K, ne = static_cast<size_t>(pieces[k].second) * K;
        if (r.host_out)
            RC_CUDA(c, cudaMemcpyAsync(const_cast<uint32_t *>(a0.outcome) + e0, ev->outcome + e0, ne * 4,
                                       cudaMemcpyHostToDevice, c->copy_stream));
        if (r.host_pay)
            RC_CUDA(c, cudaMemcpyAsync(const_cast<uint8_t *>(a0.payload) + e0 * c->P, ev->payload + e0 * c->P,
                                       ne * c->P, cudaMemcpyHostToDevice, c->copy_stream));
        if (r.host_idx)
            RC_CUDA(c, cudaMemcpyAsync(const_cast<uint32_t *>(a0.idx) + e0, ev->session_idx + e0, ne * 4,
                                       cudaMemcpyHostToDevice, c->copy_stream));
        RC_CUDA(c, cudaEventRecord(c->pipe_ev[2 + 2 * k], c->copy_stream));
    }
    uint32_t launches = 0;
    for (size_t k = 0; k < pieces.size(); ++k) {
        const uint32_t j0 = pieces[k].first, cnt = pieces[k].second;
        const size_t e0 = static_cast<size_t>(j0) * K, ne = static_cast<size_t>(cnt) * K;
        const cudaEvent_t in = c->pipe_ev[2 + 2 * k], done = c->pipe_ev[3 + 2 * k];
        RC_CUDA(c, cudaStreamWaitEvent(c->stream, in, 0));
        RC_CUDA(c, rc::launch_set_word(&c->dev->step_base, j0, c->stream));
        rc::StepArgs a = a0;
        a.outcome = a0.outcome + e0;
        a.payload = a0.payload + e0 * c->P;
        if (a0.idx) a.idx = a0.idx + e0;
        a.n_sets = cnt;
        a.n_steps = cnt;
        a.trace = nullptr;
        if (a0.decisions) a.decisions = a0.decisions + j0;
        if (a0.effects) a.effects = a0.effects + e0 * 16;
        if (a0.state_log) a.state_log = a0.state_log + e0 * c->SB;
        int rc = run_persist(c, a);
        if (rc != RC_OK) return rc;
        launches += c->last_launches + 1u;  // the piece's chain, and its step base
        RC_CUDA(c, cudaEventRecord(done, c->stream));
        RC_CUDA(c, cudaStreamWaitEvent(c->out_stream, done, 0));
        if (r.host_dec)
            RC_CUDA(c, cudaMemcpyAsync(r.user_dec + j0, a.decisions, static_cast<size_t>(cnt) * 4,
                                       cudaMemcpyDeviceToHost, c->out_stream));
        if (r.host_eff)
            RC_CUDA(c, cudaMemcpyAsync(static_cast<uint8_t *>(r.user_eff) + e0 * 16, a.effects, ne * 16,
                                       cudaMemcpyDeviceToHost, c->out_stream));
        if (r.host_log)
            RC_CUDA(c, cudaMemcpyAsync(static_cast<uint8_t *>(r.user_log) + e0 * c->SB, a.state_log, ne * c->SB,
                                       cudaMemcpyDeviceToHost, c->out_stream));
    }
    // the context stream ends after the last copies (the input stream is
    // done once the last piece started); the step base returns to 0
    RC_CUDA(c, cudaEventRecord(tail, c->out_stream));
    RC_CUDA(c, cudaStreamWaitEvent(c->stream, tail, 0));
    RC_CUDA(c, rc::launch_set_word(&c->dev->step_base, 0u, c->stream));
    c->last_launches = launches + 1u;
    return RC_OK;
}

int run_nested(rc_ctx *c, const rc::StepArgs &a) {
    if (!(c->nested.valid && c->nested.key == key_of(a, 3, 0))) {
        int rc = build_nested(c, a);
        if (rc != RC_OK) return rc;
    }
    RC_CUDA(c, cudaMemsetAsync(&c->dev->step, 0, sizeof(uint32_t), c->stream));
    RC_CUDA(c, cudaMemcpyAsync(c->h_pinned, &c->dev->sel, sizeof(uint32_t), cudaMemcpyDeviceToHost, c->stream));
    int rc = wait_stream(c);
    if (rc != RC_OK) return rc;
    uint32_t sel = c->h_pinned[0] & 1u;
    for (uint32_t n = 0; n < a.n_steps; ++n) {
        RC_CUDA(c, cudaGraphLaunch(c->nested.outer_e[sel], c->stream));
        RC_CUDA(c, cudaMemcpyAsync(c->h_pinned, &c->dev->sel, sizeof(uint32_t), cudaMemcpyDeviceToHost, c->stream));
        rc = wait_stream(c);
        if (rc != RC_OK) return rc;
        sel = c->h_pinned[0] & 1u;
    }
    return RC_OK;
}

// ---- no-decision floor -------------------------------------------------------
uint64_t fnv1a(const uint32_t *p, uint32_t n) {
    uint64_t h = 1469598103934665603ull;
    for (uint32_t i = 0; i < n; ++i) {
        h ^= p[i];
        h *= 1099511628211ull;
    }
    return h;
}

int run_floor(rc_ctx *c, const rc::StepArgs &a0, const uint32_t *seq_host) {
    rc::StepArgs a = a0;
    a.decisions = nullptr;
    const uint64_t hsh = fnv1a(seq_host, a.n_steps);
    if (!(c->floor.valid && c->floor.key == key_of(a, 4, hsh))) {
        c->floor.reset();
        RC_CUDA(c, cudaGraphCreate(&c->floor.g, 0));
        cudaGraphNode_t prev = nullptr;
        for (uint32_t n = 0; n < a.n_steps; ++n) {
            cudaGraphNode_t kn;
            const int sel = n == 0 ? -1 : static_cast<int>(seq_host[n - 1] & 1u);
            int rc = add_step_node(c, c->floor.g, prev ? &prev : nullptr, prev ? 1 : 0, a, static_cast<int>(n), sel,
                                   rc::EPI_NONE, false, &kn);
            if (rc != RC_OK) return rc;
            prev = kn;
        }
        RC_CUDA(c, cudaGraphInstantiate(&c->floor.e, c->floor.g, 0));
        RC_CUDA(c, cudaGraphUpload(c->floor.e, c->stream));
        c->floor.key = key_of(a, 4, hsh);
        c->floor.valid = true;
    }
    RC_CUDA(c, cudaGraphLaunch(c->floor.e, c->stream));
    return RC_OK;
}

}  // namespace

extern "C" {

int rc_init(rc_ctx **out, uint32_t S, const uint8_t *table, uint32_t state_bytes, uint32_t payload_bytes,
            uint32_t max_K, uint64_t n_sessions, void *cuda_stream) {
    if (!out) return RC_E_INVAL;
    *out = nullptr;
    if (S < 1 || S > 256 || (S & (S - 1)) != 0) return RC_E_INVAL;
    if (!table || (state_bytes != 16 && state_bytes != 64)) return RC_E_INVAL;
    if (payload_bytes != 32 && payload_bytes != 64 && payload_bytes != 128) return RC_E_INVAL;
    if (max_K < 1 || n_sessions < 1 || n_sessions > 0xffffffffull) return RC_E_INVAL;
    for (uint32_t i = 0; i < 2 * S * 8; ++i)
        if (table[i] >= S) return RC_E_INVAL;
    rc_ctx *c = new (std::nothrow) rc_ctx();
    if (!c) return RC_E_NOMEM;
    c->S = S;
    c->SB = state_bytes;
    c->P = payload_bytes;
    c->max_K = max_K;
    c->n_sessions = n_sessions;
    c->tab_stride = ((S * 8u + 15u) / 16u) * 16u;
    c->stream = static_cast<cudaStream_t>(cuda_stream);
    {
        const char *v = std::getenv("RC_NO_TMA");
        c->no_tma = v && v[0] == '1';
        const char *w = std::getenv("RC_NO_PIPE");
        c->no_pipe = w && w[0] == '1';
        const char *z = std::getenv("RC_NO_LINK");
        c->no_link = z && z[0] == '1';
        const char *q = std::getenv("RC_NO_PROD");
        c->no_prod = q && q[0] == '1';
        const char *pr = std::getenv("RC_NO_PAIR");
        c->no_pair = pr && pr[0] == '1';
        const char *np = std::getenv("RC_NO_PIECES");
        c->no_pieces = np && np[0] == '1';
        const char *gl = std::getenv("RC_NO_GRID_LINK");
        c->no_grid_link = gl && gl[0] == '1';
        const char *gp = std::getenv("RC_GRID_PAIR");
        c->grid_pair = gp && gp[0] == '1';
        const char *cl = std::getenv("RC_NO_CLUSTER");
        c->no_cluster = cl && cl[0] == '1';
        const char *x = std::getenv("RC_SPLIT");
        c->use_split = x && x[0] == '1';
        const char *y = std::getenv("RC_OWNED");
        c->use_owned = y && y[0] == '1';
    }
    auto bail = [&](cudaError_t e) {
        rc_free(c);
        (void)e;
        return RC_E_CUDA;
    };
    cudaError_t e;
    if ((e = cudaGetDevice(&c->device)) != cudaSuccess) return bail(e);
    if ((e = cudaDeviceGetAttribute(&c->num_sms, cudaDevAttrMultiProcessorCount, c->device)) != cudaSuccess)
        return bail(e);
    if ((e = cudaDeviceGetAttribute(&c->coop, cudaDevAttrCooperativeLaunch, c->device)) != cudaSuccess)
        return bail(e);
    std::vector<uint8_t> padded(2 * static_cast<size_t>(c->tab_stride), 0);
    for (int b = 0; b < 2; ++b) std::memcpy(padded.data() + b * c->tab_stride, table + b * S * 8, S * 8);
    if ((e = cudaMalloc(&c->d_tables, padded.size())) != cudaSuccess) return bail(e);
    if ((e = cudaMemcpy(c->d_tables, padded.data(), padded.size(), cudaMemcpyHostToDevice)) != cudaSuccess)
        return bail(e);
    if ((e = cudaMalloc(&c->dev, sizeof(rc::DevBlock))) != cudaSuccess) return bail(e);
    rc::DevBlock init;
    std::memset(&init, 0, sizeof(init));
    init.wait_ns = c->dev_wait_ns;
    if ((e = cudaMemcpy(c->dev, &init, sizeof(init), cudaMemcpyHostToDevice)) != cudaSuccess) return bail(e);
    if ((e = cudaHostAlloc(reinterpret_cast<void **>(&c->h_pinned), 64, cudaHostAllocDefault)) != cudaSuccess)
        return bail(e);
    if ((e = cudaEventCreate(&c->ev_start)) != cudaSuccess) return bail(e);
    if ((e = cudaEventCreate(&c->ev_stop)) != cudaSuccess) return bail(e);
    if ((e = cudaStreamCreateWithFlags(&c->copy_stream, cudaStreamNonBlocking)) != cudaSuccess) return bail(e);
    if ((e = cudaStreamCreateWithFlags(&c->out_stream, cudaStreamNonBlocking)) != cudaSuccess) return bail(e);

    std::memset(c->h_pinned, 0, 64);
    *out = c;
    return RC_OK;
}

int rc_cohort_step(rc_ctx *c, void *state, const rc_events *ev, uint32_t K, int64_t deadline_ns, void *effects) {
    if (!c) return RC_E_INVAL;
    c->err.clear();
    if (ev && ev->launch_ns > deadline_ns)
        return fail(c, RC_E_DEADLINE, "launch at %lld ns is after the deadline %lld ns",
                    static_cast<long long>(ev->launch_ns), static_cast<long long>(deadline_ns));
    Resolved r;
    int rc = resolve(c, state, ev, K, 1, nullptr, effects, nullptr, false, &r);
    if (rc != RC_OK) return rc;
    r.a.n_sets = 1;
    if (K == 0) {
        RC_CUDA(c, rc::launch_empty_cohorts(r.a, c->stream));
    } else {
        RC_CUDA(c, rc::launch_step(r.a, c->SB, c->P, 0, -1, rc::EPI_NONE, true, c->stream));
    }
    rc = copy_back(c, r, 1);
    if (rc != RC_OK) return rc;
    if (r.host_eff) return wait_stream(c);
    return RC_OK;
}

int rc_chain(rc_ctx *c, uint32_t n_steps, rc_mechanism mech, void *state, const rc_events *ev, uint32_t K,
             uint32_t *decisions, void *effects, void *state_log) {
    if (!c) return RC_E_INVAL;
    c->err.clear();
    if (mech == RC_MECH_RESIDENT) mech = RC_MECH_RESIDENT_PERSIST;
    if (mech < RC_MECH_HOST_RT || mech > RC_MECH_FLOOR) return fail(c, RC_E_INVAL, "unknown mechanism %d", mech);
    const bool floor = mech == RC_MECH_FLOOR;
    if (floor && (!decisions || !is_host_ptr(decisions)))
        return fail(c, RC_E_INVAL, "the floor replays a route sequence given in host memory (decisions_out)");
    Resolved r;
    const bool may_piece = mech == RC_MECH_RESIDENT_PERSIST && ev && ev->n_sets == n_steps && !c->no_pieces;
    int rc = resolve(c, state, ev, K, n_steps, decisions, effects, state_log, floor, &r, may_piece);
    if (rc != RC_OK) return rc;
    const bool pieces = may_piece && pieces_apply(r, mech);
    if (may_piece && !pieces) {
        // inputs staged whole after all
        const size_t n_ev = static_cast<size_t>(r.a.n_sets) * K;
        if (r.host_out)
            RC_CUDA(c, cudaMemcpyAsync(const_cast<uint32_t *>(r.a.outcome), ev->outcome, n_ev * 4,
                                       cudaMemcpyHostToDevice, c->stream));
        if (r.host_pay)
            RC_CUDA(c, cudaMemcpyAsync(const_cast<uint8_t *>(r.a.payload), ev->payload, n_ev * c->P,
                                       cudaMemcpyHostToDevice, c->stream));
        if (r.host_idx)
            RC_CUDA(c, cudaMemcpyAsync(const_cast<uint32_t *>(r.a.idx), ev->session_idx, n_ev * 4,
                                       cudaMemcpyHostToDevice, c->stream));
    }
    if (floor) r.a.decisions = nullptr;
    c->last_ms = 0.0;
    c->last_launches = 0;
    if (n_steps == 0) return finish(c);
    RC_CUDA(c, cudaEventRecord(c->ev_start, c->stream));
    if (K == 0) {
        if (!floor) RC_CUDA(c, rc::launch_empty_cohorts(r.a, c->stream));
        c->last_launches = floor ? 0u : 1u;
    } else {
        // kernel executions: one per step, two per step for the nested control
        // (launcher + child), one for the persistent kernel (two where it
        // starts with a pass over the event ring)
        c->last_launches = mech == RC_MECH_RESIDENT_PERSIST ? 1u
                           : mech == RC_MECH_FIXED_NESTED  ? 2u * n_steps
                                                           : n_steps;
        switch (mech) {
            case RC_MECH_HOST_RT: rc = run_host_rt(c, r.a); break;
            case RC_MECH_RESIDENT_COND: rc = run_cond(c, r.a); break;
            case RC_MECH_RESIDENT_PERSIST: rc = pieces ? run_persist_pieces(c, r) : run_persist(c, r.a); break;
            case RC_MECH_FIXED_NESTED: rc = run_nested(c, r.a); break;
            case RC_MECH_FLOOR: rc = run_floor(c, r.a, decisions); break;
            default: rc = fail(c, RC_E_INVAL, "unknown mechanism");
        }
        if (rc != RC_OK) return rc;
    }
    RC_CUDA(c, cudaEventRecord(c->ev_stop, c->stream));
    if (!pieces) {
        rc = copy_back(c, r, n_steps);
        if (rc != RC_OK) return rc;
    }
    rc = finish(c);
    float ms = 0.f;
    if (cudaEventElapsedTime(&ms, c->ev_start, c->ev_stop) == cudaSuccess) c->last_ms = ms;
    return rc;
}

int rc_free(rc_ctx *c) {
    if (!c) return RC_OK;
    if (c->stream || c->dev) cudaStreamSynchronize(c->stream);
    c->cond.reset();
    c->floor.reset();
    c->nested.reset();
    for (Buf *b : {&c->st_outcome, &c->st_payload, &c->st_idx, &c->st_dec, &c->st_eff, &c->st_log, &c->marks, &c->route_buf, &c->link_buf})
        if (b->p) cudaFree(b->p);
    if (c->d_tables) cudaFree(c->d_tables);
    if (c->dev) cudaFree(c->dev);
    if (c->h_pinned) cudaFreeHost(c->h_pinned);
    if (c->ev_start) cudaEventDestroy(c->ev_start);
    if (c->ev_stop) cudaEventDestroy(c->ev_stop);
    for (cudaStream_t st : {c->copy_stream, c->out_stream}) {
        if (st) {
            cudaStreamSynchronize(st);
            cudaStreamDestroy(st);
        }
    }
    for (cudaEvent_t e : c->pipe_ev) cudaEventDestroy(e);
    delete c;
    return RC_OK;
}

const char *rc_last_error(rc_ctx *c) { return c ? c->err.c_str() : "no context"; }

int rc_sync(rc_ctx *c) {
    if (!c) return RC_E_INVAL;
    return finish(c);
}

int rc_get_decision(rc_ctx *c, uint32_t *sel_out) {
    if (!c || !sel_out) return RC_E_INVAL;
    RC_CUDA(c, cudaMemcpyAsync(c->h_pinned, &c->dev->sel, sizeof(uint32_t), cudaMemcpyDeviceToHost, c->stream));
    int rc = wait_stream(c);
    if (rc != RC_OK) return rc;
    *sel_out = c->h_pinned[0];
    return RC_OK;
}

int rc_set_decision(rc_ctx *c, uint32_t sel) {
    if (!c || sel > 1) return RC_E_INVAL;
    RC_CUDA(c, cudaMemsetAsync(&c->dev->sel, 0, sizeof(uint32_t), c->stream));
    if (sel) RC_CUDA(c, cudaMemsetAsync(&c->dev->sel, 1, 1, c->stream));
    return RC_OK;
}

int rc_set_wait_limits(rc_ctx *c, uint64_t device_ns, uint64_t host_ns) {
    if (!c || device_ns == 0 || host_ns == 0) return RC_E_INVAL;
    c->dev_wait_ns = device_ns;
    c->host_wait_ns = host_ns;
    RC_CUDA(c, cudaMemcpy(&c->dev->wait_ns, &device_ns, sizeof(uint64_t), cudaMemcpyHostToDevice));
    return RC_OK;
}

int rc_last_chain_stats(rc_ctx *c, double *device_ms_out, uint32_t *kernel_launches_out) {
    if (!c) return RC_E_INVAL;
    if (device_ms_out) *device_ms_out = c->last_ms;
    if (kernel_launches_out) *kernel_launches_out = c->last_launches;
    return RC_OK;
}

int rc_set_trace(rc_ctx *c, void *device_buf, uint64_t bytes) {
    if (!c) return RC_E_INVAL;
    if (device_buf && (!aligned16(device_buf) || is_host_ptr(device_buf)))
        return fail(c, RC_E_INVAL, "the trace buffer must be 16-byte aligned device memory");
    c->trace = static_cast<long long *>(device_buf);
    c->trace_entries = device_buf ? bytes / sizeof(long long) : 0;
    return RC_OK;
}

int rc_debug_skip_arrival(rc_ctx *c, uint32_t armed) {
    if (!c) return RC_E_INVAL;
    const uint32_t v = armed ? 1u : 0u;
    RC_CUDA(c, cudaMemcpy(&c->dev->skip_arrival, &v, sizeof(v), cudaMemcpyHostToDevice));
    return RC_OK;
}

int rc_launch_floor(rc_ctx *c, int kind, uint32_t reps, double *us_out) {
    if (!c || !us_out || reps == 0) return RC_E_INVAL;
    using clk = std::chrono::steady_clock;
    int rc = RC_OK;
    if (kind == 0 || kind == 3) {
        for (uint32_t i = 0; i < 8; ++i) {  // warm-up
            RC_CUDA(c, cudaLaunchKernel(rc::empty_kernel(), dim3(1), dim3(32), nullptr, 0, c->stream));
            if ((rc = wait_stream(c)) != RC_OK) return rc;
        }
        const auto t0 = clk::now();
        for (uint32_t i = 0; i < reps; ++i) {
            RC_CUDA(c, cudaLaunchKernel(rc::empty_kernel(), dim3(1), dim3(32), nullptr, 0, c->stream));
            if (kind == 3)
                RC_CUDA(c, cudaMemcpyAsync(c->h_pinned, &c->dev->sel, sizeof(uint32_t), cudaMemcpyDeviceToHost,
                                           c->stream));
            if ((rc = wait_stream(c)) != RC_OK) return rc;
        }
        const double ns = std::chrono::duration<double, std::nano>(clk::now() - t0).count();
        *us_out = ns / reps / 1000.0;
        return RC_OK;
    }
    if (kind == 4) {
        cudaEvent_t e0 = nullptr, e1 = nullptr;
        cudaError_t e = cudaEventCreate(&e0);
        if (e == cudaSuccess) e = cudaEventCreate(&e1);
        float ms = 0.f;
        for (int it = 0; it < 3 && e == cudaSuccess; ++it) {  // two warm-ups, then the timed launch
            e = cudaMemsetAsync(c->dev->slot, 0, sizeof(c->dev->slot), c->stream);
            if (e == cudaSuccess) e = cudaMemsetAsync(&c->dev->abort, 0, sizeof(uint32_t), c->stream);
            if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
            if (e == cudaSuccess) e = cudaEventRecord(e0, c->stream);
            if (e == cudaSuccess) e = rc::launch_grid_barrier_floor(c->dev, reps, c->stream);
            if (e == cudaSuccess) e = cudaEventRecord(e1, c->stream);
            if (e == cudaSuccess) e = cudaEventSynchronize(e1);
            if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
        }
        if (e0) cudaEventDestroy(e0);
        if (e1) cudaEventDestroy(e1);
        if (e != cudaSuccess) return cuda_fail(c, e, "grid-barrier floor probe");
        if ((rc = finish(c)) != RC_OK) return rc;  // a barrier wait that ran out
        *us_out = static_cast<double>(ms) * 1000.0 / reps;
        return RC_OK;
    }
    if (kind != 1 && kind != 2) return fail(c, RC_E_INVAL, "unknown probe kind %d", kind);
    cudaGraph_t g = nullptr;
    cudaGraphExec_t ge = nullptr;
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    auto cleanup = [&]() {
        if (ge) cudaGraphExecDestroy(ge);
        if (g) cudaGraphDestroy(g);
        if (e0) cudaEventDestroy(e0);
        if (e1) cudaEventDestroy(e1);
    };
    cudaError_t e = cudaGraphCreate(&g, 0);
    if (e == cudaSuccess && kind == 1) {
        cudaGraphNode_t prev = nullptr;
        for (uint32_t i = 0; i < reps && e == cudaSuccess; ++i) {
            cudaKernelNodeParams kp;
            std::memset(&kp, 0, sizeof(kp));
            kp.func = const_cast<void *>(rc::empty_kernel());
            kp.gridDim = dim3(1);
            kp.blockDim = dim3(32);
            kp.kernelParams = nullptr;
            cudaGraphNode_t kn;
            e = cudaGraphAddKernelNode(&kn, g, prev ? &prev : nullptr, prev ? 1 : 0, &kp);
            prev = kn;
        }
    } else if (e == cudaSuccess) {
        cudaGraphConditionalHandle h;
        e = cudaGraphConditionalHandleCreate(&h, g, 1u, cudaGraphCondAssignDefault);
        cudaGraphNodeParams cp = {};
        cp.type = cudaGraphNodeTypeConditional;
        cp.conditional.handle = h;
        cp.conditional.type = cudaGraphCondTypeWhile;
        cp.conditional.size = 1;
        cudaGraphNode_t wn;
        if (e == cudaSuccess) e = cudaGraphAddNode(&wn, g, nullptr, nullptr, 0, &cp);
        if (e == cudaSuccess) {
            rc::DevBlock *dev = c->dev;
            void *args[] = {&dev, &h};
            cudaKernelNodeParams kp;
            std::memset(&kp, 0, sizeof(kp));
            kp.func = const_cast<void *>(rc::countdown_kernel());
            kp.gridDim = dim3(1);
            kp.blockDim = dim3(1);
            kp.kernelParams = args;
            cudaGraphNode_t kn;
            e = cudaGraphAddKernelNode(&kn, cp.conditional.phGraph_out[0], nullptr, 0, &kp);
        }
    }
    if (e == cudaSuccess) e = cudaGraphInstantiate(&ge, g, 0);
    if (e == cudaSuccess) e = cudaGraphUpload(ge, c->stream);
    if (e == cudaSuccess) e = cudaEventCreate(&e0);
    if (e == cudaSuccess) e = cudaEventCreate(&e1);
    float ms = 0.f;
    for (int it = 0; it < 3 && e == cudaSuccess; ++it) {  // two warm-ups, then the timed launch
        if (kind == 2) e = cudaMemcpyAsync(&c->dev->countdown, &reps, sizeof(reps), cudaMemcpyHostToDevice, c->stream);
        if (e == cudaSuccess) e = cudaStreamSynchronize(c->stream);
        if (e == cudaSuccess) e = cudaEventRecord(e0, c->stream);
        if (e == cudaSuccess) e = cudaGraphLaunch(ge, c->stream);
        if (e == cudaSuccess) e = cudaEventRecord(e1, c->stream);
        if (e == cudaSuccess) e = cudaEventSynchronize(e1);
        if (e == cudaSuccess) e = cudaEventElapsedTime(&ms, e0, e1);
    }
    cleanup();
    if (e != cudaSuccess) return cuda_fail(c, e, "launch-floor probe");
    *us_out = static_cast<double>(ms) * 1000.0 / reps;
    return RC_OK;
}

}  // extern "C"
