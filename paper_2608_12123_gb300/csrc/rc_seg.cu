// rc_seg.cu -- the segmented-step context of librc.so (declared in
// include/rc.h): one launch over several route-keyed cohorts, each route with
// its own pair of route bodies and its own device-resident decision flag.
#include <cuda_runtime.h>
#include <stdint.h>

#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <vector>

#include "rc.h"
#include "rc_internal.h"

struct rc_seg {
    uint32_t R = 0, S = 0, SB = 0, P = 0, max_members = 0, max_segments = 0, tab_stride = 0;
    uint64_t n_sessions = 0;
    cudaStream_t stream = nullptr;
    uint8_t *d_tables = nullptr;   // [R][2][tab_stride]
    uint32_t *d_words = nullptr;   // flags [R], counts [max_segments], ticket, meta [max_segments][route, off]
    uint32_t *h_meta = nullptr;    // pinned staging of the segment layout
    rc::DevBlock *dev = nullptr;
    cudaEvent_t meta_done = nullptr;  // the last upload of h_meta has been read
    std::vector<uint32_t> last_layout;  // the layout on the device (routes, then offsets)
    uint32_t *h_err = nullptr;     // pinned: latched error words
    std::string err;
};

namespace {

int fail(rc_seg *c, int code, const char *fmt, ...) {
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

#define SEG_CUDA(c, expr)                                                                                   \
    do {                                                                                                    \
        cudaError_t e_ = (expr);                                                                            \
        if (e_ != cudaSuccess) return fail((c), RC_E_CUDA, "%s: %s (%d)", #expr, cudaGetErrorString(e_), \
                                           static_cast<int>(e_));                                          \
    } while (0)

uint32_t *flags_of(rc_seg *c) { return c->d_words; }
uint32_t *counts_of(rc_seg *c) { return c->d_words + c->R; }
uint32_t *ticket_of(rc_seg *c) { return c->d_words + c->R + c->max_segments; }
uint32_t *meta_of(rc_seg *c) { return c->d_words + c->R + c->max_segments + 1; }  // [routes][offsets]

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" {

int rc_seg_init(rc_seg **out, uint32_t n_routes, uint32_t S, const uint8_t *tables, uint32_t state_bytes,
                uint32_t payload_bytes, uint32_t max_members, uint32_t max_segments, uint64_t n_sessions,
                void *cuda_stream) {
    if (!out) return RC_E_INVAL;
    *out = nullptr;
    if (n_routes == 0 || !tables || max_segments == 0 || n_sessions == 0) return RC_E_INVAL;
    if (S < 1 || S > 256 || (S & (S - 1)) != 0) return RC_E_INVAL;
    if (state_bytes != 16 && state_bytes != 64) return RC_E_INVAL;
    if (payload_bytes != 32 && payload_bytes != 64 && payload_bytes != 128) return RC_E_INVAL;
    for (size_t i = 0; i < static_cast<size_t>(n_routes) * 2 * S * 8; ++i)
        if (tables[i] >= S) return RC_E_INVAL;
    rc_seg *c = new rc_seg();
    c->R = n_routes;
    c->S = S;
    c->SB = state_bytes;
    c->P = payload_bytes;
    c->max_members = max_members;
    c->max_segments = max_segments;
    c->n_sessions = n_sessions;
    c->tab_stride = ((S * 8u + 15u) / 16u) * 16u;
    c->stream = static_cast<cudaStream_t>(cuda_stream);
    auto bail = [&](int code) {
        rc_seg_free(c);
        return code;
    };
    std::vector<uint8_t> padded(static_cast<size_t>(n_routes) * 2 * c->tab_stride, 0);
    for (uint32_t r = 0; r < n_routes; ++r)
        for (uint32_t b = 0; b < 2; ++b)
            std::memcpy(&padded[(static_cast<size_t>(r) * 2 + b) * c->tab_stride],
                        tables + (static_cast<size_t>(r) * 2 + b) * S * 8, S * 8);
    const size_t words = static_cast<size_t>(n_routes) + max_segments + 1 + 2ull * max_segments + 1;
    if (cudaMalloc(&c->d_tables, padded.size()) != cudaSuccess) return bail(RC_E_NOMEM);
    if (cudaMalloc(&c->d_words, words * 4) != cudaSuccess) return bail(RC_E_NOMEM);
    if (cudaMalloc(&c->dev, sizeof(rc::DevBlock)) != cudaSuccess) return bail(RC_E_NOMEM);
    if (cudaMallocHost(&c->h_meta, (2ull * max_segments + 1) * 4) != cudaSuccess) return bail(RC_E_NOMEM);
    if (cudaMallocHost(&c->h_err, 4 * sizeof(uint32_t)) != cudaSuccess) return bail(RC_E_NOMEM);
    if (cudaEventCreateWithFlags(&c->meta_done, cudaEventDisableTiming) != cudaSuccess) return bail(RC_E_CUDA);
    if (cudaMemcpyAsync(c->d_tables, padded.data(), padded.size(), cudaMemcpyHostToDevice, c->stream) != cudaSuccess ||
        cudaMemsetAsync(c->d_words, 0, words * 4, c->stream) != cudaSuccess ||
        cudaMemsetAsync(c->dev, 0, sizeof(rc::DevBlock), c->stream) != cudaSuccess ||
        cudaEventRecord(c->meta_done, c->stream) != cudaSuccess || cudaStreamSynchronize(c->stream) != cudaSuccess)
        return bail(RC_E_CUDA);
    *out = c;
    return RC_OK;
}

int rc_seg_step(rc_seg *c, void *state, const rc_events *ev, uint32_t n_segments, const uint32_t *seg_route,
                const uint32_t *seg_off, uint32_t *decisions_out, void *effects_out) {
    if (!c) return RC_E_INVAL;
    if (!state || !ev || !seg_route || !seg_off || n_segments == 0)
        return fail(c, RC_E_INVAL, "state, events and a non-empty segment layout are required");
    if (n_segments > c->max_segments) return fail(c, RC_E_INVAL, "%u segments > max_segments %u", n_segments,
                                                  c->max_segments);
    if (ev->payload_bytes != c->P) return fail(c, RC_E_INVAL, "payload_bytes %u != %u", ev->payload_bytes, c->P);
    if (seg_off[0] != 0) return fail(c, RC_E_INVAL, "seg_off[0] must be 0");
    std::vector<uint8_t> seen(c->R, 0);
    for (uint32_t g = 0; g < n_segments; ++g) {
        if (seg_off[g + 1] < seg_off[g]) return fail(c, RC_E_INVAL, "seg_off decreases at segment %u", g);
        if (seg_route[g] >= c->R) return fail(c, RC_E_INVAL, "segment %u: route %u >= %u", g, seg_route[g], c->R);
        if (seen[seg_route[g]]++) return fail(c, RC_E_INVAL, "route %u appears twice in one step", seg_route[g]);
    }
    const uint32_t total = seg_off[n_segments];
    if (total > c->max_members) return fail(c, RC_E_INVAL, "%u members > max_members %u", total, c->max_members);
    if (total > 0 && (!ev->outcome || !ev->payload)) return fail(c, RC_E_INVAL, "outcome and payload are required");
    if (!aligned16(ev->payload) || !aligned16(effects_out) || !aligned16(state))
        return fail(c, RC_E_INVAL, "buffers must start on 16-byte boundaries");
    // upload the layout unless the device already holds this one; the previous
    // upload of the pinned staging must have been read before it is rewritten
    std::vector<uint32_t> layout(seg_route, seg_route + n_segments);
    layout.insert(layout.end(), seg_off, seg_off + n_segments + 1);
    if (layout != c->last_layout) {
        SEG_CUDA(c, cudaEventSynchronize(c->meta_done));
        std::memcpy(c->h_meta, seg_route, n_segments * 4);
        std::memcpy(c->h_meta + c->max_segments, seg_off, (n_segments + 1) * 4);
        SEG_CUDA(c, cudaMemcpyAsync(meta_of(c), c->h_meta, (2ull * c->max_segments + 1) * 4,
                                    cudaMemcpyHostToDevice, c->stream));
        SEG_CUDA(c, cudaEventRecord(c->meta_done, c->stream));
        c->last_layout.swap(layout);
    }
    rc::SegArgs a{};
    a.state = static_cast<uint8_t *>(state);
    a.n_sessions = c->n_sessions;
    a.outcome = ev->outcome;
    a.payload = ev->payload;
    a.idx = ev->session_idx;
    a.total = total;
    a.n_seg = n_segments;
    a.seg_route = meta_of(c);
    a.seg_off = meta_of(c) + c->max_segments;
    a.tables = c->d_tables;
    a.S = c->S;
    a.tab_stride = c->tab_stride;
    a.flags = flags_of(c);
    a.count = counts_of(c);
    a.ticket = ticket_of(c);
    a.decisions = decisions_out;
    a.effects = static_cast<uint8_t *>(effects_out);
    a.dev = c->dev;
    SEG_CUDA(c, rc::launch_seg_step(a, static_cast<int>(c->SB), static_cast<int>(c->P), c->stream));
    return RC_OK;
}

int rc_seg_sync(rc_seg *c) {
    if (!c) return RC_E_INVAL;
    SEG_CUDA(c, cudaMemcpyAsync(c->h_err, &c->dev->err, 3 * sizeof(uint32_t), cudaMemcpyDeviceToHost, c->stream));
    SEG_CUDA(c, cudaStreamSynchronize(c->stream));
    const uint32_t code = c->h_err[0];
    if (code == 0) return RC_OK;
    const uint32_t seg = c->h_err[1], member = c->h_err[2];
    SEG_CUDA(c, cudaMemsetAsync(&c->dev->err, 0, 3 * sizeof(uint32_t), c->stream));
    SEG_CUDA(c, cudaStreamSynchronize(c->stream));
    return fail(c, -static_cast<int>(code), "%s (segment %u, member %u)",
                code == rc::DEV_E_STATE ? "state >= S or outcome >= 8" : "session index >= n_sessions", seg,
                member);
}

int rc_seg_get_flags(rc_seg *c, uint32_t *flags_out) {
    if (!c || !flags_out) return RC_E_INVAL;
    SEG_CUDA(c, cudaMemcpyAsync(flags_out, flags_of(c), c->R * 4, cudaMemcpyDeviceToHost, c->stream));
    SEG_CUDA(c, cudaStreamSynchronize(c->stream));
    return RC_OK;
}

int rc_seg_set_flags(rc_seg *c, const uint32_t *flags) {
    if (!c || !flags) return RC_E_INVAL;
    for (uint32_t r = 0; r < c->R; ++r)
        if (flags[r] > 1u) return fail(c, RC_E_INVAL, "flag of route %u is not 0 or 1", r);
    SEG_CUDA(c, cudaMemcpyAsync(flags_of(c), flags, c->R * 4, cudaMemcpyHostToDevice, c->stream));
    SEG_CUDA(c, cudaStreamSynchronize(c->stream));
    return RC_OK;
}

const char *rc_seg_last_error(rc_seg *c) { return c ? c->err.c_str() : "null context"; }

int rc_seg_free(rc_seg *c) {
    if (!c) return RC_OK;
    if (c->stream || c->d_words) cudaStreamSynchronize(c->stream);
    if (c->meta_done) cudaEventDestroy(c->meta_done);
    if (c->h_meta) cudaFreeHost(c->h_meta);
    if (c->h_err) cudaFreeHost(c->h_err);
    if (c->dev) cudaFree(c->dev);
    if (c->d_words) cudaFree(c->d_words);
    if (c->d_tables) cudaFree(c->d_tables);
    delete c;
    return RC_OK;
}

}  // extern "C"
