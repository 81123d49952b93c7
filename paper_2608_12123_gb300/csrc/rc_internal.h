// rc_internal.h -- declarations shared by the kernel and host translation units
// of librc.so.  Not part of the public ABI (see include/rc.h).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace rc {

// Library-owned device words of one context.  One 256-byte block, zeroed at
// rc_init.  The decision flag `sel` is the HBM-resident route decision that
// the next step reads (Section 7.1, device resident path).
struct alignas(256) DevBlock {
    uint32_t sel;           // route body of the next step (last decision)
    uint32_t err;           // first latched error code (0: none)
    uint32_t err_step;      // step of the first latched error
    uint32_t err_member;    // member of the first latched error
    uint32_t step;          // step counter of graph-launched chains
    uint32_t ticket;        // last-CTA ticket of a multi-CTA step
    uint32_t count;         // odd-key count of a multi-CTA step
    uint32_t skip_arrival;  // test hook: CTA 1 skips its first grid-barrier arrival
    uint32_t abort;         // set by a CTA whose bounded wait ran out
    uint32_t step_base;     // added to the step of a latched error (chains run in pieces)
    uint32_t pad0[2];
    uint64_t wait_ns;       // device spin-wait limit (ns of %globaltimer)
    unsigned long long slot[3];  // grid-barrier words of the persistent grid kernel
    uint32_t countdown;     // launch-floor probe: WHILE iterations left
    uint32_t pad1;
    unsigned long long slot4[4];  // monotonic count words of the session-owned chain
};

// Everything a step kernel needs.  Event arrays hold n_sets cohorts of K;
// step n uses cohort n % n_sets.  Output pointers may be null.
struct StepArgs {
    uint8_t *state;
    uint64_t n_sessions;
    const uint32_t *outcome;
    const uint8_t *payload;
    const uint32_t *idx;
    uint32_t n_sets;
    uint32_t K;
    const uint8_t *tables;   // [2][tab_stride] bytes: body A, body B
    uint32_t S;
    uint32_t tab_stride;     // bytes per body, a multiple of 16 (>= 8 S)
    uint32_t *decisions;     // [n_steps]
    uint8_t *effects;        // [n_steps][K][16]
    uint8_t *state_log;      // [n_steps][K][state_bytes]
    uint32_t n_steps;
    DevBlock *dev;
    cudaGraphConditionalHandle h_while;
    long long *trace;        // optional per-step phase clocks of two CTAs (profiling), or null
};

// A segmented step (rc_seg_step): n_seg route-keyed cohorts concatenated;
// segment g holds members [seg_off[g], seg_off[g+1]) and uses route
// seg_route[g], whose bodies are tables + (2 route + sel) * tab_stride and
// whose flag is flags[route].  count (n_seg words) and ticket start at zero
// and are left at zero.
struct SegArgs {
    uint8_t *state;
    uint64_t n_sessions;
    const uint32_t *outcome;
    const uint8_t *payload;
    const uint32_t *idx;  // null: member m is session m
    uint32_t total;
    uint32_t n_seg;
    const uint32_t *seg_route;
    const uint32_t *seg_off;
    const uint8_t *tables;
    uint32_t S;
    uint32_t tab_stride;
    uint32_t *flags;
    uint32_t *count;
    uint32_t *ticket;
    uint32_t *decisions;  // [n_seg] or null
    uint8_t *effects;     // [total][16] or null
    DevBlock *dev;
};

// Epilogue flags of the per-step kernel.
enum : uint32_t {
    EPI_NONE = 0u,
    EPI_SET_WHILE = 1u,  // last CTA sets the WHILE handle to (next step < n_steps)
};

// Error codes latched on the device (same values as include/rc.h).
enum : uint32_t {
    DEV_E_STATE = 4u,
    DEV_E_TIMEOUT = 5u,
    DEV_E_INDEX = 7u,
};

constexpr int kStepThreads = 256;
constexpr int kGridThreads = 256;

// Host-side launch helpers (rc_kernels.cu).
// Per-step kernel: step < 0 reads the step from dev->step (and the last CTA
// advances it); sel < 0 reads the route body from dev->sel.  decide = false
// is the no-decision floor body (no reduction, flag untouched).
const void *step_kernel(int state_bytes, int payload_bytes, bool decide);
dim3 step_grid(uint32_t K);
dim3 step_block(uint32_t K);
cudaError_t launch_step(const StepArgs &a, int state_bytes, int payload_bytes, int step, int sel,
                        uint32_t epi, bool decide, cudaStream_t s);

// Persistent chains.  The single-CTA form takes K <= 512; the grid form is a
// cooperative launch of `grid` CTAs.
cudaError_t launch_chain_cta(const StepArgs &a, int state_bytes, int payload_bytes, cudaStream_t s);
// Pipelined single-CTA chain for identity sessions (records in registers);
// with two_steps and K <= 512, two steps per block barrier.  *launched is
// false when it does not apply.
cudaError_t launch_chain_cta_fast(const StepArgs &a, int state_bytes, int payload_bytes, cudaStream_t s,
                                  bool *launched, bool two_steps);
// Single-CTA chains with explicit indices and the record gather ahead of its
// step (K <= 512): launch_link fills lnk (n_sets * K words) with each
// member's position in the two previous cohorts, then the chain runs (the
// producer-warp form when allow_prod and K is a multiple of 8 and it fits).
// shape_out points to 16 bytes of opaque shape.
bool chain_cta_link_plan(int state_bytes, int payload_bytes, uint32_t K, uint64_t n_sessions, uint32_t tab_stride,
                         bool allow_prod, size_t *smem, void *shape_out);
cudaError_t launch_link(const StepArgs &a, uint32_t *lnk, cudaStream_t s);
cudaError_t launch_chain_cta_link(const StepArgs &a, int state_bytes, int payload_bytes, size_t smem,
                                  const void *shape, const uint32_t *lnk, cudaStream_t s);
// Single-CTA chain keying two steps per block barrier (K <= 256, a multiple
// of 8, payloads of at most 64 bytes): launch_link_pair fills lnk (n_sets * K
// words) with each member's nearest earlier appearance within eight cohorts
// (distance << 16 | position, 0 for none), then the chain runs.  shape_out:
// 16 bytes.
bool chain_cta_pair_plan(int state_bytes, int payload_bytes, uint32_t K, uint32_t S, uint64_t n_sessions,
                         uint32_t tab_stride, size_t *smem, void *shape_out);
cudaError_t launch_link_pair(const StepArgs &a, uint32_t *lnk, cudaStream_t s);
cudaError_t launch_chain_cta_pair(const StepArgs &a, int state_bytes, int payload_bytes, size_t smem,
                                  const void *shape, const uint32_t *lnk, cudaStream_t s);
cudaError_t chain_grid_size(int state_bytes, int payload_bytes, uint32_t K, int *grid);
cudaError_t launch_chain_grid(const StepArgs &a, int state_bytes, int payload_bytes, int grid,
                              cudaStream_t s);

// TMA-fed persistent grid (K a multiple of 8, one CTA per SM).  plan returns
// false when it does not apply; shape_out points to 32 bytes of opaque shape.
bool chain_grid_tma_plan(int state_bytes, int payload_bytes, uint32_t K, uint32_t tab_stride, int *grid,
                         uint32_t *threads, size_t *smem, void *shape_out);
cudaError_t launch_chain_grid_tma(const StepArgs &a, int state_bytes, int payload_bytes, int grid, uint32_t threads,
                                  size_t smem, const void *shape, cudaStream_t s);

// Cluster chain for 512 < K <= 8,192: one cluster of ceil(K / 512) CTAs with
// the hardware cluster barrier per step.
bool chain_cluster_plan(int state_bytes, int payload_bytes, uint32_t K, uint32_t *cluster, uint32_t *threads);
cudaError_t launch_chain_cluster(const StepArgs &a, int state_bytes, int payload_bytes, uint32_t cluster,
                                 uint32_t threads, cudaStream_t s);

// Grid chain split by links (explicit indices, K a multiple of 8): plan
// fills 48 bytes of opaque shape and the scratch size (cohort bitmaps and
// link words); launch clears the bitmaps, marks them, derives the links and
// runs the chain.
bool chain_grid_link_plan(int state_bytes, int payload_bytes, uint32_t K, uint64_t n_sessions, uint32_t n_sets,
                          uint32_t tab_stride, int *grid, uint32_t *threads, size_t *smem, void *shape_out,
                          size_t *scratch);
cudaError_t launch_chain_grid_link(const StepArgs &a, int state_bytes, int payload_bytes, int grid, uint32_t threads,
                                   size_t smem, const void *shape, void *scratch, cudaStream_t s);

// Grid chain keying two steps per grid barrier (explicit indices, K a
// multiple of 8 and at most 65,536): plan fills 48 bytes of opaque shape and
// the scratch size (cohort bitmaps, per-cohort session positions, link
// words, input-state and key rings); launch clears the bitmaps, runs the link
// pass and the chain.
bool chain_grid_pair_plan(int state_bytes, int payload_bytes, uint32_t K, uint64_t n_sessions, uint32_t n_sets,
                          uint32_t tab_stride, int *grid, uint32_t *threads, size_t *smem, void *shape_out,
                          size_t *scratch);
cudaError_t launch_chain_grid_pair(const StepArgs &a, int state_bytes, int payload_bytes, int grid, uint32_t threads,
                                   size_t smem, const void *shape, void *scratch, cudaStream_t s);

// Split-phase persistent chain (explicit session indices, K a multiple of 8,
// at most 512 members per CTA): marks is device scratch of 3 * n_sessions
// words, filled with 0xFF bytes before each launch.
bool chain_split_plan(int state_bytes, int payload_bytes, uint32_t K, uint32_t tab_stride, int *grid,
                      uint32_t *threads, size_t *smem, void *shape_out);
cudaError_t launch_chain_split(const StepArgs &a, int state_bytes, int payload_bytes, int grid, uint32_t threads,
                               size_t smem, const void *shape, uint32_t *marks, cudaStream_t s);

// Session-owned persistent chain: k_route groups each cohort's members by the
// CTA owning their session (perm_* : n_sets * K words each, off : n_sets *
// (G + 1) words), then k_chain_owned runs the chain.
bool chain_owned_plan(int state_bytes, int payload_bytes, uint32_t K, uint64_t n_sessions, uint32_t tab_stride,
                      int *grid, uint32_t *threads, size_t *smem, void *shape_out);
cudaError_t launch_route(const StepArgs &a, const void *shape, uint32_t *perm_m, uint32_t *perm_s, uint32_t *perm_o,
                         uint32_t *off, cudaStream_t s);
// launch_permute_payload writes each cohort's payload rows in routed order
// (n_sets * K * payload_bytes bytes at pay_routed), which the chain then
// loads as tensor tiles.
cudaError_t launch_permute_payload(const StepArgs &a, int payload_bytes, const void *shape, const uint32_t *perm_m,
                                   const uint32_t *off, uint8_t *pay_routed, cudaStream_t s);
cudaError_t launch_chain_owned(const StepArgs &a, int state_bytes, int payload_bytes, int grid, uint32_t threads,
                               size_t smem, const void *shape, const uint32_t *perm_m, const uint32_t *perm_s,
                               const uint32_t *perm_o, const uint32_t *off, const uint8_t *pay_routed,
                               cudaStream_t s);

// One segmented step (at least one CTA, so that empty segments decide 0).
cudaError_t launch_seg_step(const SegArgs &a, int state_bytes, int payload_bytes, cudaStream_t s);

// Writes decisions[0..n) = 0 and sel = 0 (an empty cohort decides 0).
// Writes one word in stream order (a one-thread kernel).
cudaError_t launch_set_word(uint32_t *p, uint32_t v, cudaStream_t s);
cudaError_t launch_empty_cohorts(const StepArgs &a, cudaStream_t s);

// Fixed-nested control: a one-thread kernel that device-launches `child`.
const void *launcher_kernel();
// Launch-floor probes.
const void *empty_kernel();
const void *countdown_kernel();
// n_steps empty grid-barrier steps over one CTA per SM (cooperative launch);
// dev->slot and dev->abort must be zero.
cudaError_t launch_grid_barrier_floor(DevBlock *dev, uint32_t n_steps, cudaStream_t s);

}  // namespace rc
