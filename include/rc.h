/*
 * rc.h -- C ABI of librc.so, the GB300 (sm_103a) ready-cohort transition engine.
 *
 * What it computes (arXiv 2608.12123, "Ready Cohorts"):
 *   A cohort is K control events of one route, each addressed to one session.
 *   One cohort step (Section 2.1: a transition reads typed state and an event
 *   and emits new state, a route and possibly an effect descriptor) does, for
 *   every member m with session s = session_idx[m] (or m), outcome o and
 *   payload p, on that session's state record {state x, step, acc...}:
 *     rk  = route key of (x, o, p)          (64-bit; x is the state before the step)
 *     y   = T_sel[x][o]                     (route body sel of the two, Section 7.1)
 *     record <- {y, step + 1, acc mixed with rk}
 *     effect[m] = {rk, s, y | o << 16 | sel << 24}
 *   and one global binary decision (Section 7.1: a GPU predicate computes one
 *   global binary route decision per epoch):
 *     d = (number of members with odd rk) > floor(K / 2)
 *   which selects the route body of the next step.  The decision stays in the
 *   device memory of the context; the resident mechanisms read it there and
 *   never copy it to the host (Section 7.1, device resident path).
 *
 *   Exact arithmetic (the paper defines neither hash nor update; this library's
 *   reading, identical in the separate CPU oracle):
 *     fin(z)  = SplitMix64 output finaliser (Steele, Lea, Flood, OOPSLA 2014)
 *     rk      = fin((x | o << 32) ^ 0x9E3779B97F4A7C15), then rk = fin(rk ^ w_k)
 *               for each little-endian 64-bit payload word w_k in order
 *     acc     = (acc ^ rk) * 0x9E3779B97F4A7C15                     16-byte record
 *     acc[j]  = (acc[j] ^ rotl64(rk, 8 j)) * 0x9E3779B97F4A7C15, j<7  64-byte record
 *   State records are little-endian: 16 bytes {int32 state, uint32 step,
 *   uint64 acc} or 64 bytes {int32 state, uint32 step, uint64 acc[7]}.
 *   Effects are 16 bytes {uint64 rk, uint32 session, uint32 y|o<<16|sel<<24}.
 *
 * Conventions for every call:
 *   - Return RC_OK (0) or a negative RC_E_* code; rc_last_error() gives text.
 *   - Work is asynchronous on the context's CUDA stream, except where a call
 *     says it synchronises.  Errors that kernels find (a state >= S, an
 *     outcome >= 8, a session index >= n_sessions, a device wait that ran out)
 *     are latched in device memory and returned by the next synchronising call
 *     (rc_chain and rc_sync synchronise).
 *   - "Device pointer" means memory the GPU of the context can address
 *     (cudaMalloc / torch CUDA tensors).  Event and output buffers may also be
 *     host memory (pageable or pinned): the library then copies them through
 *     its own device staging buffers, inside the call.  A persistent chain
 *     with one cohort per step (n_sets == n_steps, at least 128 steps) over
 *     host-memory events runs as consecutive persistent launches over pieces
 *     of the steps (64, then four times the previous, up to 1,024), with
 *     the copies of later pieces' events and of earlier pieces' outputs on
 *     two library streams overlapping the running piece; the results are the
 *     ones of one launch (set RC_NO_PIECES=1 in the environment to stage
 *     whole).  The state array must be device memory.
 *   - All buffers passed in stay owned by the caller; the library owns the
 *     context, its device copy of the tables, the decision flag, counters,
 *     staging buffers, pinned host words and CUDA graphs.
 *   - Buffers must start on 16-byte boundaries.
 *   - A context is not thread-safe: one host thread at a time.
 */
#ifndef RC_H
#define RC_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define RC_OK 0
#define RC_E_INVAL (-1)       /* bad argument; nothing launched */
#define RC_E_CUDA (-2)        /* a CUDA runtime call failed */
#define RC_E_DEADLINE (-3)    /* launch_ns > deadline_ns; nothing launched (Section 2.3, Eq. 1) */
#define RC_E_STATE (-4)       /* a kernel saw state >= S or outcome >= 8 (latched) */
#define RC_E_TIMEOUT (-5)     /* a bounded device or host wait ran out */
#define RC_E_UNSUPPORTED (-6) /* shape or mechanism not available on this device */
#define RC_E_INDEX (-7)       /* a kernel saw session_idx >= n_sessions (latched) */
#define RC_E_NOMEM (-8)       /* a device or host allocation failed */
#define RC_E_SIZE (-9)        /* larger than the fixed scratch of rc_cohort_step_noalloc allows */

typedef struct rc_ctx rc_ctx;

/* How the decision of step n reaches step n + 1 (Section 7.1, Section 8.1). */
typedef enum {
    /* Host round trip: per step, launch the step kernel with the host's sel,
       copy the 4-byte decision to pinned host memory, synchronise, branch on
       the host, launch the next step. */
    RC_MECH_HOST_RT = 0,
    /* Device resident, CUDA-graph conditional node: one graph launch whose
       WHILE node re-runs the step kernel; the step's last CTA sets the loop
       handle and the flag in device memory selects the next route body. */
    RC_MECH_RESIDENT_COND = 1,
    /* Device resident, persistent kernel: one launch runs all steps; the
       decision is reduced and read on device between steps (one warp for
       K <= 32 with identity sessions, one CTA for K <= 1024, one thread-block
       cluster for K <= 8,192, a cooperative grid otherwise; the single-warp
       and single-CTA forms key two consecutive steps per barrier where they
       apply, which gives the same results). */
    RC_MECH_RESIDENT_PERSIST = 2,
    /* Fixed nested graph (Section 8.1 negative control): per step the host
       launches a graph whose launcher kernel device-launches a fixed child
       graph holding the step body it chose; then the 4-byte copy, the
       synchronisation and the host branch as in RC_MECH_HOST_RT. */
    RC_MECH_FIXED_NESTED = 3,
    /* No-decision floor (Section 7.1): replays a given route sequence as one
       graph of step kernels without computing or reading any decision.  Not
       an admissible policy; a structural floor. */
    RC_MECH_FLOOR = 4,
    /* The resident mechanism measured fastest for the shape
       (currently the persistent kernel). */
    RC_MECH_RESIDENT = 5
} rc_mechanism;

/* The events of one or more cohorts of K members.
   Cohort j (0 <= j < n_sets) owns outcome[j*K .. j*K+K-1],
   payload[(j*K) * payload_bytes ...] and session_idx[j*K ...].
   Step n of a chain uses cohort n mod n_sets (n_sets = 0 means 1). */
typedef struct {
    const uint32_t *outcome;     /* outcome class per member, < 8 */
    const uint8_t *payload;      /* payload_bytes per member */
    const uint32_t *session_idx; /* session per member, < n_sessions, no repeats within
                                    a cohort; NULL: member m is session m */
    uint32_t payload_bytes;      /* must equal the context's payload_bytes */
    uint32_t n_sets;
    int64_t launch_ns;           /* launch time tau of the (first) cohort, integer ns */
} rc_events;

/* Creates a context.
 *   S: number of automaton states, a power of two in [1, 256].
 *   transition_table: HOST pointer to uint8 [2][S][8], route body A then B;
 *     entry [b][x][o] is the next state of state x on outcome o; every entry
 *     must be < S.  Copied to device memory.
 *   state_bytes: 16 or 64.  payload_bytes: 32, 64 or 128.
 *   max_K: largest cohort size the context will be given (>= 1).
 *   n_sessions: number of records in every state array given to this context
 *     (session indices are checked against it on the device).
 *   cuda_stream: cudaStream_t to run on (NULL: the legacy default stream).
 * The decision flag starts at 0 (route body A). */
int rc_init(rc_ctx **out, uint32_t S, const uint8_t *transition_table, uint32_t state_bytes,
            uint32_t payload_bytes, uint32_t max_K, uint64_t n_sessions, void *cuda_stream);

/* One cohort step on cohort 0 of *events, with route body = the context's
 * current decision flag; afterwards the flag holds this step's decision.
 *   state: device pointer, n_sessions records.
 *   K: cohort size, <= max_K (0 is allowed: nothing changes, the flag becomes 0).
 *   deadline_ns: latest admissible launch time of the cohort (Section 2.3);
 *     events->launch_ns > deadline_ns returns RC_E_DEADLINE and launches nothing.
 *   effects_out: K x 16 bytes, or NULL.
 * Asynchronous: does not synchronise. */
int rc_cohort_step(rc_ctx *ctx, void *state, const rc_events *events, uint32_t K,
                   int64_t deadline_ns, void *effects_out);

/* A chain of n_steps cohort steps; step n uses cohort n mod events->n_sets and
 * the route body chosen by the decision of step n - 1 (step 0: the context's
 * current flag).  Results are identical for every admissible mechanism.
 *   decisions_out: uint32 [n_steps], decision of each step; for RC_MECH_FLOOR
 *     it is READ instead: it holds the route sequence to replay (step n uses
 *     body decisions_out[n-1], step 0 the context flag).  May be NULL except
 *     for RC_MECH_FLOOR.
 *   effects_out: [n_steps][K] x 16 bytes, or NULL.
 *   state_log_out: [n_steps][K] x state_bytes, the record of each member after
 *     each step, or NULL.
 * Synchronises before returning; returns latched device errors. */
int rc_chain(rc_ctx *ctx, uint32_t n_steps, rc_mechanism mechanism, void *state, const rc_events *events,
             uint32_t K, uint32_t *decisions_out, void *effects_out, void *state_log_out);

/* Releases the context (synchronises its stream first).  NULL is accepted. */
int rc_free(rc_ctx *ctx);

/* Text of the last error on this context (never NULL; empty if none). */
const char *rc_last_error(rc_ctx *ctx);

/* Waits (bounded by the host wait limit) for the context stream and returns
   any latched device error, clearing it. */
int rc_sync(rc_ctx *ctx);

/* Reads (synchronising) or sets (asynchronously) the decision flag. */
int rc_get_decision(rc_ctx *ctx, uint32_t *sel_out);
int rc_set_decision(rc_ctx *ctx, uint32_t sel);

/* Bounds for waits: device spin waits (persistent grid barrier) give up after
   device_ns and latch RC_E_TIMEOUT; host waits give up after host_ns. */
int rc_set_wait_limits(rc_ctx *ctx, uint64_t device_ns, uint64_t host_ns);

/* Launch-floor probes used to express small-K latency as a multiple of the
 * platform floor.  kind: 0 = empty kernel launch + stream synchronise (host
 * clock); 1 = empty kernel node in a graph of reps back-to-back nodes (device
 * events); 2 = one iteration of an empty WHILE conditional graph (device
 * events); 3 = empty kernel + 4-byte device-to-host copy + synchronise (host
 * clock); 4 = one empty step of a persistent chain over one CTA per SM (reps
 * steps in one cooperative launch, each one grid barrier as the large-K
 * chain keys it; device events), the floor of a large-K step.  *us_out
 * receives microseconds per unit.  Kind 4 synchronises and returns
 * RC_E_TIMEOUT if a barrier wait ran out; other kinds return RC_E_INVAL for
 * an unknown kind. */
int rc_launch_floor(rc_ctx *ctx, int kind, uint32_t reps, double *us_out);

/* Device time of the last rc_chain's mechanism work, from CUDA events the
   library records on the context stream just before the first and just after
   the last operation of the mechanism (staging copies excluded), and the
   number of executions of this library's kernels that work caused (host or
   graph launched). */
int rc_last_chain_stats(rc_ctx *ctx, double *device_ms_out, uint32_t *kernel_launches_out);

/* Profiling aid: with a device buffer of at least 16 * n_steps int64 words
   set, the persistent kernels that support it record up to eight SM clock
   readings (clock64) per step at their phase boundaries: the grid kernels
   for their first and last CTA (layout [2][n_steps][8]), the single-CTA and
   single-warp ones for thread 0 (the first half); the two-step forms record
   at their even steps.  The phases are listed beside each kernel in the library
   source.  NULL (the default) turns it off. */
int rc_set_trace(rc_ctx *ctx, void *device_buf, uint64_t bytes);

/* Test hook (device-side bounded-wait check): when armed, CTA 1 of the next
   cooperative persistent launch skips its first barrier arrival, so the other
   CTAs' bounded waits run out and RC_E_TIMEOUT is latched. */
int rc_debug_skip_arrival(rc_ctx *ctx, uint32_t armed);

/* One cohort step that allocates nothing, for callers that cannot call
 * cudaMalloc: a serving process whose device memory is owned by another
 * allocator, or code that must not allocate (and so must not synchronise the
 * device) once it is running.  There is no counterpart in the paper; the
 * arithmetic is exactly that of rc_cohort_step.
 *   tables: DEVICE pointer to uint8 [2][S][8] (body A then B), 16-byte
 *     aligned, every entry < S; S a power of two in [2, 256].
 *   state (device, n_sessions records), events (device buffers, cohort 0
 *     used), effects_out (device, K x 16 bytes, or NULL) as for rc_cohort_step.
 *   flag: device uint32; read as this step's route body (0 = A, else B) and
 *     overwritten with the step's decision, so consecutive calls chain on the
 *     device without a host round trip.
 *   status_out: device uint32 or NULL; receives 0 or the positive code of the
 *     first bad member (4: state >= S or outcome >= 8, 7: index >= n_sessions).
 * Its only scratch is a fixed array in the library's device code (16.6 KB on
 * every GPU that loads the library, held until exit): up to 4,096 CTAs, so
 * K <= 1,048,576; a larger K returns RC_E_SIZE and launches nothing.  The
 * first call on a device resolves the array's device address (make that
 * first call before any stream capture).  Every call shares the array and it
 * keeps the previous call's contents: each call clears what must start at
 * zero, and calls that overlap on the GPU race.  Asynchronous on cuda_stream;
 * returns RC_OK, RC_E_INVAL, RC_E_SIZE or RC_E_CUDA. */
int rc_cohort_step_noalloc(const uint8_t *tables, uint32_t S, uint32_t state_bytes, uint32_t payload_bytes,
                           void *state, uint64_t n_sessions, const rc_events *events, uint32_t K,
                           uint32_t *flag, void *effects_out, uint32_t *status_out, void *cuda_stream);

/* ------------------------------------------------------------------------ */
/* Online cohort former (host).  Section 9.1 (online runtime queueing events
 * by route and deadline; A counts events launched by their deadline),
 * feasibility of Eq. 1.  Events must be pushed in (t_ns, event_id) order.
 * One open cohort per route with capacity and threshold K:
 *   - on an arrival for route r at now = t_ns, members of r's open cohort
 *     and of r's deferred queue with t + delta_ns < now go to fallback;
 *   - an event whose session already sits in r's open cohort is deferred;
 *   - the deferred queue (then the arrival) fills the open cohort in order;
 *     at K members the cohort launches with tau = now and the queue refills
 *     the next one.
 * Cohorts are returned in launch order.                                      */
typedef struct rc_former rc_former;

int rc_former_create(rc_former **out, uint32_t n_routes, uint32_t K, int64_t delta_ns);
/* Pushes one event.  Returns RC_E_INVAL on a route >= n_routes or an event
   out of (t_ns, event_id) order. */
int rc_former_push(rc_former *f, int64_t t_ns, uint32_t route, uint32_t session, int64_t event_id);
/* Pops the oldest launched cohort: members_out (K event ids in cohort order),
   *tau_out, *route_out.  Returns 1 if a cohort was popped, 0 if none is ready. */
int rc_former_pop(rc_former *f, int64_t *members_out, int64_t *tau_out, uint32_t *route_out);
/* Pushes n events with ids first_event_id, first_event_id + 1, ... in order;
   stops at the first rejected event and returns its RC_E_* code. */
int rc_former_push_many(rc_former *f, uint64_t n, const int64_t *t_ns, const uint32_t *route,
                        const uint32_t *session, int64_t first_event_id);
/* Pops up to max_cohorts launched cohorts into members_out [max_cohorts][K],
   tau_out and route_out (host arrays); returns how many were popped. */
int64_t rc_former_pop_many(rc_former *f, uint64_t max_cohorts, int64_t *members_out, int64_t *tau_out,
                           uint32_t *route_out);
/* Counters: events pushed, events launched, events dropped to fallback so far
   (events still open are neither). */
int rc_former_counts(rc_former *f, int64_t *pushed, int64_t *launched, int64_t *fallback);
int rc_former_free(rc_former *f);

/* Segmented step: one launch over several route-keyed cohorts (per-route
 * compaction with variable route bodies; Section 9.1 describes the route
 * service, and the scope paragraph of Section 10 lists what a single global
 * decision leaves out).  A context holds n_routes routes, each with its own
 * pair of bodies (tables: host [n_routes][2][S][8], entries < S; body A then
 * B) and its own decision flag (0 after rc_seg_init), resident in device
 * memory.  rc_seg_step transitions, in one launch, n_segments cohorts given
 * back to back in one event set: segment g holds members [seg_off[g],
 * seg_off[g+1]) of route seg_route[g].  Each member transitions as in
 * rc_cohort_step with its route's body T_r selected by flag[r]; then for
 * every segment d_g = (odd route keys in g) > floor(size_g / 2) (0 for an
 * empty segment) becomes flag[seg_route[g]] and decisions_out[g].
 * Contract: seg_route and seg_off are host arrays (n_segments and
 * n_segments + 1 words; seg_off[0] = 0, non-decreasing, total <=
 * max_members); a route appears at most once per step; sessions are distinct
 * across the whole step, so the segments commute.  state, events,
 * decisions_out (device, [n_segments] u32 or NULL) and effects_out (device,
 * [total][16] or NULL) as in rc_cohort_step.  Asynchronous on the context
 * stream; rc_seg_sync waits and returns a latched error (state >= S or
 * outcome >= 8: RC_E_STATE; index >= n_sessions: RC_E_INDEX; the text names
 * the segment and member).  RC_E_INVAL for a layout that breaks the
 * contract (nothing launched).                                              */
typedef struct rc_seg rc_seg;
int rc_seg_init(rc_seg **out, uint32_t n_routes, uint32_t S, const uint8_t *tables, uint32_t state_bytes,
                uint32_t payload_bytes, uint32_t max_members, uint32_t max_segments, uint64_t n_sessions,
                void *cuda_stream);
int rc_seg_step(rc_seg *ctx, void *state, const rc_events *events, uint32_t n_segments, const uint32_t *seg_route,
                const uint32_t *seg_off, uint32_t *decisions_out, void *effects_out);
int rc_seg_sync(rc_seg *ctx);
/* Flags of all routes (host [n_routes]); both synchronise. */
int rc_seg_get_flags(rc_seg *ctx, uint32_t *flags_out);
int rc_seg_set_flags(rc_seg *ctx, const uint32_t *flags);
const char *rc_seg_last_error(rc_seg *ctx);
int rc_seg_free(rc_seg *ctx);

/* Opportunity counts of an event set (host, Section 4), at threshold K and
 * deadline delta_ns for every route:
 *   fixed  events in (route, window) buckets holding >= K events, windows
 *          [origin_ns + w delta, origin_ns + (w + 1) delta) (Eq. 2, F);
 *   exact  the most events that batches of >= K same-route events, each
 *          spanning at most delta, can hold (Eq. 6, P*; computed by the
 *          deque recurrence of Algorithm 1);
 *   upper  events i for which some release tau in [t_i, t_i + delta] sees
 *          >= K same-route events in [tau - delta, tau] (Eqs. 3-4, U).
 * Shares are these counts over n; with the former's launched count A,
 * G = (P* - F) / (U - F) (Eq. 7) and R_A = (A - F) / (P* - F) (Eq. 9).
 * Inputs are host arrays of n events in any order; route < n_routes.
 * Returns RC_E_INVAL on K == 0, delta_ns <= 0 or a route out of range.   */
typedef struct {
    uint64_t n, fixed, exact, upper;
} rc_opportunity_counts;
int rc_opportunity(const int64_t *t_ns, const uint32_t *route, uint64_t n, uint32_t n_routes, uint32_t K,
                   int64_t delta_ns, int64_t origin_ns, rc_opportunity_counts *out);

/* The same three counts for every (delta, K) pair of a grid, on the GPU (the
 * exact-packing grid of Section 5.2: deadlines x thresholds per event set and
 * grouping).  One GPU thread per (route, delta) runs the fixed-window runs
 * and the U scan for every K, one per (route, delta, K) the P* recurrence,
 * over that route's times; the host groups the events by route (a counting
 * pass when they come in time order).  counts_out (host, u64
 * [n_delta][n_K][3]) receives {fixed, exact, upper} per pair.  Scratch of
 * 8 n n_delta n_K bytes is allocated and freed inside the call, which
 * synchronises cuda_stream.  RC_E_INVAL as for rc_opportunity, for n >= 2^31
 * or n_K > 32; RC_E_NOMEM when the scratch does not fit.                   */
int rc_opportunity_grid(const int64_t *t_ns, const uint32_t *route, uint64_t n, uint32_t n_routes,
                        const uint32_t *K_list, uint32_t n_K, const int64_t *delta_list, uint32_t n_delta,
                        int64_t origin_ns, uint64_t *counts_out, void *cuda_stream);

#ifdef __cplusplus
}
#endif

#endif /* RC_H */
