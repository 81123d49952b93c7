/*
 * rc_oracle.c -- plain, slow CPU oracle for the ready-cohort transition path.
 *
 * TEST INFRASTRUCTURE.  Only the tests, the package smoke check and the
 * CPU-baseline leg of the benchmark call this code; the product path never
 * does.  It shares no code, header, table or constant generator with the CUDA
 * path.  Every function is the plain definition (or the paper's algorithm, in
 * the paper's order) written out, single-threaded, with no blocking or fusion.
 *
 * Parts and the passages they follow (arXiv 2608.12123, "Ready Cohorts"):
 *   transition unit ........ Section 2.1 (state + event -> new state, route, effect)
 *   two route bodies, one global binary decision per epoch ... Section 7.1
 *   exactness contract ..... Sections 2.2 and 7.3 (every state field, every decision)
 *   feasible batch ......... Eq. 1          fixed-partition share F ... Eq. 2
 *   active count, U ........ Eqs. 3-4       online share A ............ Section 3.2, Eq. 8
 *   exact share P* ......... Eq. 6 (direct) and Algorithm 1 (monotone deque)
 *   integer-ns clock, inclusive comparisons ... Section 4, "Exact clock"
 *
 * The paper does not define the route-key hash, the state update, the effect
 * record or the cohort former's tie rules.  The readings used here:
 *   mix64(z)   = SplitMix64 output finaliser (Steele, Lea, Flood, OOPSLA 2014)
 *   route key  = h0 = mix64((x | o << 32) XOR gamma), then h = mix64(h XOR w_k)
 *                for each little-endian 64-bit payload word w_k in order;
 *                x is the state BEFORE the transition
 *   transition = y = T_sel[x][o]; step += 1 (mod 2^32);
 *                acc = (acc XOR rk) * gamma                     (16-byte record)
 *                acc[j] = (acc[j] XOR rotl(rk, 8j)) * gamma      (64-byte record, j = 0..6)
 *   effect     = { rk (u64), session (u32), y | o << 16 | sel << 24 (u32) }
 *   decision   = (number of members with odd rk) > floor(K / 2), strictly
 *   chain      = sel_0 given, sel_{n+1} = d_n
 * Parity of the paper's own trace figures (F = 30.19 %, P* = 43.00 %, ...) is
 * unpinned: they need the public trace panel, which is not reproduced here.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_E_INVAL (-1)
#define ORC_E_STATE (-4)
#define ORC_E_INDEX (-7)
#define ORC_E_NOMEM (-8)

static const uint64_t ORC_GAMMA = 0x9E3779B97F4A7C15ull;

/* ------------------------------------------------------------------------- */
/* Route key                                                                  */
/* ------------------------------------------------------------------------- */

/* SplitMix64 finaliser, exactly as published (xor-shift 30, multiply,
   xor-shift 27, multiply, xor-shift 31; arithmetic mod 2^64). */
static uint64_t mix64(uint64_t z)
{
    z = z ^ (z >> 30);
    z = z * 0xBF58476D1CE4E5B9ull;
    z = z ^ (z >> 27);
    z = z * 0x94D049BB133111EBull;
    z = z ^ (z >> 31);
    return z;
}

uint64_t orc_mix64(uint64_t z) { return mix64(z); }

static uint64_t get_le64(const uint8_t *p)
{
    uint64_t w = 0;
    for (int b = 0; b < 8; ++b) w |= (uint64_t)p[b] << (8 * b);
    return w;
}

static uint32_t get_le32(const uint8_t *p)
{
    uint32_t w = 0;
    for (int b = 0; b < 4; ++b) w |= (uint32_t)p[b] << (8 * b);
    return w;
}

static void put_le64(uint8_t *p, uint64_t w)
{
    for (int b = 0; b < 8; ++b) p[b] = (uint8_t)(w >> (8 * b));
}

static void put_le32(uint8_t *p, uint32_t w)
{
    for (int b = 0; b < 4; ++b) p[b] = (uint8_t)(w >> (8 * b));
}

/* Route key of one event (Section 2.1: the transition routes the outcome).
   x: the session's state before the transition; o: outcome class;
   payload: P bytes, read as P/8 little-endian words. */
uint64_t orc_route_key(uint32_t x, uint32_t o, const uint8_t *payload, uint32_t P)
{
    uint64_t packed = (uint64_t)x | ((uint64_t)o << 32);
    uint64_t h = mix64(packed ^ ORC_GAMMA);
    for (uint32_t k = 0; k < P / 8; ++k)
        h = mix64(h ^ get_le64(payload + 8 * (size_t)k));
    return h;
}

static uint64_t rotl64(uint64_t v, unsigned r)
{
    r &= 63u;
    if (r == 0) return v;
    return (v << r) | (v >> (64u - r));
}

/* ------------------------------------------------------------------------- */
/* One cohort step: Sections 2.1 and 7.1                                      */
/* ------------------------------------------------------------------------- */

/* Applies the transition to every member of one cohort, in member order.
 *   tables: uint8 [2][S][8] (route body A, then B); sel picks the body.
 *   state:  N records of SB bytes (16: {i32 state, u32 step, u64 acc};
 *           64: {i32 state, u32 step, u64 acc[7]}), updated in place.
 *   outcome[K], payload[K][P], idx[K] (NULL: member m is session m).
 *   effects (K x 16 bytes) and member_state (K x SB bytes, the record after
 *   the update) may be NULL.
 * Returns ORC_OK and the decision in *d_out, or an error code on the first
 * member whose state, outcome or session index is out of range (the oracle
 * stops there; state up to that member has been updated). */
int orc_cohort_step(uint32_t S, const uint8_t *tables, uint32_t SB, uint8_t *state, uint64_t N,
                    const uint32_t *outcome, const uint8_t *payload, uint32_t P,
                    const uint32_t *idx, uint32_t K, uint32_t sel,
                    uint8_t *effects, uint8_t *member_state, uint32_t *d_out)
{
    if ((SB != 16 && SB != 64) || (P % 8) != 0 || sel > 1 || S == 0 || S > 256) return ORC_E_INVAL;
    uint32_t odd = 0;
    for (uint32_t m = 0; m < K; ++m) {
        uint64_t s = idx ? (uint64_t)idx[m] : (uint64_t)m;
        if (s >= N) return ORC_E_INDEX;
        uint8_t *rec = state + s * SB;
        uint32_t x = get_le32(rec + 0);
        uint32_t step = get_le32(rec + 4);
        uint32_t o = outcome[m];
        if (x >= S || o >= 8) return ORC_E_STATE;
        uint64_t rk = orc_route_key(x, o, payload + (size_t)m * P, P);
        uint32_t y = tables[(size_t)sel * S * 8 + (size_t)x * 8 + o];
        put_le32(rec + 0, y);
        put_le32(rec + 4, step + 1u);
        if (SB == 16) {
            uint64_t acc = get_le64(rec + 8);
            put_le64(rec + 8, (acc ^ rk) * ORC_GAMMA);
        } else {
            for (unsigned j = 0; j < 7; ++j) {
                uint64_t acc = get_le64(rec + 8 + 8 * j);
                put_le64(rec + 8 + 8 * j, (acc ^ rotl64(rk, 8 * j)) * ORC_GAMMA);
            }
        }
        if (effects) {
            uint8_t *e = effects + (size_t)m * 16;
            put_le64(e + 0, rk);
            put_le32(e + 8, (uint32_t)s);
            put_le32(e + 12, y | (o << 16) | (sel << 24));
        }
        if (member_state) memcpy(member_state + (size_t)m * SB, rec, SB);
        odd += (uint32_t)(rk & 1u);
    }
    *d_out = (odd > K / 2) ? 1u : 0u;
    return ORC_OK;
}

/* A chain of n_steps cohort steps.  Step n uses event set n mod n_sets
 * (outcome[n_sets][K], payload[n_sets][K][P], idx[n_sets][K] or NULL) and
 * route body sel_n, where sel_0 = sel0 and sel_{n+1} = d_n: the decision of
 * one step selects the body of the next (Section 7.1, device-resident path).
 * decisions[n] receives d_n; effects_log [n_steps][K][16] and state_log
 * [n_steps][K][SB] may be NULL.  *sel_out receives the last decision. */
int orc_chain(uint32_t S, const uint8_t *tables, uint32_t SB, uint8_t *state, uint64_t N,
              const uint32_t *outcome, const uint8_t *payload, uint32_t P, const uint32_t *idx,
              uint32_t n_sets, uint32_t K, uint32_t n_steps, uint32_t sel0,
              uint32_t *decisions, uint8_t *effects_log, uint8_t *state_log, uint32_t *sel_out)
{
    if (n_sets == 0) n_sets = 1;
    uint32_t sel = sel0;
    for (uint32_t n = 0; n < n_steps; ++n) {
        size_t set = n % n_sets;
        uint32_t d = 0;
        int rc = orc_cohort_step(S, tables, SB, state, N,
                                 outcome + set * K, payload + set * K * (size_t)P, P,
                                 idx ? idx + set * K : NULL, K, sel,
                                 effects_log ? effects_log + (size_t)n * K * 16 : NULL,
                                 state_log ? state_log + (size_t)n * K * SB : NULL, &d);
        if (rc != ORC_OK) return rc;
        if (decisions) decisions[n] = d;
        sel = d;
    }
    if (sel_out) *sel_out = sel;
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* Event ordering helpers                                                     */
/* ------------------------------------------------------------------------- */

typedef struct {
    int64_t t;
    uint32_t route;
    int64_t id;
} ev_t;

static int cmp_route_t_id(const void *a, const void *b)
{
    const ev_t *x = (const ev_t *)a, *y = (const ev_t *)b;
    if (x->route != y->route) return x->route < y->route ? -1 : 1;
    if (x->t != y->t) return x->t < y->t ? -1 : 1;
    if (x->id != y->id) return x->id < y->id ? -1 : 1;
    return 0;
}

static int cmp_t_id(const void *a, const void *b)
{
    const ev_t *x = (const ev_t *)a, *y = (const ev_t *)b;
    if (x->t != y->t) return x->t < y->t ? -1 : 1;
    if (x->id != y->id) return x->id < y->id ? -1 : 1;
    return 0;
}

/* Events sorted by (route, t, id); grp[r]..grp[r+1]-1 are route r's events. */
static ev_t *group_by_route(int64_t n, const int64_t *t, const uint32_t *route, uint32_t R,
                            int64_t **grp_out)
{
    ev_t *ev = (ev_t *)malloc(sizeof(ev_t) * (size_t)(n > 0 ? n : 1));
    int64_t *grp = (int64_t *)calloc((size_t)R + 1, sizeof(int64_t));
    if (!ev || !grp) { free(ev); free(grp); return NULL; }
    for (int64_t i = 0; i < n; ++i) { ev[i].t = t[i]; ev[i].route = route[i]; ev[i].id = i; }
    qsort(ev, (size_t)n, sizeof(ev_t), cmp_route_t_id);
    for (int64_t i = 0; i < n; ++i) grp[ev[i].route + 1]++;
    for (uint32_t r = 0; r < R; ++r) grp[r + 1] += grp[r];
    *grp_out = grp;
    return ev;
}

static int routes_in_range(int64_t n, const uint32_t *route, uint32_t R)
{
    for (int64_t i = 0; i < n; ++i)
        if (route[i] >= R) return 0;
    return 1;
}

/* ------------------------------------------------------------------------- */
/* F: fixed-partition share, Eq. 2                                            */
/* ------------------------------------------------------------------------- */

typedef struct {
    int64_t window;
    uint32_t route;
} bucket_t;

static int cmp_bucket(const void *a, const void *b)
{
    const bucket_t *x = (const bucket_t *)a, *y = (const bucket_t *)b;
    if (x->window != y->window) return x->window < y->window ? -1 : 1;
    if (x->route != y->route) return x->route < y->route ? -1 : 1;
    return 0;
}

static int64_t floor_div(int64_t a, int64_t b)
{
    int64_t q = a / b;
    if ((a % b != 0) && ((a < 0) != (b < 0))) --q;
    return q;
}

/* Number of events in buckets (window, route) holding at least K_r events.
   Windows are half-open [origin + w*delta, origin + (w+1)*delta)
   (Section 5.2: origin-aligned half-open windows of width delta). */
int64_t orc_fixed_count(int64_t n, const int64_t *t, const uint32_t *route, uint32_t R,
                        const uint32_t *Kr, int64_t delta, int64_t origin)
{
    if (delta <= 0 || !routes_in_range(n, route, R)) return ORC_E_INVAL;
    bucket_t *b = (bucket_t *)malloc(sizeof(bucket_t) * (size_t)(n > 0 ? n : 1));
    if (!b) return ORC_E_NOMEM;
    for (int64_t i = 0; i < n; ++i) {
        b[i].window = floor_div(t[i] - origin, delta);
        b[i].route = route[i];
    }
    qsort(b, (size_t)n, sizeof(bucket_t), cmp_bucket);
    int64_t count = 0;
    for (int64_t i = 0; i < n;) {
        int64_t j = i;
        while (j < n && b[j].window == b[i].window && b[j].route == b[i].route) ++j;
        int64_t nb = j - i;
        if (nb >= (int64_t)Kr[b[i].route]) count += nb;
        i = j;
    }
    free(b);
    return count;
}

/* ------------------------------------------------------------------------- */
/* U: local-overlap bound, Eqs. 3-4                                           */
/* ------------------------------------------------------------------------- */

/* first position p in [lo, hi) with a[p].t >= v */
static int64_t lower_bound_t(const ev_t *a, int64_t lo, int64_t hi, int64_t v)
{
    while (lo < hi) {
        int64_t mid = lo + (hi - lo) / 2;
        if (a[mid].t < v) lo = mid + 1; else hi = mid;
    }
    return lo;
}

/* first position p in [lo, hi) with a[p].t > v */
static int64_t upper_bound_t(const ev_t *a, int64_t lo, int64_t hi, int64_t v)
{
    while (lo < hi) {
        int64_t mid = lo + (hi - lo) / 2;
        if (a[mid].t <= v) lo = mid + 1; else hi = mid;
    }
    return lo;
}

/* Number of events i with max over tau in [t_i, t_i + delta] of
   Q_r(tau) >= K_r, where Q_r(tau) = #{j on route r : t_j <= tau <= t_j + delta}.
   Q_r only rises at a release, so the maximum over the closed interval is
   attained at a release time inside it (t_i itself included).  eligible (n
   bytes, optional) receives the per-event indicator. */
int64_t orc_upper_count(int64_t n, const int64_t *t, const uint32_t *route, uint32_t R,
                        const uint32_t *Kr, int64_t delta, uint8_t *eligible)
{
    if (delta < 0 || !routes_in_range(n, route, R)) return ORC_E_INVAL;
    int64_t *grp = NULL;
    ev_t *ev = group_by_route(n, t, route, R, &grp);
    if (!ev) return ORC_E_NOMEM;
    int64_t *W = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n > 0 ? n : 1));
    if (!W) { free(ev); free(grp); return ORC_E_NOMEM; }
    int64_t count = 0;
    for (uint32_t r = 0; r < R; ++r) {
        int64_t lo = grp[r], hi = grp[r + 1];
        /* W[p] = Q_r(t_p) = #{k : t_p - delta <= t_k <= t_p} */
        for (int64_t p = lo; p < hi; ++p)
            W[p] = upper_bound_t(ev, lo, hi, ev[p].t) - lower_bound_t(ev, lo, hi, ev[p].t - delta);
        for (int64_t p = lo; p < hi; ++p) {
            int64_t best = 0;
            for (int64_t q = lower_bound_t(ev, lo, hi, ev[p].t); q < hi && ev[q].t <= ev[p].t + delta; ++q)
                if (W[q] > best) best = W[q];
            int ok = best >= (int64_t)Kr[r];
            count += ok;
            if (eligible) eligible[ev[p].id] = (uint8_t)ok;
        }
    }
    free(W);
    free(ev);
    free(grp);
    return count;
}

/* ------------------------------------------------------------------------- */
/* P*: exact offline share for equal relative deadlines, Section 4            */
/* ------------------------------------------------------------------------- */

/* Eq. 6 evaluated directly on one route's sorted releases t[1..n]:
   D[j] = max(D[j-1], max over i <= j-K+1 with t_j - t_i <= delta of
              D[i-1] + j - i + 1).  O(n * window). */
static int64_t dp_direct(const ev_t *a, int64_t n, int64_t K, int64_t delta, int64_t *D)
{
    D[0] = 0;
    for (int64_t j = 1; j <= n; ++j) {
        D[j] = D[j - 1];
        for (int64_t i = j - K + 1; i >= 1; --i) {
            if (a[j - 1].t - a[i - 1].t > delta) break;
            int64_t v = D[i - 1] + (j - i + 1);
            if (v > D[j]) D[j] = v;
        }
    }
    return D[n];
}

/* Algorithm 1 on one route: a monotone deque over candidate starts i holding
   D[i-1] - i + 1, a left boundary from LowerBound(t, t_j - delta), and
   D[j] = max(D[j-1], j + head value).  start_of[j] (1-based) records the
   block start that achieves D[j], or 0 when D[j] = D[j-1] (ties prefer the
   skip, which keeps the fewest events in batches among equal choices). */
static int64_t dp_deque(const ev_t *a, int64_t n, int64_t K, int64_t delta, int64_t *D,
                        int64_t *start_of, int64_t *dq_i, int64_t *dq_v)
{
    int64_t head = 0, tail = 0; /* deque occupies [head, tail) */
    D[0] = 0;
    start_of[0] = 0;
    for (int64_t j = 1; j <= n; ++j) {
        D[j] = D[j - 1];
        start_of[j] = 0;
        int64_t i = j - K + 1;
        if (i >= 1) {
            int64_t v = D[i - 1] - i + 1;
            while (tail > head && dq_v[tail - 1] <= v) --tail;
            dq_i[tail] = i;
            dq_v[tail] = v;
            ++tail;
        }
        /* LowerBound: first 1-based index l with t_l >= t_j - delta */
        int64_t l = lower_bound_t(a, 0, n, a[j - 1].t - delta) + 1;
        while (tail > head && dq_i[head] < l) ++head;
        if (tail > head && j + dq_v[head] > D[j]) {
            D[j] = j + dq_v[head];
            start_of[j] = dq_i[head];
        }
    }
    return D[n];
}

/* Exact assigned-event count over all routes (Lemma 1: each route packs
   independently into contiguous blocks).  method 0: Algorithm 1 with a
   witness written to batch_of (n entries: batch number, or -1 when the event
   is left out; may be NULL); method 1: Eq. 6 directly, no witness.
   *n_batches receives the witness's batch count (method 0). */
int64_t orc_exact_count(int64_t n, const int64_t *t, const uint32_t *route, uint32_t R,
                        const uint32_t *Kr, int64_t delta, int method,
                        int64_t *batch_of, int64_t *n_batches)
{
    if (delta < 0 || !routes_in_range(n, route, R)) return ORC_E_INVAL;
    for (uint32_t r = 0; r < R; ++r)
        if (Kr[r] == 0) return ORC_E_INVAL;
    int64_t *grp = NULL;
    ev_t *ev = group_by_route(n, t, route, R, &grp);
    if (!ev) return ORC_E_NOMEM;
    size_t cap = (size_t)(n + 1);
    int64_t *D = (int64_t *)malloc(sizeof(int64_t) * cap);
    int64_t *st = (int64_t *)malloc(sizeof(int64_t) * cap);
    int64_t *dqi = (int64_t *)malloc(sizeof(int64_t) * cap);
    int64_t *dqv = (int64_t *)malloc(sizeof(int64_t) * cap);
    if (!D || !st || !dqi || !dqv) {
        free(D); free(st); free(dqi); free(dqv); free(ev); free(grp);
        return ORC_E_NOMEM;
    }
    if (batch_of)
        for (int64_t i = 0; i < n; ++i) batch_of[i] = -1;
    int64_t total = 0, nb = 0;
    for (uint32_t r = 0; r < R; ++r) {
        int64_t lo = grp[r], m = grp[r + 1] - grp[r];
        if (m == 0) continue;
        if (method == 1) {
            total += dp_direct(ev + lo, m, (int64_t)Kr[r], delta, D);
            continue;
        }
        total += dp_deque(ev + lo, m, (int64_t)Kr[r], delta, D, st, dqi, dqv);
        /* back-pointers recover one maximum-cardinality set of blocks */
        for (int64_t j = m; j > 0;) {
            if (st[j] == 0) { --j; continue; }
            for (int64_t p = st[j]; p <= j; ++p)
                if (batch_of) batch_of[ev[lo + p - 1].id] = nb;
            ++nb;
            j = st[j] - 1;
        }
    }
    if (n_batches) *n_batches = nb;
    free(D); free(st); free(dqi); free(dqv); free(ev); free(grp);
    return total;
}

/* ------------------------------------------------------------------------- */
/* Online cohort former and A (Sections 3.2 and 9.1)                          */
/* ------------------------------------------------------------------------- */

/* An online former with one open cohort per route, capacity and threshold K:
 *   - events are taken in (t, event id) order; now = t of the arrival;
 *   - on an arrival for route r, members of r's open cohort (and r's deferred
 *     queue) whose deadline t + delta is before now are dropped to fallback;
 *   - an event whose session is already in r's open cohort waits in r's
 *     deferred queue (so a cohort never holds one session twice);
 *   - when the open cohort reaches K members it launches at tau = now, then
 *     the deferred queue refills the fresh cohort in order (and may launch
 *     again at the same now);
 *   - whatever is left at the end of the horizon is fallback.
 * Every launched cohort satisfies Eq. 1 with |B| = K.  Outputs, for at most
 * cap cohorts in launch order: members[c*K + k] (event ids, in cohort order),
 * tau[c], croute[c].  Returns the number of cohorts formed (which may exceed
 * cap; only the first cap are written) or a negative error. */
int64_t orc_former(int64_t n, const int64_t *t, const uint32_t *route, const uint32_t *session,
                   uint32_t R, uint32_t K, int64_t delta,
                   int64_t *members, int64_t *tau, uint32_t *croute, int64_t cap)
{
    if (K == 0 || delta < 0 || !routes_in_range(n, route, R)) return ORC_E_INVAL;
    ev_t *ord = (ev_t *)malloc(sizeof(ev_t) * (size_t)(n > 0 ? n : 1));
    int64_t *open = (int64_t *)malloc(sizeof(int64_t) * (size_t)R * K);
    int64_t *open_n = (int64_t *)calloc(R, sizeof(int64_t));
    int64_t *dq = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n > 0 ? n : 1));  /* all deferred queues, per-route linked */
    int64_t *dq_next = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n > 0 ? n : 1));
    int64_t *dq_head = (int64_t *)malloc(sizeof(int64_t) * R);
    int64_t *dq_tail = (int64_t *)malloc(sizeof(int64_t) * R);
    if (!ord || !open || !open_n || !dq || !dq_next || !dq_head || !dq_tail) {
        free(ord); free(open); free(open_n); free(dq); free(dq_next); free(dq_head); free(dq_tail);
        return ORC_E_NOMEM;
    }
    for (uint32_t r = 0; r < R; ++r) { dq_head[r] = -1; dq_tail[r] = -1; }
    int64_t dq_used = 0;
    for (int64_t i = 0; i < n; ++i) { ord[i].t = t[i]; ord[i].route = route[i]; ord[i].id = i; }
    qsort(ord, (size_t)n, sizeof(ev_t), cmp_t_id);
    int64_t nc = 0;

    for (int64_t a = 0; a < n; ++a) {
        int64_t e = ord[a].id, now = ord[a].t;
        uint32_t r = ord[a].route;
        int64_t *coh = open + (size_t)r * K;
        /* purge expired members (inclusive deadline: kept while now <= t + delta) */
        int64_t keep = 0;
        for (int64_t k = 0; k < open_n[r]; ++k)
            if (!(t[coh[k]] + delta < now)) coh[keep++] = coh[k];
        open_n[r] = keep;
        /* purge expired deferred events */
        {
            int64_t prev = -1, cur = dq_head[r];
            while (cur != -1) {
                int64_t nx = dq_next[cur];
                if (t[dq[cur]] + delta < now) {
                    if (prev == -1) dq_head[r] = nx; else dq_next[prev] = nx;
                    if (dq_tail[r] == cur) dq_tail[r] = prev;
                } else {
                    prev = cur;
                }
                cur = nx;
            }
        }
        /* the arrival joins the deferred queue's tail; then the queue is
           drained in order into the open cohort */
        dq[dq_used] = e;
        dq_next[dq_used] = -1;
        if (dq_tail[r] == -1) dq_head[r] = dq_used; else dq_next[dq_tail[r]] = dq_used;
        dq_tail[r] = dq_used;
        ++dq_used;
        int progress = 1;
        while (progress) {
            progress = 0;
            int64_t prev = -1, cur = dq_head[r];
            while (cur != -1) {
                int64_t nx = dq_next[cur];
                int64_t ev_id = dq[cur];
                int dup = 0;
                for (int64_t k = 0; k < open_n[r]; ++k)
                    if (session[coh[k]] == session[ev_id]) { dup = 1; break; }
                if (dup) { prev = cur; cur = nx; continue; }
                /* unlink and append to the cohort */
                if (prev == -1) dq_head[r] = nx; else dq_next[prev] = nx;
                if (dq_tail[r] == cur) dq_tail[r] = prev;
                coh[open_n[r]++] = ev_id;
                if (open_n[r] == (int64_t)K) {
                    if (nc < cap) {
                        for (uint32_t k = 0; k < K; ++k) members[(size_t)nc * K + k] = coh[k];
                        tau[nc] = now;
                        croute[nc] = r;
                    }
                    ++nc;
                    open_n[r] = 0;
                    progress = 1;   /* a fresh cohort: rescan the queue from its head */
                    break;
                }
                cur = nx;
            }
        }
    }
    free(ord); free(open); free(open_n); free(dq); free(dq_next); free(dq_head); free(dq_tail);
    return nc;
}
