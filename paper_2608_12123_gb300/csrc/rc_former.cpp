// rc_former.cpp -- online cohort former of librc.so (declared in include/rc.h).
//
// Feeds the cohort step: packs arrivals into deadline-feasible cohorts of K
// events of one route (Eq. 1 with |B| = K; Section 9.1's online runtime that
// queues events by route and launch deadline).  Events arrive in (t, id)
// order.  Per route there is one open cohort and one queue of deferred events
// (events whose session already sits in the open cohort).  On an arrival at
// time now for route r:
//   1. members of r's open cohort and of r's deferred queue whose deadline
//      t + delta is before now are dropped to fallback (deadlines are
//      inclusive on the integer clock, Section 4);
//   2. the arrival joins the tail of r's deferred queue;
//   3. the queue is drained in order into the open cohort, skipping events
//      whose session is already in it; when the cohort reaches K it launches
//      at tau = now and the drain restarts from the queue head.
#include <stdint.h>

#include <deque>
#include <new>
#include <unordered_set>
#include <vector>

#include "rc.h"

namespace {

struct Pending {
    int64_t t;
    int64_t id;
    uint32_t session;
};

struct RouteState {
    std::vector<Pending> open;               // open cohort, in joining order
    std::unordered_set<uint32_t> sessions;   // sessions in the open cohort
    int64_t open_min_t = INT64_MAX;          // earliest release in the open cohort
    std::deque<Pending> deferred;
};

struct Cohort {
    std::vector<int64_t> members;
    int64_t tau;
    uint32_t route;
};

}  // namespace

struct rc_former {
    uint32_t n_routes = 0;
    uint32_t K = 0;
    int64_t delta = 0;
    std::vector<RouteState> routes;
    std::deque<Cohort> ready;
    bool have_last = false;
    int64_t last_t = 0, last_id = 0;
    int64_t pushed = 0, launched = 0, fallback = 0;

    void purge(RouteState &rs, int64_t now) {
        if (rs.open_min_t != INT64_MAX && rs.open_min_t + delta < now) {
            size_t keep = 0;
            int64_t mn = INT64_MAX;
            for (size_t k = 0; k < rs.open.size(); ++k) {
                const Pending &p = rs.open[k];
                if (p.t + delta < now) {
                    rs.sessions.erase(p.session);
                    ++fallback;
                } else {
                    rs.open[keep++] = p;
                    if (p.t < mn) mn = p.t;
                }
            }
            rs.open.resize(keep);
            rs.open_min_t = mn;
        }
        for (auto it = rs.deferred.begin(); it != rs.deferred.end();) {
            if (it->t + delta < now) {
                it = rs.deferred.erase(it);
                ++fallback;
            } else {
                ++it;
            }
        }
    }

    void launch(RouteState &rs, uint32_t r, int64_t now) {
        Cohort c;
        c.members.reserve(K);
        for (const Pending &p : rs.open) c.members.push_back(p.id);
        c.tau = now;
        c.route = r;
        ready.push_back(std::move(c));
        launched += K;
        rs.open.clear();
        rs.sessions.clear();
        rs.open_min_t = INT64_MAX;
    }

    void drain(RouteState &rs, uint32_t r, int64_t now) {
        for (auto it = rs.deferred.begin(); it != rs.deferred.end();) {
            if (rs.sessions.count(it->session)) {
                ++it;
                continue;
            }
            rs.open.push_back(*it);
            rs.sessions.insert(it->session);
            if (it->t < rs.open_min_t) rs.open_min_t = it->t;
            it = rs.deferred.erase(it);
            if (rs.open.size() == K) {
                launch(rs, r, now);
                it = rs.deferred.begin();
            }
        }
    }
};

extern "C" {

int rc_former_create(rc_former **out, uint32_t n_routes, uint32_t K, int64_t delta_ns) {
    if (!out || n_routes == 0 || K == 0 || delta_ns < 0) return RC_E_INVAL;
    rc_former *f = new (std::nothrow) rc_former();
    if (!f) return RC_E_NOMEM;
    f->n_routes = n_routes;
    f->K = K;
    f->delta = delta_ns;
    f->routes.resize(n_routes);
    *out = f;
    return RC_OK;
}

int rc_former_push(rc_former *f, int64_t t_ns, uint32_t route, uint32_t session, int64_t event_id) {
    if (!f || route >= f->n_routes) return RC_E_INVAL;
    if (f->have_last && (t_ns < f->last_t || (t_ns == f->last_t && event_id <= f->last_id))) return RC_E_INVAL;
    f->have_last = true;
    f->last_t = t_ns;
    f->last_id = event_id;
    ++f->pushed;
    RouteState &rs = f->routes[route];
    f->purge(rs, t_ns);
    rs.deferred.push_back(Pending{t_ns, event_id, session});
    f->drain(rs, route, t_ns);
    return RC_OK;
}

int rc_former_pop(rc_former *f, int64_t *members_out, int64_t *tau_out, uint32_t *route_out) {
    if (!f || !members_out || !tau_out || !route_out) return RC_E_INVAL;
    if (f->ready.empty()) return 0;
    const Cohort &c = f->ready.front();
    for (uint32_t k = 0; k < f->K; ++k) members_out[k] = c.members[k];
    *tau_out = c.tau;
    *route_out = c.route;
    f->ready.pop_front();
    return 1;
}

int rc_former_push_many(rc_former *f, uint64_t n, const int64_t *t_ns, const uint32_t *route,
                        const uint32_t *session, int64_t first_event_id) {
    if (!f || (n && (!t_ns || !route || !session))) return RC_E_INVAL;
    for (uint64_t i = 0; i < n; ++i) {
        const int rc = rc_former_push(f, t_ns[i], route[i], session[i], first_event_id + static_cast<int64_t>(i));
        if (rc != RC_OK) return rc;
    }
    return RC_OK;
}

int64_t rc_former_pop_many(rc_former *f, uint64_t max_cohorts, int64_t *members_out, int64_t *tau_out,
                           uint32_t *route_out) {
    if (!f || (max_cohorts && (!members_out || !tau_out || !route_out))) return RC_E_INVAL;
    int64_t got = 0;
    while (static_cast<uint64_t>(got) < max_cohorts &&
           rc_former_pop(f, members_out + static_cast<size_t>(got) * f->K, tau_out + got, route_out + got) == 1)
        ++got;
    return got;
}

int rc_former_counts(rc_former *f, int64_t *pushed, int64_t *launched, int64_t *fallback) {
    if (!f) return RC_E_INVAL;
    if (pushed) *pushed = f->pushed;
    if (launched) *launched = f->launched;
    if (fallback) *fallback = f->fallback;
    return RC_OK;
}

int rc_former_free(rc_former *f) {
    delete f;
    return RC_OK;
}

}  // extern "C"
