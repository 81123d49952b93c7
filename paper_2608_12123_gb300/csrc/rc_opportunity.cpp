// rc_opportunity.cpp -- opportunity counts of an event set (Section 4):
// fixed windows F (Eq. 2), the exact offline packing P* (Eq. 6, computed by
// the monotone-deque recurrence of Algorithm 1) and the upper bound U
// (Eqs. 3-4), at one threshold K and one deadline delta for every route.
//
// Host code of librc.so beside the online former; it serves the measurement
// of how much of a workload the resident cohort path can reach, and shares no
// code with any other implementation of these quantities.

#include <stdint.h>

#include <algorithm>
#include <deque>
#include <numeric>
#include <vector>

#include "rc.h"

namespace {

// Floor division toward minus infinity (windows before the origin are
// numbered negatively, not folded onto window 0).
int64_t floor_div(int64_t a, int64_t b) {
    const int64_t q = a / b;
    return (a % b != 0 && ((a < 0) != (b < 0))) ? q - 1 : q;
}

// Eq. 2: an event counts when its (route, window) bucket holds at least K
// events; windows are [origin + w delta, origin + (w + 1) delta).
uint64_t fixed_count(const std::vector<int64_t> &ts, uint32_t K, int64_t delta, int64_t origin) {
    // ts: one route's times in ascending order, so buckets are runs
    uint64_t served = 0;
    size_t a = 0;
    while (a < ts.size()) {
        const int64_t w = floor_div(ts[a] - origin, delta);
        size_t b = a + 1;
        while (b < ts.size() && floor_div(ts[b] - origin, delta) == w) ++b;
        if (b - a >= K) served += b - a;
        a = b;
    }
    return served;
}

// Eqs. 3-4: event i counts when some release time tau in [t_i, t_i + delta]
// sees at least K same-route events in [tau - delta, tau].  The count
// W(tau) only rises at a release, so the releases t_j themselves are the
// times to look at: W_j = #{k : t_j - delta <= t_k <= t_j}, and event i
// counts when max{W_j : t_i <= t_j <= t_i + delta} >= K.  Both ends of that
// range move forward with i, so a monotone deque gives the maxima.
uint64_t upper_count(const std::vector<int64_t> &ts, uint32_t K, int64_t delta) {
    const size_t n = ts.size();
    if (n == 0) return 0;
    std::vector<uint64_t> W(n);
    size_t lo = 0, hi = 0;  // [lo, hi): times in [t_j - delta, t_j] (ties included)
    for (size_t j = 0; j < n; ++j) {
        while (hi < n && ts[hi] <= ts[j]) ++hi;
        while (ts[lo] < ts[j] - delta) ++lo;
        W[j] = hi - lo;
    }
    uint64_t served = 0;
    std::deque<size_t> dq;  // indices j with decreasing W
    size_t first = 0, end = 0;  // window [first, end) = {j : t_i <= t_j <= t_i + delta}
    for (size_t i = 0; i < n; ++i) {
        while (first < n && ts[first] < ts[i]) ++first;
        while (end < n && ts[end] <= ts[i] + delta) {
            while (!dq.empty() && W[dq.back()] <= W[end]) dq.pop_back();
            dq.push_back(end);
            ++end;
        }
        while (!dq.empty() && dq.front() < first) dq.pop_front();
        if (!dq.empty() && W[dq.front()] >= K) ++served;
    }
    return served;
}

// Eq. 6 / Algorithm 1: the largest number of events that batches of at least
// K events, each spanning at most delta, can hold, over one route's sorted
// times.  D[j] = max(D[j-1], max{D[i-1] + (j - i + 1) : i <= j - K + 1 and
// t_i >= t_j - delta}); the inner maximum is D[i-1] - i + 1 plus j, kept in
// a deque of candidates i with decreasing D[i-1] - i + 1 (a new candidate
// removes the tail candidates it is at least as good as; the head leaves
// once t_i < t_j - delta).  Indices here are 1-based as in the paper.
uint64_t exact_count(const std::vector<int64_t> &ts, uint32_t K, int64_t delta) {
    const size_t n = ts.size();
    std::vector<int64_t> D(n + 1, 0);
    std::deque<std::pair<size_t, int64_t>> cand;  // (i, D[i-1] - i + 1)
    size_t ell = 1;                               // first index with t >= t_j - delta
    for (size_t j = 1; j <= n; ++j) {
        if (j >= K) {
            const size_t i = j - K + 1;
            const int64_t v = D[i - 1] - static_cast<int64_t>(i) + 1;
            while (!cand.empty() && cand.back().second <= v) cand.pop_back();
            cand.emplace_back(i, v);
        }
        while (ts[ell - 1] < ts[j - 1] - delta) ++ell;
        while (!cand.empty() && cand.front().first < ell) cand.pop_front();
        D[j] = D[j - 1];
        if (!cand.empty()) D[j] = std::max(D[j], cand.front().second + static_cast<int64_t>(j));
    }
    return static_cast<uint64_t>(D[n]);
}

}  // namespace

extern "C" int rc_opportunity(const int64_t *t_ns, const uint32_t *route, uint64_t n, uint32_t n_routes, uint32_t K,
                              int64_t delta_ns, int64_t origin_ns, rc_opportunity_counts *out) {
    if (!out || K == 0 || delta_ns <= 0 || n_routes == 0 || (n > 0 && (!t_ns || !route))) return RC_E_INVAL;
    for (uint64_t e = 0; e < n; ++e)
        if (route[e] >= n_routes) return RC_E_INVAL;
    // events grouped by route, each route in ascending time
    std::vector<uint64_t> order(n);
    std::iota(order.begin(), order.end(), uint64_t{0});
    std::stable_sort(order.begin(), order.end(), [&](uint64_t a, uint64_t b) {
        return route[a] != route[b] ? route[a] < route[b] : t_ns[a] < t_ns[b];
    });
    rc_opportunity_counts c{};
    c.n = n;
    std::vector<int64_t> ts;
    size_t a = 0;
    while (a < n) {
        size_t b = a;
        ts.clear();
        while (b < n && route[order[b]] == route[order[a]]) ts.push_back(t_ns[order[b++]]);
        c.fixed += fixed_count(ts, K, delta_ns, origin_ns);
        c.exact += exact_count(ts, K, delta_ns);
        c.upper += upper_count(ts, K, delta_ns);
        a = b;
    }
    *out = c;
    return RC_OK;
}
