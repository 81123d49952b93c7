// rc_grid.cu -- the opportunity grid on the GPU (rc_opportunity_grid in
// include/rc.h): F (Eq. 2), P* (Eq. 6 by the deque recurrence of Algorithm
// 1) and U (Eqs. 3-4) of one event set for every (deadline, threshold) pair
// of a grid: one GPU thread per (route, deadline) for F and U at every
// threshold, one per (route, deadline, threshold) for P*.  The host only
// groups the events by route, each route in time order.
#include <cuda_runtime.h>
#include <stdint.h>

#include <algorithm>
#include <numeric>
#include <vector>

#include "rc.h"

namespace {

__device__ __forceinline__ int64_t floor_div_d(int64_t a, int64_t b) {
    const int64_t q = a / b;
    return (a % b != 0 && ((a < 0) != (b < 0))) ? q - 1 : q;
}

constexpr uint32_t kMaxK = 32;  // thresholds per call

// F and U of one route (times ts[0, n), ascending) at one delta, for every
// threshold at once (neither the windows nor the counts W depend on K).
__global__ void k_opportunity_fu(const int64_t *ts_all, const uint64_t *route_off, uint32_t n_routes,
                                 const uint32_t *Ks, uint32_t nK, const int64_t *deltas, uint32_t nD,
                                 int64_t origin, unsigned long long *out) {
    const uint64_t job = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (job >= static_cast<uint64_t>(n_routes) * nD) return;
    const uint32_t r = static_cast<uint32_t>(job / nD), di = static_cast<uint32_t>(job % nD);
    const uint64_t a0 = route_off[r], n = route_off[r + 1] - a0;
    if (n == 0) return;
    const int64_t *ts = ts_all + a0;
    const int64_t delta = deltas[di];
    uint64_t fixed[kMaxK], upper[kMaxK], nxt[kMaxK];
    for (uint32_t k = 0; k < nK; ++k) {
        fixed[k] = 0;
        upper[k] = 0;
        nxt[k] = n;
    }
    // F (Eq. 2): runs of equal window index along the sorted times (one
    // division per window: the run ends at the first time past its window)
    for (uint64_t i = 0; i < n;) {
        const int64_t w_end = origin + (floor_div_d(ts[i] - origin, delta) + 1) * delta;
        uint64_t j = i + 1;
        while (j < n && ts[j] < w_end) ++j;
        for (uint32_t k = 0; k < nK; ++k)
            if (j - i >= Ks[k]) fixed[k] += j - i;
        i = j;
    }
    // U (Eqs. 3-4), right to left: W_j = #{k : t_j - delta <= t_k <= t_j};
    // nxt[k] = smallest index >= j with W >= K_k; a tie group [f, g) counts
    // for K_k when nxt[k] (taken at f) lies before the first index with
    // t > t_f + delta
    uint64_t p_up = n, p_lo = n, p_end = n, group = 0;
    for (uint64_t jj = n; jj-- > 0;) {
        while (p_up > 0 && ts[p_up - 1] > ts[jj]) --p_up;
        while (p_lo > 0 && ts[p_lo - 1] >= ts[jj] - delta) --p_lo;
        const uint64_t W = p_up - p_lo;
        for (uint32_t k = 0; k < nK; ++k)
            if (W >= Ks[k]) nxt[k] = jj;
        while (p_end > 0 && ts[p_end - 1] > ts[jj] + delta) --p_end;
        ++group;
        if (jj == 0 || ts[jj - 1] < ts[jj]) {
            for (uint32_t k = 0; k < nK; ++k)
                if (nxt[k] < p_end) upper[k] += group;
            group = 0;
        }
    }
    for (uint32_t k = 0; k < nK; ++k) {
        unsigned long long *o = out + (static_cast<uint64_t>(di) * nK + k) * 3;
        atomicAdd(o + 0, static_cast<unsigned long long>(fixed[k]));
        atomicAdd(o + 2, static_cast<unsigned long long>(upper[k]));
    }
}

// P* (Eq. 6, Algorithm 1) of one route at one (delta, K), 1-based j:
// candidates i <= j - K + 1 with value D[i-1] - i + 1 in a deque of
// decreasing values; the head leaves once t_i < t_j - delta; D[j] =
// max(D[j-1], head value + j).  scratch: 2 n int32 words of this job (deque
// indices and values); ring: K + 1 int64 words (the last D values).
__global__ void k_opportunity_p(const int64_t *ts_all, const uint64_t *route_off, uint32_t n_routes,
                                const uint32_t *Ks, uint32_t nK, const int64_t *deltas, uint32_t nD, uint32_t Kmax,
                                int32_t *scratch, int64_t *rings, unsigned long long *out) {
    const uint64_t job = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    const uint64_t J = static_cast<uint64_t>(nD) * nK;
    if (job >= static_cast<uint64_t>(n_routes) * J) return;
    const uint32_t r = static_cast<uint32_t>(job / J);
    const uint32_t di = static_cast<uint32_t>((job % J) / nK), ki = static_cast<uint32_t>(job % nK);
    const uint64_t a0 = route_off[r], n = route_off[r + 1] - a0;
    if (n == 0) return;
    const int64_t *ts = ts_all + a0;
    const int64_t delta = deltas[di];
    const uint32_t K = Ks[ki];
    int32_t *dq_i = scratch + (a0 * J + static_cast<uint64_t>(di * nK + ki) * n) * 2;
    int32_t *dq_v = dq_i + n;
    int64_t *ring = rings + job * (static_cast<uint64_t>(Kmax) + 1);
    // the ring holds D[j-K .. j]: slots advance by one per step, wrapping at
    // K + 1 (no division in the loop)
    const uint32_t R = K + 1u;
    ring[0] = 0;
    // slots of D[j-1] and D[j-K] at j = 1: 0 and (1 - K) mod (K + 1) = 2 mod (K + 1)
    uint32_t slot_prev = 0, slot_cand = 2u % R;
    uint64_t head = 0, tail = 0, ell = 1;
    int64_t Dj = 0;
    for (uint64_t j = 1; j <= n; ++j) {
        if (j >= K) {
            const uint64_t i = j - K + 1;
            const int64_t v = ring[slot_cand] - static_cast<int64_t>(i) + 1;
            while (tail > head && dq_v[tail - 1] <= v) --tail;
            dq_i[tail] = static_cast<int32_t>(i);
            dq_v[tail] = static_cast<int32_t>(v);
            ++tail;
        }
        while (ts[ell - 1] < ts[j - 1] - delta) ++ell;
        while (tail > head && static_cast<uint64_t>(dq_i[head]) < ell) ++head;
        Dj = ring[slot_prev];
        if (tail > head) Dj = max(Dj, static_cast<int64_t>(dq_v[head]) + static_cast<int64_t>(j));
        slot_prev = slot_prev + 1u == R ? 0u : slot_prev + 1u;  // slot of D[j]
        ring[slot_prev] = Dj;
        slot_cand = slot_cand + 1u == R ? 0u : slot_cand + 1u;
    }
    atomicAdd(out + (static_cast<uint64_t>(di) * nK + ki) * 3 + 1, static_cast<unsigned long long>(Dj));
}

}  // namespace

extern "C" int rc_opportunity_grid(const int64_t *t_ns, const uint32_t *route, uint64_t n, uint32_t n_routes,
                                   const uint32_t *K_list, uint32_t n_K, const int64_t *delta_list, uint32_t n_delta,
                                   int64_t origin_ns, uint64_t *counts_out, void *cuda_stream) {
    if (!counts_out || !K_list || !delta_list || n_K == 0 || n_delta == 0 || n_routes == 0 ||
        (n > 0 && (!t_ns || !route)))
        return RC_E_INVAL;
    if (n >= (1ull << 31) || n_K > kMaxK) return RC_E_INVAL;  // deque words are 32-bit
    uint32_t Kmax = 0;
    for (uint32_t k = 0; k < n_K; ++k) {
        if (K_list[k] == 0) return RC_E_INVAL;
        Kmax = std::max(Kmax, K_list[k]);
    }
    for (uint32_t d = 0; d < n_delta; ++d)
        if (delta_list[d] <= 0) return RC_E_INVAL;
    for (uint64_t e = 0; e < n; ++e)
        if (route[e] >= n_routes) return RC_E_INVAL;
    std::fill(counts_out, counts_out + 3ull * n_delta * n_K, uint64_t{0});
    if (n == 0) return RC_OK;
    // group by route, each route in ascending time: a stable counting pass
    // when the events come in time order (the usual case), a sort otherwise
    std::vector<int64_t> ts(n);
    std::vector<uint64_t> off(n_routes + 1, 0);
    for (uint64_t e = 0; e < n; ++e) ++off[route[e] + 1];
    for (uint32_t r = 0; r < n_routes; ++r) off[r + 1] += off[r];
    bool sorted = true;
    for (uint64_t e = 1; e < n && sorted; ++e) sorted = t_ns[e - 1] <= t_ns[e];
    if (sorted) {
        std::vector<uint64_t> fill(off.begin(), off.end() - 1);
        for (uint64_t e = 0; e < n; ++e) ts[fill[route[e]]++] = t_ns[e];
    } else {
        std::vector<uint64_t> order(n);
        std::iota(order.begin(), order.end(), uint64_t{0});
        std::stable_sort(order.begin(), order.end(), [&](uint64_t x, uint64_t y) {
            return route[x] != route[y] ? route[x] < route[y] : t_ns[x] < t_ns[y];
        });
        for (uint64_t e = 0; e < n; ++e) ts[e] = t_ns[order[e]];
    }
    const uint64_t J = static_cast<uint64_t>(n_delta) * n_K;
    const uint64_t jobs = static_cast<uint64_t>(n_routes) * J;
    cudaStream_t s = static_cast<cudaStream_t>(cuda_stream);
    int64_t *d_ts = nullptr, *d_del = nullptr, *d_ring = nullptr;
    uint64_t *d_off = nullptr;
    uint32_t *d_K = nullptr;
    int32_t *d_scr = nullptr;
    unsigned long long *d_out = nullptr;
    int rc = RC_OK;
    auto alloc = [&](void **p, size_t bytes) {
        if (rc == RC_OK && cudaMalloc(p, bytes) != cudaSuccess) {
            cudaGetLastError();
            rc = RC_E_NOMEM;
        }
    };
    alloc(reinterpret_cast<void **>(&d_ts), n * 8);
    alloc(reinterpret_cast<void **>(&d_off), (n_routes + 1) * 8ull);
    alloc(reinterpret_cast<void **>(&d_K), n_K * 4ull);
    alloc(reinterpret_cast<void **>(&d_del), n_delta * 8ull);
    alloc(reinterpret_cast<void **>(&d_scr), n * J * 2 * 4);
    alloc(reinterpret_cast<void **>(&d_ring), jobs * (static_cast<uint64_t>(Kmax) + 1) * 8);
    alloc(reinterpret_cast<void **>(&d_out), J * 3 * 8);
    if (rc == RC_OK) {
        if (cudaMemcpyAsync(d_ts, ts.data(), n * 8, cudaMemcpyHostToDevice, s) != cudaSuccess ||
            cudaMemcpyAsync(d_off, off.data(), (n_routes + 1) * 8ull, cudaMemcpyHostToDevice, s) != cudaSuccess ||
            cudaMemcpyAsync(d_K, K_list, n_K * 4ull, cudaMemcpyHostToDevice, s) != cudaSuccess ||
            cudaMemcpyAsync(d_del, delta_list, n_delta * 8ull, cudaMemcpyHostToDevice, s) != cudaSuccess ||
            cudaMemsetAsync(d_out, 0, J * 3 * 8, s) != cudaSuccess)
            rc = RC_E_CUDA;
    }
    if (rc == RC_OK) {
        const unsigned threads = 64;
        const uint64_t fu_jobs = static_cast<uint64_t>(n_routes) * n_delta;
        k_opportunity_fu<<<static_cast<unsigned>((fu_jobs + threads - 1) / threads), threads, 0, s>>>(
            d_ts, d_off, n_routes, d_K, n_K, d_del, n_delta, origin_ns, d_out);
        k_opportunity_p<<<static_cast<unsigned>((jobs + threads - 1) / threads), threads, 0, s>>>(
            d_ts, d_off, n_routes, d_K, n_K, d_del, n_delta, Kmax, d_scr, d_ring, d_out);
        if (cudaGetLastError() != cudaSuccess ||
            cudaMemcpyAsync(counts_out, d_out, J * 3 * 8, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
            cudaStreamSynchronize(s) != cudaSuccess)
            rc = RC_E_CUDA;
    }
    for (void *p : {static_cast<void *>(d_ts), static_cast<void *>(d_off), static_cast<void *>(d_K),
                    static_cast<void *>(d_del), static_cast<void *>(d_scr), static_cast<void *>(d_ring),
                    static_cast<void *>(d_out)})
        if (p) cudaFree(p);
    return rc;
}
