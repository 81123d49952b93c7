// rc_kernels.cu -- sm_103a kernels of the ready-cohort transition path.
//
// One cohort step (Section 2.1 transition unit; Section 7.1 route bodies and
// global binary decision) per member m, one thread per member:
//   16-byte vector loads of the member's event (outcome, payload) and of its
//   session's state record; route key in registers (SplitMix64 finaliser
//   chained over the little-endian payload words); next state from the
//   selected route body's table staged in shared memory; 16-byte vector
//   stores of the record and the effect; odd-key count by warp ballot +
//   popcount, per-CTA sum in shared memory, then one atomic per CTA and a
//   last-CTA ticket (per-step kernel) or a grid barrier word (persistent).
//
// All work is integer; results are bit-identical to the CPU oracle.
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <cstring>
#include <mutex>
#include <type_traits>

#include "rc.h"
#include "rc_internal.h"

namespace rc {
namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;  // golden-ratio increment of SplitMix64
constexpr uint64_t kFinA = 0xBF58476D1CE4E5B9ull;   // finaliser multipliers
constexpr uint64_t kFinB = 0x94D049BB133111EBull;

// z * c mod 2^64 from 32-bit parts: the wide product of the low words, plus
// the two cross products (the high x high term vanishes mod 2^64) in the
// high word.  Written out because the dependent chain is a little shorter
// than the compiler's 64-bit multiply sequence (measured on GB300: 63.5 vs
// 69 cycles a finaliser round with one warp, 79 vs 91 with two warps per SM
// sub-partition); the result is the same.
__device__ __forceinline__ uint64_t mul64c(uint64_t z, uint64_t c) {
    const uint32_t zl = static_cast<uint32_t>(z), zh = static_cast<uint32_t>(z >> 32);
    const uint32_t cl = static_cast<uint32_t>(c), ch = static_cast<uint32_t>(c >> 32);
    uint64_t w;
    asm("mul.wide.u32 %0, %1, %2;" : "=l"(w) : "r"(zl), "r"(cl));
    uint32_t cross;
    asm("mad.lo.u32 %0, %1, %2, %3;" : "=r"(cross) : "r"(zl), "r"(ch), "r"(zh * cl));
    return w + (static_cast<uint64_t>(cross) << 32);
}

__device__ __forceinline__ uint64_t fin64(uint64_t z) {
    z ^= z >> 30;
    z = mul64c(z, kFinA);
    z ^= z >> 27;
    z = mul64c(z, kFinB);
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t pack64(uint32_t lo, uint32_t hi) {
    return (static_cast<uint64_t>(hi) << 32) | lo;
}

template <int R>
__device__ __forceinline__ uint64_t rotl64c(uint64_t v) {
    if constexpr (R % 64 == 0) {
        return v;
    } else {
        return (v << (R % 64)) | (v >> (64 - R % 64));
    }
}

// Route key: (state, outcome) packed low/high and offset by gamma, then one
// finaliser round per 64-bit payload word.  The state is the pre-step state.
template <int P>
__device__ __forceinline__ uint64_t route_key(uint32_t x, uint32_t o, const uint4 (&pw)[P / 16]) {
    uint64_t h = fin64(pack64(x, o) ^ kGamma);
#pragma unroll
    for (int k = 0; k < P / 16; ++k) {
        h = fin64(h ^ pack64(pw[k].x, pw[k].y));
        h = fin64(h ^ pack64(pw[k].z, pw[k].w));
    }
    return h;
}

// Two independent route keys advanced round by round, so that the two
// dependent chains interleave in the instruction stream.
template <int P>
__device__ __forceinline__ void route_key_pair(uint32_t xa, uint32_t oa, const uint4 (&pa)[P / 16], uint32_t xb,
                                               uint32_t ob, const uint4 (&pb)[P / 16], uint64_t &ra, uint64_t &rb) {
    uint64_t ha = fin64(pack64(xa, oa) ^ kGamma);
    uint64_t hb = fin64(pack64(xb, ob) ^ kGamma);
#pragma unroll
    for (int k = 0; k < P / 16; ++k) {
        ha = fin64(ha ^ pack64(pa[k].x, pa[k].y));
        hb = fin64(hb ^ pack64(pb[k].x, pb[k].y));
        ha = fin64(ha ^ pack64(pa[k].z, pa[k].w));
        hb = fin64(hb ^ pack64(pb[k].z, pb[k].w));
    }
    ra = ha;
    rb = hb;
}

// 64-bit word j (1..) of a record held as 16-byte vectors.
template <int W, int NV>
__device__ __forceinline__ uint64_t rec_word(const uint4 (&r)[NV]) {
    return (W & 1) ? pack64(r[W / 2].z, r[W / 2].w) : pack64(r[W / 2].x, r[W / 2].y);
}
template <int W, int NV>
__device__ __forceinline__ void rec_set_word(uint4 (&r)[NV], uint64_t v) {
    if (W & 1) {
        r[W / 2].z = static_cast<uint32_t>(v);
        r[W / 2].w = static_cast<uint32_t>(v >> 32);
    } else {
        r[W / 2].x = static_cast<uint32_t>(v);
        r[W / 2].y = static_cast<uint32_t>(v >> 32);
    }
}

template <int J, int NV>
__device__ __forceinline__ void mix_acc_word(uint4 (&r)[NV], uint64_t rk) {
    rec_set_word<1 + J, NV>(r, mul64c(rec_word<1 + J, NV>(r) ^ rotl64c<8 * J>(rk), kGamma));
}

// acc update: one word for the 16-byte record, seven rotated words for 64.
template <int SB>
__device__ __forceinline__ void mix_acc(uint4 (&r)[SB / 16], uint64_t rk) {
    constexpr int NV = SB / 16;
    mix_acc_word<0, NV>(r, rk);
    if constexpr (SB == 64) {
        mix_acc_word<1, NV>(r, rk);
        mix_acc_word<2, NV>(r, rk);
        mix_acc_word<3, NV>(r, rk);
        mix_acc_word<4, NV>(r, rk);
        mix_acc_word<5, NV>(r, rk);
        mix_acc_word<6, NV>(r, rk);
    }
}

__device__ __forceinline__ void latch_error(DevBlock *dev, uint32_t code, uint32_t step, uint32_t member) {
    if (atomicCAS(&dev->err, 0u, code) == 0u) {
        dev->err_step = step + dev->step_base;
        dev->err_member = member;
    }
}

__device__ __forceinline__ uint32_t ld_volatile_u32(const uint32_t *p) {
    return *reinterpret_cast<const volatile uint32_t *>(p);
}

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long *p) {
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void red_release_add_u64(unsigned long long *p, unsigned long long v) {
    asm volatile("red.release.gpu.global.add.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// ---- shared-memory barriers and bulk / tensor copies (sm_90+ PTX) ----------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count) : "memory");
}

// One arrival that also announces `bytes` of asynchronous copies.
__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_addr(bar)), "r"(parity)
        : "memory");
    return done != 0u;
}

// Spin-wait clock: the first call stamps t0, later calls report whether
// limit_ns has passed since then (the clock is not read on the fast path).
__device__ __forceinline__ bool timed_out(uint64_t &t0, uint64_t limit_ns) {
    const uint64_t now = globaltimer_ns();
    if (t0 == 0) {
        t0 = now;
        return false;
    }
    return now - t0 > limit_ns;
}

// Bounded wait for an mbarrier phase.  The clock is read only once the phase
// is found incomplete, so a phase that has already completed costs one
// try_wait.  False when limit_ns ran out.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity, uint64_t limit_ns) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    uint32_t spins = 0;
    while (!mbar_try_wait(bar, parity)) {
        if ((++spins & 255u) == 0u && globaltimer_ns() - t0 > limit_ns) return false;
    }
    return true;
}

// L2 eviction-priority policies (applied to whole accesses).
__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t policy_evict_last() {
    uint64_t p;
    asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}

__device__ __forceinline__ void tma_load_2d_hint(void *dst, const CUtensorMap *map, int32_t x, int32_t y,
                                                 uint64_t *bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(smem_addr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

__device__ __forceinline__ void bulk_load_hint(void *dst, const void *src, uint32_t bytes, uint64_t *bar,
                                               uint64_t policy) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], %4;" ::
            "r"(smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar)), "l"(policy)
        : "memory");
}

// 16-byte global load / store at L2 (L1 bypassed) with an L2 eviction policy.
__device__ __forceinline__ uint4 ld_cg_hint(const uint4 *p, uint64_t policy) {
    uint4 v;
    asm volatile("ld.global.cg.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p), "l"(policy)
                 : "memory");
    return v;
}
__device__ __forceinline__ void st_hint(uint4 *p, uint4 v, uint64_t policy) {
    asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(p), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w), "l"(policy)
                 : "memory");
}

// Orders this thread's earlier generic-proxy shared accesses before later
// async-proxy (TMA) accesses of the same shared memory.
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// Makes mbarrier initialisation visible to the async proxy.
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// ---- per-thread asynchronous copies global -> shared (LDGSTS) ----------------
__device__ __forceinline__ void cp_async4(void *dst, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async16(void *dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_addr(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// Position of 16-byte chunk k of member m's payload in a per-member shared
// ring: an XOR of the chunk index with bits of m so that the eight lanes of a
// shared-memory phase hit eight different 16-byte bank groups.
template <int P>
__device__ __forceinline__ uint32_t pay_chunk(uint32_t m, uint32_t k) {
    constexpr uint32_t nc = P / 16;                          // 2, 4 or 8 chunks
    constexpr uint32_t shift = nc == 8 ? 0u : (nc == 4 ? 1u : 2u);
    return m * nc + (k ^ ((m >> shift) & (nc - 1u)));
}

// Copies both route bodies' tables into shared memory (16-byte vectors).
__device__ __forceinline__ void stage_tables(uint8_t *smem, const uint8_t *tables, uint32_t tab_stride,
                                             uint32_t n_bodies, uint32_t first_body) {
    const uint32_t nvec = tab_stride / 16 * n_bodies;
    const uint4 *src = reinterpret_cast<const uint4 *>(tables + static_cast<size_t>(first_body) * tab_stride);
    uint4 *dst = reinterpret_cast<uint4 *>(smem);
    for (uint32_t i = threadIdx.x; i < nvec; i += blockDim.x) dst[i] = __ldg(src + i);
}

// The event of member m of cohort `set`.
template <int P>
struct Event {
    uint32_t s;
    uint32_t o;
    uint4 pw[P / 16];
};

template <int P>
__device__ __forceinline__ void load_event(Event<P> &ev, const StepArgs &a, uint32_t set, uint32_t m) {
    const size_t e = static_cast<size_t>(set) * a.K + m;
    ev.s = a.idx ? __ldg(a.idx + e) : m;
    ev.o = __ldg(a.outcome + e);
    const uint4 *p = reinterpret_cast<const uint4 *>(a.payload + e * P);
#pragma unroll
    for (int k = 0; k < P / 16; ++k) ev.pw[k] = __ldg(p + k);
}

// One member's transition.  Returns 1 for an odd route key, 0 for an even key
// or a rejected member (error latched, nothing written).  `cg_state` reads the
// state record at L2 (bypassing L1), as needed when other CTAs of a persistent
// grid wrote it after this SM last cached it.
template <int SB, int P, bool CG_STATE, bool HINT = false>
__device__ __forceinline__ uint32_t transition(const StepArgs &a, const Event<P> &ev, const uint8_t *tab,
                                               uint32_t sel, uint32_t n, uint32_t m, uint64_t keep = 0) {
    constexpr int NV = SB / 16;
    if (ev.s >= a.n_sessions) {
        latch_error(a.dev, DEV_E_INDEX, n, m);
        return 0u;
    }
    uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(ev.s) * SB);
    uint4 r[NV];
#pragma unroll
    for (int k = 0; k < NV; ++k) {
        if constexpr (HINT)
            r[k] = ld_cg_hint(rp + k, keep);
        else
            r[k] = CG_STATE ? __ldcg(rp + k) : rp[k];
    }
    const uint32_t x = r[0].x;
    if (x >= a.S || ev.o >= 8u) {
        latch_error(a.dev, DEV_E_STATE, n, m);
        return 0u;
    }
    const uint64_t rk = route_key<P>(x, ev.o, ev.pw);
    const uint32_t y = tab[x * 8u + ev.o];
    r[0].x = y;
    r[0].y = r[0].y + 1u;
    mix_acc<SB>(r, rk);
#pragma unroll
    for (int k = 0; k < NV; ++k) {
        if constexpr (HINT)
            st_hint(rp + k, r[k], keep);
        else
            rp[k] = r[k];
    }
    const size_t slot = static_cast<size_t>(n) * a.K + m;
    if (a.effects) {
        uint4 e;
        e.x = static_cast<uint32_t>(rk);
        e.y = static_cast<uint32_t>(rk >> 32);
        e.z = ev.s;
        e.w = y | (ev.o << 16) | (sel << 24);
        __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
    }
    if (a.state_log) {
        uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
    }
    return static_cast<uint32_t>(rk & 1u);
}

// ---------------------------------------------------------------------------
// Per-step kernel: one launch = one cohort step (rc_cohort_step, the host
// round trip, the graph mechanisms).
// ---------------------------------------------------------------------------
template <int SB, int P, bool DECIDE>
__global__ void __launch_bounds__(kStepThreads) k_step(StepArgs a, int step_arg, int sel_arg, uint32_t epi) {
    __shared__ __align__(16) uint8_t tab[256 * 8];
    __shared__ uint32_t warp_odd[kStepThreads / 32];
    __shared__ uint32_t s_step, s_sel;
    const uint32_t tid = threadIdx.x;
    if (tid == 0) {
        s_step = step_arg >= 0 ? static_cast<uint32_t>(step_arg) : ld_volatile_u32(&a.dev->step);
        s_sel = sel_arg >= 0 ? static_cast<uint32_t>(sel_arg) : (ld_volatile_u32(&a.dev->sel) & 1u);
    }
    __syncthreads();
    const uint32_t n = s_step;
    const uint32_t sel = s_sel;
    stage_tables(tab, a.tables, a.tab_stride, 1, sel);
    __syncthreads();

    const uint32_t m = blockIdx.x * blockDim.x + tid;
    uint32_t odd = 0;
    if (m < a.K) {
        Event<P> ev;
        load_event<P>(ev, a, n % a.n_sets, m);
        odd = transition<SB, P, false>(a, ev, tab, sel, n, m);
    }
    if constexpr (!DECIDE) return;

    const uint32_t ball = __ballot_sync(0xffffffffu, odd);
    if ((tid & 31u) == 0) warp_odd[tid >> 5] = __popc(ball);
    __syncthreads();
    if (tid != 0) return;
    uint32_t c = 0;
    for (uint32_t w = 0; w < (blockDim.x + 31u) / 32u; ++w) c += warp_odd[w];
    uint32_t total = c;
    if (gridDim.x > 1) {
        atomicAdd(&a.dev->count, c);
        __threadfence();
        const uint32_t ticket = atomicAdd(&a.dev->ticket, 1u);
        if (ticket != gridDim.x - 1) return;
        __threadfence();
        total = atomicExch(&a.dev->count, 0u);
        atomicExch(&a.dev->ticket, 0u);
    }
    const uint32_t d = total > a.K / 2u ? 1u : 0u;
    a.dev->sel = d;
    if (a.decisions) a.decisions[n] = d;
    a.dev->step = n + 1u;
    if (epi & EPI_SET_WHILE) cudaGraphSetConditional(a.h_while, (n + 1u < a.n_steps) ? 1u : 0u);
}

// ---------------------------------------------------------------------------
// Persistent chain, one CTA (K <= 512): all n_steps in one launch.  The
// decision is reduced in shared memory and read from a register: it never
// leaves the SM.  Events are fetched two steps ahead.
// ---------------------------------------------------------------------------
template <int SB, int P>
__global__ void __launch_bounds__(512) k_chain_cta(StepArgs a) {
    __shared__ __align__(16) uint8_t tab[2 * 256 * 8];
    __shared__ uint32_t warp_odd[2][32];
    const uint32_t tid = threadIdx.x;
    const uint32_t nw = (blockDim.x + 31u) / 32u;
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    uint32_t sel = ld_volatile_u32(&a.dev->sel) & 1u;
    __syncthreads();
    const bool active = tid < a.K;
    // events travel two steps ahead of their use, so a step's session index
    // is already in a register when the step starts its record gather
    Event<P> ev0, ev1;
    if (active && a.n_steps > 0) load_event<P>(ev0, a, 0, tid);
    if (active && a.n_steps > 1) load_event<P>(ev1, a, 1 % a.n_sets, tid);
    for (uint32_t n = 0; n < a.n_steps; ++n) {
        uint32_t odd = 0;
        if (active) {
            const Event<P> ev = ev0;
            ev0 = ev1;
            if (n + 2u < a.n_steps) load_event<P>(ev1, a, (n + 2u) % a.n_sets, tid);
            odd = transition<SB, P, false>(a, ev, tab + sel * a.tab_stride, sel, n, tid);
        }
        const uint32_t ball = __ballot_sync(0xffffffffu, odd);
        if ((tid & 31u) == 0) warp_odd[n & 1u][tid >> 5] = __popc(ball);
        __syncthreads();  // also orders this step's state stores before the next step's loads
        uint32_t total = 0;
        for (uint32_t w = 0; w < nw; ++w) total += warp_odd[n & 1u][w];
        sel = total > a.K / 2u ? 1u : 0u;
        if (tid == 0 && a.decisions) a.decisions[n] = sel;
    }
    if (tid == 0) {
        if (a.n_steps > 0) a.dev->sel = sel;
        a.dev->step = a.n_steps;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, one CTA, member m is session m (no index array): each
// thread keeps its session's record in registers for the whole chain and
// writes it back once at the end (and to the state log per step when asked).
// Outcomes and payloads stream through a D-deep ring of per-thread
// asynchronous copies.
// ---------------------------------------------------------------------------
template <int SB, int P, int D>
__global__ void __launch_bounds__(1024, 1) k_chain_cta_ident(StepArgs a) {
    constexpr uint32_t RD = D + 1;
    constexpr uint32_t NC = P / 16;
    constexpr int NV = SB / 16;
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ uint32_t warp_odd[2][32];
    const uint32_t K = a.K;
    const uint32_t Kp = (K + 3u) & ~3u;
    const uint32_t tid = threadIdx.x;
    const uint32_t nw = (blockDim.x + 31u) / 32u;
    uint8_t *tab = dsm;
    uint32_t *out_r = reinterpret_cast<uint32_t *>(dsm + 2 * a.tab_stride);
    uint4 *pay_r = reinterpret_cast<uint4 *>(out_r + RD * Kp);
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    uint32_t sel = ld_volatile_u32(&a.dev->sel) & 1u;
    const bool act = tid < K;
    const uint32_t m = tid;
    const uint32_t nst = a.n_steps;
    const bool in_range = m < a.n_sessions;
    uint4 r[NV];
    if (act && in_range) {
        const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(m) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) r[k] = rp[k];
    }
    auto issue_data = [&](uint32_t j) {
        if (!act || j >= nst) return;
        const size_t e = static_cast<size_t>(j % a.n_sets) * K + m;
        cp_async4(&out_r[(j % RD) * Kp + m], a.outcome + e);
        const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + e * P);
        uint4 *ring = pay_r + (j % RD) * Kp * NC;
#pragma unroll
        for (uint32_t k = 0; k < NC; ++k) cp_async16(ring + pay_chunk<P>(m, k), src + k);
    };
    for (uint32_t j = 0; j < D; ++j) {
        issue_data(j);
        cp_async_commit();
    }
    __syncthreads();
    for (uint32_t n = 0; n < nst; ++n) {
        cp_async_wait<D - 1>();
        uint32_t odd = 0;
        if (act) {
            const uint32_t o = out_r[(n % RD) * Kp + m];
            if (!in_range) {
                latch_error(a.dev, DEV_E_INDEX, n, m);
            } else if (r[0].x >= a.S || o >= 8u) {
                latch_error(a.dev, DEV_E_STATE, n, m);
            } else {
                uint4 pw[NC];
                const uint4 *ring = pay_r + (n % RD) * Kp * NC;
#pragma unroll
                for (uint32_t k = 0; k < NC; ++k) pw[k] = ring[pay_chunk<P>(m, k)];
                const uint32_t x = r[0].x;
                const uint64_t rk = route_key<P>(x, o, pw);
                const uint32_t y = tab[sel * a.tab_stride + x * 8u + o];
                r[0].x = y;
                r[0].y = r[0].y + 1u;
                mix_acc<SB>(r, rk);
                const size_t slot = static_cast<size_t>(n) * K + m;
                if (a.effects) {
                    uint4 e;
                    e.x = static_cast<uint32_t>(rk);
                    e.y = static_cast<uint32_t>(rk >> 32);
                    e.z = m;
                    e.w = y | (o << 16) | (sel << 24);
                    __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
                }
                if (a.state_log) {
                    uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
                    for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
                }
                odd = static_cast<uint32_t>(rk & 1u);
            }
        }
        issue_data(n + D);
        cp_async_commit();
        const uint32_t ball = __ballot_sync(0xffffffffu, odd);
        if ((tid & 31u) == 0) warp_odd[n & 1u][tid >> 5] = __popc(ball);
        __syncthreads();
        uint32_t total = 0;
        for (uint32_t w = 0; w < nw; ++w) total += warp_odd[n & 1u][w];
        sel = total > K / 2u ? 1u : 0u;
        if (tid == 0 && a.decisions) a.decisions[n] = sel;
    }
    cp_async_wait<0>();
    if (act && in_range) {
        uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(m) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) rp[k] = r[k];
    }
    if (tid == 0) {
        if (nst > 0) a.dev->sel = sel;
        a.dev->step = nst;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, one CTA, member m = session m (K <= 512), two steps per
// block barrier.  Thread m holds its session's record in registers for the
// whole chain.  The key of step j reads the state the session left in step
// j - 1, T_sel(j-1)[x][o] with sel(j-1) = d(j-2); so once d(2r-1) is known the
// keys of steps 2r and 2r+1 are two independent hash chains of one thread,
// and one block barrier counts both (the two counts packed in one word per
// warp).  The record update of step 2r+1 needs d(2r) and is applied at the
// start of the next region.  Outcomes and payload rows come through a ring of
// per-thread asynchronous copies D steps deep (two steps consumed per region,
// D + 2 slots).
// ---------------------------------------------------------------------------
template <int SB, int P, int D>
__global__ void __launch_bounds__(512, 1) k_chain_cta_ident2(StepArgs a) {
    static_assert(D >= 2, "two steps per region");
    constexpr uint32_t RD = D + 2;
    constexpr uint32_t NC = P / 16;
    constexpr int NV = SB / 16;
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ uint32_t warp_odd[2][16];
    const uint32_t K = a.K;
    const uint32_t Kp = (K + 3u) & ~3u;
    const uint32_t tid = threadIdx.x;
    const uint32_t nw = (blockDim.x + 31u) / 32u;
    uint8_t *tab = dsm;
    uint32_t *out_r = reinterpret_cast<uint32_t *>(dsm + 2 * a.tab_stride);
    uint4 *pay_r = reinterpret_cast<uint4 *>(out_r + RD * Kp);
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    const bool act = tid < K;
    const uint32_t m = tid;
    const uint32_t nst = a.n_steps;
    const bool in_range = m < a.n_sessions;
    uint4 r[NV];
#pragma unroll
    for (int k = 0; k < NV; ++k) r[k] = make_uint4(0, 0, 0, 0);
    if (act && in_range) {
        const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(m) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) r[k] = rp[k];
    }
    // event set of the next copy: advanced one step per call instead of a
    // modulo (the copies go out in step order)
    uint32_t next_set = 0;
    auto issue_data = [&](uint32_t j) {
        const uint32_t set = next_set;
        next_set = next_set + 1u == a.n_sets ? 0u : next_set + 1u;
        if (act && j < nst) {
            const size_t e = static_cast<size_t>(set) * K + m;
            cp_async4(&out_r[(j % RD) * Kp + m], a.outcome + e);
            const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + e * P);
            uint4 *ring = pay_r + (j % RD) * Kp * NC;
#pragma unroll
            for (uint32_t k = 0; k < NC; ++k) cp_async16(ring + pay_chunk<P>(m, k), src + k);
        }
        cp_async_commit();
    };
    // this thread's record update for step n under decision sel (a valid member)
    auto apply = [&](uint32_t n, uint32_t sel, uint32_t o, uint64_t rk) {
        const uint32_t x = r[0].x;
        const uint32_t y = tab[sel * a.tab_stride + x * 8u + o];
        r[0].x = y;
        r[0].y = r[0].y + 1u;
        mix_acc<SB>(r, rk);
        const size_t slot = static_cast<size_t>(n) * K + m;
        if (a.effects) {
            uint4 e;
            e.x = static_cast<uint32_t>(rk);
            e.y = static_cast<uint32_t>(rk >> 32);
            e.z = m;
            e.w = y | (o << 16) | (sel << 24);
            __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
        }
        if (a.state_log) {
            uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
            for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
        }
    };
    for (uint32_t j = 0; j < D; ++j) issue_data(j);
    __syncthreads();
    uint32_t sel_a = ld_volatile_u32(&a.dev->sel) & 1u;  // decision for step 2r: d(2r-1)
    uint32_t sel_b = 0;                                  // decision for step 2r-1: d(2r-2)
    bool pend = false;                                   // step 2r-1 keyed, record update pending
    uint32_t pend_o = 0;
    uint64_t pend_rk = 0;
    uint32_t last = sel_a;  // the decision of the last step decided
    for (uint32_t ja = 0; ja < nst; ja += 2u) {
        const uint32_t jb = ja + 1u;
        const bool has_b = jb < nst;
        cp_async_wait<D - 2>();  // this thread's data of steps ja and jb
        // the copies of steps ja + D and ja + D + 1 (into the slots of steps
        // ja - 2 and ja - 1, read last region) go out first
        issue_data(ja + D);
        issue_data(ja + D + 1u);
        if (pend) apply(ja - 1u, sel_b, pend_o, pend_rk);
        pend = false;
        uint32_t odd_a = 0, odd_b = 0;
        if (act) {
            const uint32_t o_a = out_r[(ja % RD) * Kp + m];
            const uint32_t o_b = has_b ? out_r[(jb % RD) * Kp + m] : 0u;
            if (!in_range) {
                latch_error(a.dev, DEV_E_INDEX, ja, m);
                if (has_b) latch_error(a.dev, DEV_E_INDEX, jb, m);
            } else {
                const uint32_t x_a = r[0].x;
                const bool ok_a = x_a < a.S && o_a < 8u;
                if (!ok_a) latch_error(a.dev, DEV_E_STATE, ja, m);
                const uint32_t x_b = ok_a ? static_cast<uint32_t>(tab[sel_a * a.tab_stride + x_a * 8u + o_a]) : x_a;
                const bool ok_b = has_b && x_b < a.S && o_b < 8u;
                if (has_b && !ok_b) latch_error(a.dev, DEV_E_STATE, jb, m);
                uint4 pa[NC], pb[NC];
                const uint4 *ra = pay_r + (ja % RD) * Kp * NC;
                const uint4 *rb = pay_r + (jb % RD) * Kp * NC;
#pragma unroll
                for (uint32_t k = 0; k < NC; ++k) {
                    pa[k] = ra[pay_chunk<P>(m, k)];
                    pb[k] = ok_b ? rb[pay_chunk<P>(m, k)] : make_uint4(0, 0, 0, 0);
                }
                // two independent key chains (the second on a valid dummy when unused)
                uint64_t rk_a, rk_b;
                route_key_pair<P>(ok_a ? x_a : 0u, ok_a ? o_a : 0u, pa, ok_b ? x_b : 0u, ok_b ? o_b : 0u, pb, rk_a,
                                  rk_b);
                if (ok_a) {
                    apply(ja, sel_a, o_a, rk_a);
                    odd_a = static_cast<uint32_t>(rk_a & 1u);
                }
                if (ok_b) {
                    pend = true;
                    pend_o = o_b;
                    pend_rk = rk_b;
                    odd_b = static_cast<uint32_t>(rk_b & 1u);
                }
            }
        }
        const uint32_t ca = __popc(__ballot_sync(0xffffffffu, odd_a != 0u));
        const uint32_t cb = __popc(__ballot_sync(0xffffffffu, odd_b != 0u));
        const uint32_t rr = (ja >> 1) & 1u;
        if ((tid & 31u) == 0) warp_odd[rr][tid >> 5] = ca | (cb << 16);
        __syncthreads();
        uint32_t total = 0;
        for (uint32_t w = 0; w < nw; ++w) total += warp_odd[rr][w];
        const uint32_t da = (total & 0xFFFFu) > K / 2u ? 1u : 0u;
        const uint32_t db = (total >> 16) > K / 2u ? 1u : 0u;
        if (tid == 0 && a.decisions) {
            a.decisions[ja] = da;
            if (has_b) a.decisions[jb] = db;
        }
        sel_b = da;
        sel_a = db;
        last = has_b ? db : da;
    }
    if (pend) apply(nst - 1u, sel_b, pend_o, pend_rk);
    cp_async_wait<0>();
    if (act && in_range) {
        uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(m) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) rp[k] = r[k];
    }
    if (tid == 0) {
        if (nst > 0) a.dev->sel = last;
        a.dev->step = nst;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, one warp, member m = session m (K <= 32): the chain of
// k_chain_cta_ident2 (two steps keyed side by side, the record of step 2r+1
// updated at the next region's start) with the cohort inside one warp, so the
// two counts of a region are the two ballots' popcounts and no block barrier
// is needed; each lane reads only the ring slots its own copies fill.  Trace
// points (lane 0, at step 2r): 0 region start, 1 data landed and copies
// issued, 2 pending record updated, 3 second state ready, 4 keys done,
// 5 record updated, 6 decisions.
// ---------------------------------------------------------------------------
template <int SB, int P, int D>
__global__ void __launch_bounds__(32, 1) k_chain_warp_ident(StepArgs a) {
    static_assert(D >= 2, "two steps per region");
    constexpr uint32_t RD = D + 2;
    constexpr uint32_t NC = P / 16;
    constexpr int NV = SB / 16;
    extern __shared__ __align__(16) uint8_t dsm[];
    const uint32_t K = a.K;
    const uint32_t Kp = (K + 3u) & ~3u;
    const uint32_t tid = threadIdx.x;
    uint8_t *tab = dsm;
    uint32_t *out_r = reinterpret_cast<uint32_t *>(dsm + 2 * a.tab_stride);
    uint4 *pay_r = reinterpret_cast<uint4 *>(out_r + RD * Kp);
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    const bool act = tid < K;
    const uint32_t m = tid;
    const uint32_t nst = a.n_steps;
    const bool in_range = m < a.n_sessions;
    long long *trace = (a.trace && tid == 0) ? a.trace : nullptr;
    uint4 r[NV];
#pragma unroll
    for (int k = 0; k < NV; ++k) r[k] = make_uint4(0, 0, 0, 0);
    if (act && in_range) {
        const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(m) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) r[k] = rp[k];
    }
    // event set of the next copy: advanced one step per call instead of a
    // modulo (the copies go out in step order)
    uint32_t next_set = 0;
    auto issue_data = [&](uint32_t j) {
        const uint32_t set = next_set;
        next_set = next_set + 1u == a.n_sets ? 0u : next_set + 1u;
        if (act && j < nst) {
            const size_t e = static_cast<size_t>(set) * K + m;
            cp_async4(&out_r[(j % RD) * Kp + m], a.outcome + e);
            const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + e * P);
            uint4 *ring = pay_r + (j % RD) * Kp * NC;
#pragma unroll
            for (uint32_t k = 0; k < NC; ++k) cp_async16(ring + pay_chunk<P>(m, k), src + k);
        }
        cp_async_commit();
    };
    // this thread's record update for step n under decision sel (a valid member)
    auto apply = [&](uint32_t n, uint32_t sel, uint32_t o, uint64_t rk) {
        const uint32_t x = r[0].x;
        const uint32_t y = tab[sel * a.tab_stride + x * 8u + o];
        r[0].x = y;
        r[0].y = r[0].y + 1u;
        mix_acc<SB>(r, rk);
        const size_t slot = static_cast<size_t>(n) * K + m;
        if (a.effects) {
            uint4 e;
            e.x = static_cast<uint32_t>(rk);
            e.y = static_cast<uint32_t>(rk >> 32);
            e.z = m;
            e.w = y | (o << 16) | (sel << 24);
            __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
        }
        if (a.state_log) {
            uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
            for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
        }
    };
    for (uint32_t j = 0; j < D; ++j) issue_data(j);
    __syncwarp();  // the tables staged by every lane
    uint32_t sel_a = ld_volatile_u32(&a.dev->sel) & 1u;  // decision for step 2r: d(2r-1)
    uint32_t sel_b = 0;                                  // decision for step 2r-1: d(2r-2)
    bool pend = false;                                   // step 2r-1 keyed, record update pending
    uint32_t pend_o = 0;
    uint64_t pend_rk = 0;
    uint32_t last = sel_a;  // the decision of the last step decided
    for (uint32_t ja = 0; ja < nst; ja += 2u) {
        const uint32_t jb = ja + 1u;
        const bool has_b = jb < nst;
        if (trace) trace[ja * 8 + 0] = clock64();
        cp_async_wait<D - 2>();  // this thread's data of steps ja and jb
        // the copies of steps ja + D and ja + D + 1 (into the slots of steps
        // ja - 2 and ja - 1, read last region) go out first: their issue fills
        // the stalls of the dependent lookups and keys below
        issue_data(ja + D);
        issue_data(ja + D + 1u);
        if (trace) trace[ja * 8 + 1] = clock64();
        if (pend) apply(ja - 1u, sel_b, pend_o, pend_rk);
        pend = false;
        if (trace) {
            asm volatile("" ::"r"(r[0].x));
            trace[ja * 8 + 2] = clock64();
        }
        uint32_t odd_a = 0, odd_b = 0;
        if (act) {
            const uint32_t o_a = out_r[(ja % RD) * Kp + m];
            const uint32_t o_b = has_b ? out_r[(jb % RD) * Kp + m] : 0u;
            if (!in_range) {
                latch_error(a.dev, DEV_E_INDEX, ja, m);
                if (has_b) latch_error(a.dev, DEV_E_INDEX, jb, m);
            } else {
                const uint32_t x_a = r[0].x;
                const bool ok_a = x_a < a.S && o_a < 8u;
                if (!ok_a) latch_error(a.dev, DEV_E_STATE, ja, m);
                const uint32_t x_b = ok_a ? static_cast<uint32_t>(tab[sel_a * a.tab_stride + x_a * 8u + o_a]) : x_a;
                const bool ok_b = has_b && x_b < a.S && o_b < 8u;
                if (has_b && !ok_b) latch_error(a.dev, DEV_E_STATE, jb, m);
                if (trace) {
                    asm volatile("" ::"r"(x_b));
                    trace[ja * 8 + 3] = clock64();
                }
                uint4 pa[NC], pb[NC];
                const uint4 *ra = pay_r + (ja % RD) * Kp * NC;
                const uint4 *rb = pay_r + (jb % RD) * Kp * NC;
#pragma unroll
                for (uint32_t k = 0; k < NC; ++k) {
                    pa[k] = ra[pay_chunk<P>(m, k)];
                    pb[k] = ok_b ? rb[pay_chunk<P>(m, k)] : make_uint4(0, 0, 0, 0);
                }
                // two independent key chains (the second on a valid dummy when unused)
                uint64_t rk_a, rk_b;
                route_key_pair<P>(ok_a ? x_a : 0u, ok_a ? o_a : 0u, pa, ok_b ? x_b : 0u, ok_b ? o_b : 0u, pb, rk_a,
                                  rk_b);
                if (trace) {
                    asm volatile("" ::"l"(rk_a ^ rk_b));
                    trace[ja * 8 + 4] = clock64();
                }
                if (ok_a) {
                    apply(ja, sel_a, o_a, rk_a);
                    odd_a = static_cast<uint32_t>(rk_a & 1u);
                }
                if (ok_b) {
                    pend = true;
                    pend_o = o_b;
                    pend_rk = rk_b;
                    odd_b = static_cast<uint32_t>(rk_b & 1u);
                }
            }
        }
        if (trace) trace[ja * 8 + 5] = clock64();
        // the whole cohort is this warp: the counts are the ballots' own
        const uint32_t ca = __popc(__ballot_sync(0xffffffffu, odd_a != 0u));
        const uint32_t cb = __popc(__ballot_sync(0xffffffffu, odd_b != 0u));
        const uint32_t da = ca > K / 2u ? 1u : 0u;
        const uint32_t db = cb > K / 2u ? 1u : 0u;
        if (trace) {
            asm volatile("" ::"r"(da), "r"(db));
            trace[ja * 8 + 6] = clock64();
        }
        if (tid == 0 && a.decisions) {
            a.decisions[ja] = da;
            if (has_b) a.decisions[jb] = db;
        }
        sel_b = da;
        sel_a = db;
        last = has_b ? db : da;
    }
    if (pend) apply(nst - 1u, sel_b, pend_o, pend_rk);
    cp_async_wait<0>();
    if (act && in_range) {
        uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(m) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) rp[k] = r[k];
    }
    if (tid == 0) {
        if (nst > 0) a.dev->sel = last;
        a.dev->step = nst;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, cooperative grid (any K): each CTA owns a grid-stride
// slice of members.  Per step, after a block barrier, thread 0 of each CTA
// adds (1 << 32 | odd count) to the step's barrier word with release
// semantics and spins with acquire loads until all CTAs have arrived, then a
// block barrier hands the result on: the release is cumulative over the
// block's stores (ordered before it by the first block barrier) and the
// acquire over the block's later loads, so no separate fence is needed.  The
// low half is then the full odd count, so every CTA derives the decision.  Three rotating words:
// CTA 0 clears word (n+1) % 3 before arriving at step n, when no CTA can still
// be reading it.  Spins are bounded by dev->wait_ns; on expiry the CTA latches
// RC_E_TIMEOUT, raises dev->abort and returns, and the others follow.
// ---------------------------------------------------------------------------
template <int SB, int P>
__global__ void __launch_bounds__(kGridThreads) k_chain_grid(StepArgs a) {
    __shared__ __align__(16) uint8_t tab[2 * 256 * 8];
    __shared__ uint32_t warp_odd[kGridThreads / 32];
    __shared__ uint32_t s_sel, s_abort;
    const uint32_t tid = threadIdx.x;
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    if (tid == 0) {
        s_sel = ld_volatile_u32(&a.dev->sel) & 1u;
        s_abort = 0;
    }
    __syncthreads();
    uint32_t sel = s_sel;
    const uint32_t stride = gridDim.x * blockDim.x;
    const uint64_t limit = a.dev->wait_ns;
    for (uint32_t n = 0; n < a.n_steps; ++n) {
        const uint32_t set = n % a.n_sets;
        uint32_t odd = 0;
        for (uint32_t m = blockIdx.x * blockDim.x + tid; m < a.K; m += stride) {
            Event<P> ev;
            load_event<P>(ev, a, set, m);
            odd += transition<SB, P, true>(a, ev, tab + sel * a.tab_stride, sel, n, m);
        }
        // per-CTA odd count (each thread may hold more than one)
        uint32_t v = odd;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if ((tid & 31u) == 0) warp_odd[tid >> 5] = v;
        __syncthreads();
        if (tid == 0) {
            uint32_t c = 0;
            for (uint32_t w = 0; w < blockDim.x / 32u; ++w) c += warp_odd[w];
            unsigned long long *word = &a.dev->slot[n % 3u];
            if (blockIdx.x == 0) {
                a.dev->slot[(n + 1u) % 3u] = 0ull;
            }
            const bool skip = (n == 0 && blockIdx.x == 1 && ld_volatile_u32(&a.dev->skip_arrival) != 0u);
            if (!skip) red_release_add_u64(word, (1ull << 32) | c);
            uint64_t t0 = 0;
            unsigned long long w;
            uint32_t spins = 0;
            for (;;) {
                w = ld_acquire_u64(word);
                if ((w >> 32) >= gridDim.x) break;
                if ((++spins & 63u) == 0u) {
                    if (ld_volatile_u32(&a.dev->abort) != 0u) {
                        s_abort = 1;
                        break;
                    }
                    if (timed_out(t0, limit)) {
                        latch_error(a.dev, DEV_E_TIMEOUT, n, blockIdx.x);
                        atomicExch(&a.dev->abort, 1u);
                        s_abort = 1;
                        break;
                    }
                }
            }
            const uint32_t d = (static_cast<uint32_t>(w & 0xffffffffull) > a.K / 2u) ? 1u : 0u;
            s_sel = d;
            if (blockIdx.x == 0 && a.decisions && !s_abort) a.decisions[n] = d;
        }
        __syncthreads();
        if (s_abort) return;
        sel = s_sel;
    }
    if (blockIdx.x == 0 && tid == 0) {
        if (a.n_steps > 0) a.dev->sel = sel;
        a.dev->step = a.n_steps;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, cooperative grid, TMA-fed (K a multiple of 8; one CTA per
// SM).  CTA b owns the contiguous members [b*chunk, b*chunk + cnt).  Each step
// its events arrive in shared memory ahead of time: the payload rows as
// n_boxes tiles of box_rows x P bytes through a 2-D tensor map whose 32/64/128
// byte swizzle makes the per-member row reads bank-conflict free, the outcome
// and session-index runs as 1-D bulk copies; all complete on one mbarrier per
// stage.  Two stages: the copies for step n + 2 are issued right after the CTA
// arrives at the grid barrier of step n, so they stream while the barrier
// resolves.  The state gather stays after the barrier (records written by
// other CTAs in step n must be visible).  The barrier and the decision are
// those of k_chain_grid.  Every wait is bounded; a CTA that gives up waits
// (bounded) for its own copies in flight before it returns.
// ---------------------------------------------------------------------------
struct TmaShape {
    uint32_t chunk;        // members per CTA (multiple of 8)
    uint32_t box_rows;     // rows per tensor tile (multiple of 8, <= 256)
    uint32_t n_boxes;      // tiles per stage
    uint32_t stage_pay;    // payload bytes per stage (multiple of 1024)
    uint32_t stage_words;  // 32-bit words per outcome / index stage (multiple of 4)
};

template <int P>
__device__ __forceinline__ void read_payload_swizzled(uint4 (&pw)[P / 16], const uint8_t *stage, uint32_t row) {
    // TMA swizzle: 16-byte chunk bits [4..] of the shared address XOR address
    // bits [7..] (3 bits for 128-byte rows, 2 for 64, 1 for 32); stages are
    // 1024-byte aligned, so offsets stand for addresses.
    constexpr uint32_t mask = P == 128 ? 7u : (P == 64 ? 3u : 1u);
#pragma unroll
    for (int k = 0; k < P / 16; ++k) {
        uint32_t off = row * P + static_cast<uint32_t>(k) * 16u;
        off ^= ((off >> 7) & mask) << 4;
        pw[k] = *reinterpret_cast<const uint4 *>(stage + off);
    }
}

// One step of the members [m0, m0 + cnt) of a TMA-fed CTA whose records are
// 64 bytes or more, one member per thread (cnt <= blockDim.x).  The records are
// gathered and stored warp-cooperatively (NV lanes per record, chunks staged in
// shared memory), so a copy instruction of a warp touches 32 / NV records
// rather than one chunk of 32 records.  Same results and error latching as
// transition(); returns this thread's odd-key count.
template <int SB, int P>
__device__ __forceinline__ uint32_t coop_transition(const StepArgs &a, const uint32_t *idx_st, const uint32_t *out_st,
                                                    const uint8_t *pay_st, uint4 *rec_st, uint32_t cnt, uint32_t m0,
                                                    const uint8_t *tab, uint32_t sel, uint32_t n, uint64_t keep) {
    constexpr uint32_t NV = SB / 16;
    constexpr uint32_t RPI = 32u / NV;
    const uint32_t tid = threadIdx.x;
    const uint32_t lane = tid & 31u, wbase = tid & ~31u;
    const uint32_t c = lane % NV;
    auto session_of = [&](uint32_t t) { return a.idx ? idx_st[t] : m0 + t; };
    // gather the warp's records (a copy whose stage slot would leave the
    // block's stage is refused and latched: the stage holds blockDim.x records)
#pragma unroll
    for (uint32_t k = 0; k < NV; ++k) {
        const uint32_t t = wbase + k * RPI + lane / NV;
        if (t < cnt) {
            const uint32_t s = session_of(t);
            const uint32_t slot = pay_chunk<SB>(t, c);
            if (slot >= blockDim.x * NV)
                latch_error(a.dev, DEV_E_INDEX, n, 0xFFFFFF00u | t);
            else if (s < a.n_sessions)
                cp_async16(rec_st + slot, reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s) * SB) + c);
        }
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncwarp();
    uint32_t odd = 0, updated = 0;
    if (tid < cnt) {
        const uint32_t m = m0 + tid;
        const uint32_t s = session_of(tid);
        const uint32_t o = out_st[tid];
        if (s >= a.n_sessions) {
            latch_error(a.dev, DEV_E_INDEX, n, m);
        } else {
            uint4 r[NV];
#pragma unroll
            for (uint32_t k = 0; k < NV; ++k) r[k] = rec_st[pay_chunk<SB>(tid, k)];
            const uint32_t x = r[0].x;
            if (x >= a.S || o >= 8u) {
                latch_error(a.dev, DEV_E_STATE, n, m);
            } else {
                uint4 pw[P / 16];
                read_payload_swizzled<P>(pw, pay_st, tid);
                const uint64_t rk = route_key<P>(x, o, pw);
                const uint32_t y = tab[x * 8u + o];
                r[0].x = y;
                r[0].y = r[0].y + 1u;
                mix_acc<SB>(r, rk);
#pragma unroll
                for (uint32_t k = 0; k < NV; ++k) rec_st[pay_chunk<SB>(tid, k)] = r[k];
                const size_t slot = static_cast<size_t>(n) * a.K + m;
                if (a.effects) {
                    uint4 e;
                    e.x = static_cast<uint32_t>(rk);
                    e.y = static_cast<uint32_t>(rk >> 32);
                    e.z = s;
                    e.w = y | (o << 16) | (sel << 24);
                    __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
                }
                if (a.state_log) {
                    uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
                    for (uint32_t k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
                }
                odd = static_cast<uint32_t>(rk & 1u);
                updated = 1;
            }
        }
    }
    // store the warp's updated records
    const uint32_t upd = __ballot_sync(0xffffffffu, updated);
    __syncwarp();
#pragma unroll
    for (uint32_t k = 0; k < NV; ++k) {
        const uint32_t q = k * RPI + lane / NV;
        const uint32_t t = wbase + q;
        if ((upd >> q) & 1u) {
            const uint32_t s = session_of(t);
            st_hint(reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s) * SB) + c, rec_st[pay_chunk<SB>(t, c)], keep);
        }
    }
    return odd;
}

template <int SB, int P>
__global__ void __launch_bounds__(512, 1)
    k_chain_grid_tma(const __grid_constant__ CUtensorMap tmap, StepArgs a, TmaShape sh) {
    constexpr int NV = SB / 16;
    extern __shared__ uint8_t dsm_raw[];
    __shared__ __align__(8) uint64_t bar[2];
    __shared__ uint32_t warp_odd[16];
    __shared__ uint32_t s_sel, s_abort, s_pending, s_pend_step[2];
    // carve the dynamic shared memory: [pay 0][pay 1][out 0][out 1][idx 0][idx 1][tables]
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    uint32_t *const words = reinterpret_cast<uint32_t *>(base + 2 * sh.stage_pay);
    uint8_t *const tab = reinterpret_cast<uint8_t *>(words + 4 * sh.stage_words);
    // 64-byte records: a shared stage of one record per thread (chunks placed
    // by pay_chunk, so that quarter-warps hit eight bank groups)
    uint4 *const rec_st = reinterpret_cast<uint4 *>(tab + ((2 * a.tab_stride + 15u) & ~15u));
    auto pay_of = [&](uint32_t st) { return base + st * sh.stage_pay; };
    auto out_of = [&](uint32_t st) { return words + st * sh.stage_words; };
    auto idx_of = [&](uint32_t st) { return words + (2u + st) * sh.stage_words; };

    const uint32_t tid = threadIdx.x;
    const uint32_t m0 = blockIdx.x * sh.chunk;
    const uint32_t cnt = m0 < a.K ? min(sh.chunk, a.K - m0) : 0u;
    const uint64_t limit = a.dev->wait_ns;
    // event streams are read once: evict them first; session records are
    // re-read by later steps: keep them
    const uint64_t stream_pol = policy_evict_first();
    const uint64_t keep_pol = policy_evict_last();
    const uint32_t issuer = blockDim.x > 32u ? 32u : 0u;  // lane 0 of warp 1 issues the copies
    // profiling: thread 0 of the first and last CTA records phase clocks per step
    long long *trace = (a.trace && tid == 0 && (blockIdx.x == 0 || blockIdx.x == gridDim.x - 1))
                           ? a.trace + (blockIdx.x == 0 ? 0 : static_cast<size_t>(a.n_steps) * 8)
                           : nullptr;

    // thread 0 issues the copies of step j into stage j & 1
    auto issue = [&](uint32_t j) {
        const uint32_t st = j & 1u;
        const uint32_t row0 = (j % a.n_sets) * a.K + m0;
        const uint32_t bytes = sh.n_boxes * sh.box_rows * P + cnt * 4u * (a.idx ? 2u : 1u);
        mbar_arrive_expect_tx(&bar[st], bytes);
        for (uint32_t b = 0; b < sh.n_boxes; ++b)
            tma_load_2d_hint(pay_of(st) + b * sh.box_rows * P, &tmap, 0,
                             static_cast<int32_t>(row0 + b * sh.box_rows), &bar[st], stream_pol);
        bulk_load_hint(out_of(st), a.outcome + row0, cnt * 4u, &bar[st], stream_pol);
        if (a.idx) bulk_load_hint(idx_of(st), a.idx + row0, cnt * 4u, &bar[st], stream_pol);
        s_pending |= 1u << st;
        s_pend_step[st] = j;
    };
    // bounded wait for stage st's copies; false when it gave up
    auto wait_stage = [&](uint32_t st, uint32_t parity) -> bool { return mbar_wait_bounded(&bar[st], parity, limit); };

    if (tid == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        fence_mbar_init();
        s_sel = ld_volatile_u32(&a.dev->sel) & 1u;
        s_abort = 0;
        s_pending = 0;
    }
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    __syncthreads();
    if (tid == 0 && cnt > 0) {
        if (a.n_steps > 0) issue(0);
        if (a.n_steps > 1) issue(1);
    }
    uint32_t sel = s_sel;
    for (uint32_t n = 0; n < a.n_steps; ++n) {
        const uint32_t st = n & 1u;
        uint32_t odd = 0;
        if (trace) trace[n * 8 + 0] = clock64();
        if (cnt > 0) {
            if (!wait_stage(st, (n >> 1) & 1u)) {
                latch_error(a.dev, DEV_E_TIMEOUT, n, blockIdx.x);
                atomicExch(&a.dev->abort, 1u);
                s_abort = 1;
            }
        }
        __syncthreads();
        if (s_abort) break;
        if (trace) trace[n * 8 + 1] = clock64();
        if (NV >= 2 && cnt <= blockDim.x) {
            odd = coop_transition<SB, P>(a, idx_of(st), out_of(st), pay_of(st), rec_st, cnt, m0,
                                         tab + sel * a.tab_stride, sel, n, keep_pol);
        } else {
            for (uint32_t t = tid; t < cnt; t += blockDim.x) {
                Event<P> ev;
                ev.s = a.idx ? idx_of(st)[t] : m0 + t;
                ev.o = out_of(st)[t];
                read_payload_swizzled<P>(ev.pw, pay_of(st), t);
                odd += transition<SB, P, true, true>(a, ev, tab + sel * a.tab_stride, sel, n, m0 + t, keep_pol);
            }
        }
        uint32_t v = odd;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if ((tid & 31u) == 0) warp_odd[tid >> 5] = v;
        __syncthreads();  // every thread is done with stage st and has stored this step's records
        if (tid == 0) {
            if (trace) trace[n * 8 + 2] = clock64();
            uint32_t c = 0;
            for (uint32_t w = 0; w < (blockDim.x + 31u) / 32u; ++w) c += warp_odd[w];
            unsigned long long *word = &a.dev->slot[n % 3u];
            if (blockIdx.x == 0) a.dev->slot[(n + 1u) % 3u] = 0ull;
            const bool skip = (n == 0 && blockIdx.x == 1 && ld_volatile_u32(&a.dev->skip_arrival) != 0u);
            if (!skip) red_release_add_u64(word, (1ull << 32) | c);
            if (trace) trace[n * 8 + 3] = clock64();
            if (issuer == 0) {
                if (cnt > 0) s_pending &= ~(1u << st);
                if (cnt > 0 && n + 2u < a.n_steps) {
                    fence_proxy_async_smem();
                    issue(n + 2u);
                }
            }
            if (trace) trace[n * 8 + 4] = clock64();
            uint64_t t0 = 0;
            unsigned long long w;
            uint32_t spins = 0;
            for (;;) {
                w = ld_acquire_u64(word);
                if ((w >> 32) >= gridDim.x) break;
                if ((++spins & 63u) == 0u) {
                    if (ld_volatile_u32(&a.dev->abort) != 0u) {
                        s_abort = 1;
                        break;
                    }
                    if (timed_out(t0, limit)) {
                        latch_error(a.dev, DEV_E_TIMEOUT, n, blockIdx.x);
                        atomicExch(&a.dev->abort, 1u);
                        s_abort = 1;
                        break;
                    }
                }
            }
            if (trace) trace[n * 8 + 5] = clock64();
            const uint32_t d = (static_cast<uint32_t>(w & 0xffffffffull) > a.K / 2u) ? 1u : 0u;
            s_sel = d;
            if (blockIdx.x == 0 && a.decisions && !s_abort) a.decisions[n] = d;
        } else if (tid == issuer) {
            // the copies for step n + 2 go out while thread 0 arrives and waits
            if (cnt > 0) s_pending &= ~(1u << st);
            if (cnt > 0 && n + 2u < a.n_steps) {
                fence_proxy_async_smem();
                issue(n + 2u);
            }
        }
        __syncthreads();
        if (s_abort) break;
        sel = s_sel;
    }
    if (s_abort) {
        // drain this CTA's copies still in flight (bounded) before leaving
        if (tid == 0) {
            for (uint32_t st = 0; st < 2; ++st) {
                if (!(s_pending & (1u << st))) continue;
                // the pending use of stage st is step s_pend_step[st]: its phase parity
                const uint32_t parity = (s_pend_step[st] >> 1) & 1u;
                const uint64_t t0 = globaltimer_ns();
                while (!mbar_try_wait(&bar[st], parity)) {
                    if (globaltimer_ns() - t0 > limit) break;
                }
            }
        }
        __syncthreads();
        return;
    }
    if (blockIdx.x == 0 && tid == 0) {
        if (a.n_steps > 0) a.dev->sel = sel;
        a.dev->step = a.n_steps;
    }
}

// ---------------------------------------------------------------------------
// Links between consecutive cohorts of the event ring (explicit session
// indices, K <= 512).  For member m of cohort j, lnk[j][m] holds 1 + the
// position of the same session in cohort j - 1 (low 16 bits) and in cohort
// j - 2 (high 16 bits), 0 where it is absent; cohorts are taken modulo n_sets,
// as the chain takes them.  Sessions are distinct within a cohort, so each
// position is unique; an index >= N is never linked (its member is rejected
// anyway).  One CTA per cohort at a time, two open-addressing tables in shared
// memory (1024 slots for at most 512 keys, so every probe sequence ends).
// ---------------------------------------------------------------------------
constexpr uint32_t kLinkSlots = 1024;
constexpr uint32_t kLinkEmpty = 0xFFFFFFFFu;

__device__ __forceinline__ uint32_t link_hash(uint32_t s) { return (s * 0x9E3779B1u) >> 22; }

__global__ void __launch_bounds__(512) k_link(const uint32_t *idx, uint32_t n_sets, uint32_t K, uint64_t N,
                                              uint32_t *lnk) {
    __shared__ uint32_t key[2][kLinkSlots];
    __shared__ uint16_t pos[2][kLinkSlots];
    for (uint32_t j = blockIdx.x; j < n_sets; j += gridDim.x) {
        for (uint32_t i = threadIdx.x; i < 2 * kLinkSlots; i += blockDim.x) (&key[0][0])[i] = kLinkEmpty;
        __syncthreads();
        for (uint32_t t = 0; t < 2; ++t) {
            const uint32_t src = static_cast<uint32_t>((static_cast<uint64_t>(j) + 2ull * n_sets - 1u - t) % n_sets);
            for (uint32_t m = threadIdx.x; m < K; m += blockDim.x) {
                const uint32_t s = __ldg(idx + static_cast<size_t>(src) * K + m);
                if (s >= N) continue;
                uint32_t h = link_hash(s);
                for (uint32_t probe = 0; probe < kLinkSlots; ++probe) {
                    const uint32_t prev = atomicCAS(&key[t][h], kLinkEmpty, s);
                    if (prev == kLinkEmpty || prev == s) {
                        pos[t][h] = static_cast<uint16_t>(m);
                        break;
                    }
                    h = (h + 1u) & (kLinkSlots - 1u);
                }
            }
        }
        __syncthreads();
        for (uint32_t m = threadIdx.x; m < K; m += blockDim.x) {
            const uint32_t s = __ldg(idx + static_cast<size_t>(j) * K + m);
            uint32_t l = 0;
            if (s < N) {
#pragma unroll
                for (uint32_t t = 0; t < 2; ++t) {
                    uint32_t h = link_hash(s);
                    for (uint32_t probe = 0; probe < kLinkSlots; ++probe) {
                        const uint32_t k = key[t][h];
                        if (k == s) {
                            l |= (static_cast<uint32_t>(pos[t][h]) + 1u) << (16u * t);
                            break;
                        }
                        if (k == kLinkEmpty) break;
                        h = (h + 1u) & (kLinkSlots - 1u);
                    }
                }
            }
            lnk[static_cast<size_t>(j) * K + m] = l;
        }
        __syncthreads();
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, one CTA, explicit session indices (K <= 512), with the
// state gather off the critical path.  The record of a step-n member is
// fetched (per-thread asynchronous copy) at the top of step n - 2, when every
// store of steps <= n - 3 is visible to the CTA.  A member whose session was
// also in step n - 1 or n - 2 (its link) takes that step's result from the
// shared record ring instead: each step leaves there, in its own slot, the
// record it wrote, or the record as it stood for a rejected member.
//
// Every copy is a per-thread asynchronous copy of the thread's own member:
// records, outcomes and payload rows two steps ahead, session indices and
// links four.  The decision is the block barrier's own count (bar.red.popc),
// the only block barrier of a step.  This form takes any K <= 512; for K a
// multiple of 8, k_chain_cta_prod below moves every copy to a producer warp.
// ---------------------------------------------------------------------------
constexpr uint32_t kLinkRI = 5;  // index / link slots
constexpr uint32_t kLinkRP = 3;  // outcome / payload slots
constexpr uint32_t kLinkRR = 5;  // record slots

struct LinkShape {
    uint32_t box_rows;   // payload rows per tensor tile (producer form)
    uint32_t n_boxes;    // tiles per step (producer form)
    uint32_t stage_pay;  // payload bytes per slot (a multiple of 1024)
    uint32_t prod;       // 1: k_chain_cta_prod, 0: k_chain_cta_link
};

template <int SB, int P>
__global__ void __launch_bounds__(512, 1) k_chain_cta_link(StepArgs a, const uint32_t *lnk, LinkShape sh) {
    constexpr uint32_t NC = P / 16;
    constexpr int NV = SB / 16;
    constexpr uint32_t RI = kLinkRI, RP = kLinkRP, RR = kLinkRR;
    extern __shared__ uint8_t dsm_raw[];
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t K = a.K;
    const uint32_t Kp = (K + 3u) & ~3u;
    const uint32_t tid = threadIdx.x;
    const uint32_t nst = a.n_steps;
    // layout: [payload slots][records][indices][links][outcomes][tables]
    uint8_t *const pay = base;
    uint4 *const rec = reinterpret_cast<uint4 *>(base + static_cast<size_t>(RP) * sh.stage_pay);  // [RR][Kp][NV]
    uint32_t *const sidx = reinterpret_cast<uint32_t *>(rec + static_cast<size_t>(RR) * Kp * NV);  // [RI][Kp]
    uint32_t *const slnk = sidx + RI * Kp;                                                         // [RI][Kp]
    uint32_t *const sout = slnk + RI * Kp;                                                         // [RP][Kp]
    uint8_t *const tab = reinterpret_cast<uint8_t *>(sout + RP * Kp);
    const bool act = tid < K;
    const uint32_t m = tid;
    long long *trace = (a.trace && tid == 0) ? a.trace : nullptr;

    auto issue_idx = [&](uint32_t j) {  // session index and link of step j
        if (!act || j >= nst) return;
        const size_t e = static_cast<size_t>(j % a.n_sets) * K + m;
        cp_async4(&sidx[(j % RI) * Kp + m], a.idx + e);
        cp_async4(&slnk[(j % RI) * Kp + m], lnk + e);
    };
    auto issue_rec = [&](uint32_t j) {  // record (by the index already here) and outcome of step j
        if (!act || j >= nst) return;
        const size_t e = static_cast<size_t>(j % a.n_sets) * K + m;
        const uint32_t s = sidx[(j % RI) * Kp + m];
        if (s < a.n_sessions) {
            const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s) * SB);
            uint4 *dst = rec + (static_cast<size_t>(j % RR) * Kp + m) * NV;
#pragma unroll
            for (int k = 0; k < NV; ++k) cp_async16(dst + k, rp + k);
        }
        cp_async4(&sout[(j % RP) * Kp + m], a.outcome + e);
        const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + e * P);
        uint4 *ring = reinterpret_cast<uint4 *>(pay + static_cast<size_t>(j % RP) * sh.stage_pay);
#pragma unroll
        for (uint32_t k = 0; k < NC; ++k) cp_async16(ring + pay_chunk<P>(m, k), src + k);
    };
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    uint32_t sel = ld_volatile_u32(&a.dev->sel) & 1u;
    // prologue: indices of steps 0..3, then the records of steps 0 and 1 in
    // the group pattern of the loop (record group, index group) per step
    for (uint32_t j = 0; j < 4; ++j) issue_idx(j);
    cp_async_commit();
    cp_async_wait<0>();
    issue_rec(0);
    cp_async_commit();
    cp_async_commit();
    issue_rec(1);
    cp_async_commit();
    cp_async_commit();
    __syncthreads();

    for (uint32_t n = 0; n < nst; ++n) {
        if (trace) trace[n * 8 + 0] = clock64();
        cp_async_wait<2>();  // record, outcome and payload of step n; index of step n + 2
        if (trace) trace[n * 8 + 1] = clock64();
        issue_rec(n + 2u);
        cp_async_commit();
        issue_idx(n + 4u);
        cp_async_commit();
        if (trace) trace[n * 8 + 2] = clock64();
        uint32_t odd = 0;
        if (act) {
            const uint32_t s = sidx[(n % RI) * Kp + m];
            const uint32_t l = slnk[(n % RI) * Kp + m];
            const uint32_t o = sout[(n % RP) * Kp + m];
            uint4 *mine = rec + (static_cast<size_t>(n % RR) * Kp + m) * NV;
            if (s >= a.n_sessions) {
                latch_error(a.dev, DEV_E_INDEX, n, m);
            } else {
                const uint32_t p1 = l & 0xFFFFu, p2 = l >> 16;
                const uint4 *src = mine;
                if (p1 != 0u && n >= 1u)
                    src = rec + (static_cast<size_t>((n - 1u) % RR) * Kp + (p1 - 1u)) * NV;
                else if (p2 != 0u && n >= 2u)
                    src = rec + (static_cast<size_t>((n - 2u) % RR) * Kp + (p2 - 1u)) * NV;
                uint4 r[NV];
#pragma unroll
                for (int k = 0; k < NV; ++k) r[k] = src[k];
                const uint32_t x = r[0].x;
                if (x >= a.S || o >= 8u) {
                    latch_error(a.dev, DEV_E_STATE, n, m);
                    if (src != mine) {
#pragma unroll
                        for (int k = 0; k < NV; ++k) mine[k] = r[k];
                    }
                } else {
                    uint4 pw[NC];
                    const uint4 *ring = reinterpret_cast<const uint4 *>(pay + static_cast<size_t>(n % RP) * sh.stage_pay);
#pragma unroll
                    for (uint32_t k = 0; k < NC; ++k) pw[k] = ring[pay_chunk<P>(m, k)];
                    const uint64_t rk = route_key<P>(x, o, pw);
                    const uint32_t y = tab[sel * a.tab_stride + x * 8u + o];
                    r[0].x = y;
                    r[0].y = r[0].y + 1u;
                    mix_acc<SB>(r, rk);
                    uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s) * SB);
#pragma unroll
                    for (int k = 0; k < NV; ++k) {
                        mine[k] = r[k];
                        rp[k] = r[k];
                    }
                    const size_t slot = static_cast<size_t>(n) * K + m;
                    if (a.effects) {
                        uint4 e;
                        e.x = static_cast<uint32_t>(rk);
                        e.y = static_cast<uint32_t>(rk >> 32);
                        e.z = s;
                        e.w = y | (o << 16) | (sel << 24);
                        __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
                    }
                    if (a.state_log) {
                        uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
                        for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
                    }
                    odd = static_cast<uint32_t>(rk & 1u);
                }
            }
        }
        if (trace) trace[n * 8 + 3] = clock64();
        // the block barrier counts the odd keys; it also publishes this step's
        // record slots and orders its state stores
        const uint32_t total = static_cast<uint32_t>(__syncthreads_count(odd));
        if (trace) trace[n * 8 + 4] = clock64();
        sel = total > K / 2u ? 1u : 0u;
        if (tid == 0 && a.decisions) a.decisions[n] = sel;
    }
    cp_async_wait<0>();
    if (tid == 0) {
        if (nst > 0) a.dev->sel = sel;
        a.dev->step = nst;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, one CTA, explicit session indices, K a multiple of 8 up
// to 512, with a producer warp for the streams.  Warps 0 .. ceil(K/32) - 1
// transition one member per thread; lane 0 of the last warp, in region n
// (from the block barrier of step n - 1 to that of step n):
//   - stores decision n - 1;
//   - issues the outcome, session-index and link runs of step n + 5 (1-D bulk
//     copies onto mbarrier W[(n + 5) % 6]) and the payload tiles of step
//     n + 3 (tensor copies onto mbarrier P[(n + 3) % 4]);
//   - waits (bounded) for the runs of step n + 3 and the tiles of step n + 1.
// The barrier of step n then tells every member warp that what it reads in
// region n + 1 has landed, so member warps never wait on an mbarrier and
// never issue a load for the streams.
//
// The one scattered access, the gather of state records, stays with the
// member warps: in step n each thread gathers (asynchronous copy) the record
// of its member of step n + 2, even warps before their transition and odd
// warps after it.  The gather of step j thus starts once every store of
// steps <= j - 3 is visible; a member whose session was in step j - 1 or
// j - 2 takes that step's result from the shared record ring (links from
// k_link), as in k_chain_cta_link.  The decision is the barrier's own count.
// A producer wait that runs out latches RC_E_TIMEOUT; the CTA stops after
// that step, the producer first waiting (bounded) for the copies it still
// has in flight.  Trace points (thread 0): 0 region start, 1 record landed,
// 4 input state read, 5 payload read, 6 key done, 2 transition done, 3 after
// the barrier.
// ---------------------------------------------------------------------------
constexpr uint32_t kProdRW = 6;  // word slots (issued five steps ahead)
constexpr uint32_t kProdRP = 4;  // payload slots (issued three steps ahead)
constexpr uint32_t kProdRR = 5;  // record slots (two ahead, two of forwarding)

template <int SB, int P>
__global__ void __launch_bounds__(544, 1)
    k_chain_cta_prod(const __grid_constant__ CUtensorMap tmap, StepArgs a, const uint32_t *lnk, LinkShape sh) {
    constexpr int NV = SB / 16;
    constexpr uint32_t RW = kProdRW, RP = kProdRP, RR = kProdRR;
    extern __shared__ uint8_t dsm_raw[];
    __shared__ __align__(8) uint64_t wbar[RW];
    __shared__ __align__(8) uint64_t pbar[RP];
    __shared__ uint32_t s_ab[2];
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t K = a.K;
    const uint32_t Kw = (K + 31u) & ~31u;  // member threads; the producer warp follows
    const uint32_t tid = threadIdx.x;
    const bool prod = tid >= Kw;
    const bool early = ((tid >> 5) & 1u) == 0u;  // even member warps gather before their transition
    const uint32_t nst = a.n_steps;
    const uint64_t limit = a.dev->wait_ns;
    // layout: [payload slots][records][word slots: outcome, index, link][tables]
    uint8_t *const pay = base;
    uint4 *const rec = reinterpret_cast<uint4 *>(base + static_cast<size_t>(RP) * sh.stage_pay);  // [RR][K][NV]
    uint32_t *const words = reinterpret_cast<uint32_t *>(rec + static_cast<size_t>(RR) * K * NV);  // [RW][3][K]
    uint8_t *const tab = reinterpret_cast<uint8_t *>(words + static_cast<size_t>(RW) * 3 * K);
    auto word_of = [&](uint32_t j, uint32_t which) { return words + (static_cast<size_t>(j % RW) * 3 + which) * K; };
    const uint64_t stream_pol = policy_evict_first();
    long long *trace = (a.trace && tid == 0) ? a.trace : nullptr;

    // producer lane 0 only
    auto issue_words = [&](uint32_t j) {
        if (j >= nst) return;
        const size_t e0 = static_cast<size_t>(j % a.n_sets) * K;
        uint64_t *b = &wbar[j % RW];
        mbar_arrive_expect_tx(b, 3u * K * 4u);
        bulk_load_hint(word_of(j, 0), a.outcome + e0, K * 4u, b, stream_pol);
        bulk_load_hint(word_of(j, 1), a.idx + e0, K * 4u, b, stream_pol);
        bulk_load_hint(word_of(j, 2), lnk + e0, K * 4u, b, stream_pol);
    };
    auto issue_pay = [&](uint32_t j) {
        if (j >= nst) return;
        const uint32_t st = j % RP;
        const int32_t row0 = static_cast<int32_t>((j % a.n_sets) * K);
        mbar_arrive_expect_tx(&pbar[st], sh.n_boxes * sh.box_rows * P);
        for (uint32_t b = 0; b < sh.n_boxes; ++b)
            tma_load_2d_hint(pay + static_cast<size_t>(st) * sh.stage_pay + b * sh.box_rows * P, &tmap, 0,
                             row0 + static_cast<int32_t>(b * sh.box_rows), &pbar[st], stream_pol);
    };
    auto landed_words = [&](uint32_t j) { return j >= nst || mbar_wait_bounded(&wbar[j % RW], (j / RW) & 1u, limit); };
    auto landed_pay = [&](uint32_t j) { return j >= nst || mbar_wait_bounded(&pbar[j % RP], (j / RP) & 1u, limit); };
    // member thread: gather its record of step j (one commit group, empty past the end);
    // the index run of step j is known to have landed
    auto gather = [&](uint32_t j) {
        if (j < nst && tid < K) {
            const uint32_t s = word_of(j, 1)[tid];
            if (s < a.n_sessions) {
                const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s) * SB);
                uint4 *dst = rec + (static_cast<size_t>(j % RR) * K + tid) * NV;
#pragma unroll
                for (int k = 0; k < NV; ++k) cp_async16(dst + k, rp + k);
            }
        }
        cp_async_commit();
    };

    if (tid == 0) {
        for (uint32_t i = 0; i < RW; ++i) mbar_init(&wbar[i], 1);
        for (uint32_t i = 0; i < RP; ++i) mbar_init(&pbar[i], 1);
        fence_mbar_init();
        s_ab[0] = 0;
        s_ab[1] = 0;
    }
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    uint32_t sel = ld_volatile_u32(&a.dev->sel) & 1u;
    __syncthreads();
    // prologue: runs of steps 0..4 and tiles of steps 0..2 go out; the runs
    // of steps 0..2 and the tiles of step 0 are waited for; the member warps
    // then gather the records of steps 0 and 1
    if (tid == Kw) {
        for (uint32_t j = 0; j + 1u < RW; ++j) issue_words(j);
        for (uint32_t j = 0; j + 1u < RP; ++j) issue_pay(j);
        if (!(landed_words(0) && landed_words(1) && landed_words(2) && landed_pay(0))) {
            latch_error(a.dev, DEV_E_TIMEOUT, 0, tid);
            s_ab[0] = 1;
        }
    }
    __syncthreads();
    const bool started = s_ab[0] == 0u;  // false: the prologue gave up a wait, no step runs
    if (started && !prod) {
        gather(0);
        gather(1);
    }

    // A thread that gives up a wait in region n raises s_ab[n & 1]; all
    // threads read it after the barrier of step n, before anyone can write it
    // again.
    uint32_t n = 0;
    for (; started && n < nst; ++n) {
        uint32_t odd = 0;
        if (prod) {
            if (tid == Kw) {
                if (n > 0 && a.decisions) a.decisions[n - 1u] = sel;
                issue_words(n + RW - 1u);
                issue_pay(n + RP - 1u);
                if (!(landed_words(n + 3u) && landed_pay(n + 1u))) {
                    latch_error(a.dev, DEV_E_TIMEOUT, n, tid);
                    s_ab[n & 1u] = 1;
                }
            }
        } else {
            if (trace) trace[n * 8 + 0] = clock64();
            if (early) {
                gather(n + 2u);
                cp_async_wait<2>();  // this thread's record of step n
            } else {
                cp_async_wait<1>();
            }
            if (trace) trace[n * 8 + 1] = clock64();
            if (tid < K) {
                const uint32_t m = tid;
                const uint32_t o = word_of(n, 0)[m];
                const uint32_t s = word_of(n, 1)[m];
                const uint32_t l = word_of(n, 2)[m];
                uint4 *mine = rec + (static_cast<size_t>(n % RR) * K + m) * NV;
                if (s >= a.n_sessions) {
                    latch_error(a.dev, DEV_E_INDEX, n, m);
                } else {
                    const uint32_t p1 = l & 0xFFFFu, p2 = l >> 16;
                    const uint4 *src = mine;
                    if (p1 != 0u && n >= 1u)
                        src = rec + (static_cast<size_t>((n - 1u) % RR) * K + (p1 - 1u)) * NV;
                    else if (p2 != 0u && n >= 2u)
                        src = rec + (static_cast<size_t>((n - 2u) % RR) * K + (p2 - 1u)) * NV;
                    uint4 r[NV];
#pragma unroll
                    for (int k = 0; k < NV; ++k) r[k] = src[k];
                    const uint32_t x = r[0].x;
                    if (trace) {
                        asm volatile("" ::"r"(x));
                        trace[n * 8 + 4] = clock64();
                    }
                    if (x >= a.S || o >= 8u) {
                        latch_error(a.dev, DEV_E_STATE, n, m);
                        if (src != mine) {
#pragma unroll
                            for (int k = 0; k < NV; ++k) mine[k] = r[k];
                        }
                    } else {
                        uint4 pw[P / 16];
                        read_payload_swizzled<P>(pw, pay + static_cast<size_t>(n % RP) * sh.stage_pay, m);
                        if (trace) {
                            asm volatile("" ::"r"(pw[P / 16 - 1].w));
                            trace[n * 8 + 5] = clock64();
                        }
                        const uint64_t rk = route_key<P>(x, o, pw);
                        if (trace) {
                            asm volatile("" ::"l"(rk));
                            trace[n * 8 + 6] = clock64();
                        }
                        const uint32_t y = tab[sel * a.tab_stride + x * 8u + o];
                        r[0].x = y;
                        r[0].y = r[0].y + 1u;
                        mix_acc<SB>(r, rk);
                        uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s) * SB);
#pragma unroll
                        for (int k = 0; k < NV; ++k) {
                            mine[k] = r[k];
                            rp[k] = r[k];
                        }
                        const size_t slot = static_cast<size_t>(n) * K + m;
                        if (a.effects) {
                            uint4 e;
                            e.x = static_cast<uint32_t>(rk);
                            e.y = static_cast<uint32_t>(rk >> 32);
                            e.z = s;
                            e.w = y | (o << 16) | (sel << 24);
                            __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
                        }
                        if (a.state_log) {
                            uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
                            for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
                        }
                        odd = static_cast<uint32_t>(rk & 1u);
                    }
                }
            }
            if (trace) {
                asm volatile("" ::"r"(odd));
                trace[n * 8 + 2] = clock64();
            }
            if (!early) gather(n + 2u);
        }
        // the count of odd keys; the barrier also publishes this step's record
        // slots and the producer's news, orders the state stores and frees the
        // slots of step n
        const uint32_t total = static_cast<uint32_t>(__syncthreads_count(odd));
        if (trace) trace[n * 8 + 3] = clock64();
        if (s_ab[n & 1u] != 0u) break;
        sel = total > K / 2u ? 1u : 0u;
    }
    cp_async_wait<0>();
    if (tid == Kw) {
        if (n == nst && nst > 0 && a.decisions) a.decisions[nst - 1u] = sel;
        if (n < nst) {
            // stopped early: wait (bounded) for the runs and tiles issued so
            // far (through step n + 5 and n + 3 once the loop ran)
            const uint32_t w_end = started ? n + RW : RW - 1u, p_end = started ? n + RP : RP - 1u;
            for (uint32_t j = n; j < w_end && j < nst; ++j) (void)landed_words(j);
            for (uint32_t j = n; j < p_end && j < nst; ++j) (void)landed_pay(j);
        }
    }
    if (tid == 0 && n == nst) {
        if (nst > 0) a.dev->sel = sel;
        a.dev->step = nst;
    }
}

// ---------------------------------------------------------------------------
// Links of reach D: for member m of cohort j, the distance t (1..D) to the
// nearest earlier cohort holding the same session (cohorts taken cyclically,
// as a chain walks them) and its position q there, packed as t << 16 | q; 0
// when none of the D cohorts before holds the session or the index is out of
// range.  One CTA per cohort and one open-addressing table of SLOTS slots
// (at most SLOTS / 2 keys: D * K <= SLOTS / 2): every member of the D earlier
// cohorts is inserted under its session, the packed value kept by atomicMin
// (the nearest cohort wins), and each member of cohort j probes once.
// ---------------------------------------------------------------------------
constexpr uint32_t kPairD = 8;  // reach of k_chain_cta_pair's links

template <uint32_t D, uint32_t SLOTS>
__global__ void __launch_bounds__(512) k_link_reach(const uint32_t *idx, uint32_t n_sets, uint32_t K, uint64_t N,
                                                    uint32_t *lnk) {
    static_assert((SLOTS & (SLOTS - 1)) == 0 && SLOTS >= 64 && SLOTS <= 65536, "slots: a power of two");
    constexpr uint32_t shift = 32u - static_cast<uint32_t>(__builtin_ctz(SLOTS));
    __shared__ uint32_t key[SLOTS];
    __shared__ uint32_t val[SLOTS];
    __shared__ uint32_t src[D];
    auto hash = [](uint32_t s) { return (s * 0x9E3779B1u) >> shift; };
    for (uint32_t j = blockIdx.x; j < n_sets; j += gridDim.x) {
        for (uint32_t i = threadIdx.x; i < SLOTS; i += blockDim.x) {
            key[i] = kLinkEmpty;
            val[i] = 0xFFFFFFFFu;
        }
        if (threadIdx.x < D)
            src[threadIdx.x] = static_cast<uint32_t>(
                (static_cast<uint64_t>(j) + D * static_cast<uint64_t>(n_sets) - 1u - threadIdx.x) % n_sets);
        __syncthreads();
        // D elements per thread at a time: their loads go out together, ahead
        // of the table's atomics
        for (uint32_t base = 0; base < D * K; base += D * blockDim.x) {
            uint32_t sv[D], tv[D], mv[D];
#pragma unroll
            for (uint32_t i = 0; i < D; ++i) {
                const uint32_t e = base + i * blockDim.x + threadIdx.x;
                const bool in = e < D * K;
                tv[i] = in ? e / K : 0u;
                mv[i] = in ? e - tv[i] * K : 0u;
                sv[i] = in ? __ldg(idx + static_cast<size_t>(src[tv[i]]) * K + mv[i]) : kLinkEmpty;
            }
#pragma unroll
            for (uint32_t i = 0; i < D; ++i) {
                const uint32_t s = sv[i];
                if (s >= N) continue;
                uint32_t h = hash(s);
                for (uint32_t probe = 0; probe < SLOTS; ++probe) {
                    const uint32_t prev = atomicCAS(&key[h], kLinkEmpty, s);
                    if (prev == kLinkEmpty || prev == s) {
                        atomicMin(&val[h], ((tv[i] + 1u) << 16) | mv[i]);
                        break;
                    }
                    h = (h + 1u) & (SLOTS - 1u);
                }
            }
        }
        __syncthreads();
        for (uint32_t m = threadIdx.x; m < K; m += blockDim.x) {
            const uint32_t s = __ldg(idx + static_cast<size_t>(j) * K + m);
            uint32_t l = 0;
            if (s < N) {
                uint32_t h = hash(s);
                for (uint32_t probe = 0; probe < SLOTS; ++probe) {
                    const uint32_t k = key[h];
                    if (k == s) {
                        l = val[h];
                        break;
                    }
                    if (k == kLinkEmpty) break;
                    h = (h + 1u) & (SLOTS - 1u);
                }
            }
            lnk[static_cast<size_t>(j) * K + m] = l;
        }
        __syncthreads();
    }
}

// Named barrier `id` over `count` threads (a multiple of 32): arrive and wait.
__device__ __forceinline__ void named_sync(uint32_t id, uint32_t count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}

// Route key from its first finaliser round h0 = fin64((x | o << 32) ^ gamma),
// taken from a table: one more round per 64-bit payload word.
template <int P>
__device__ __forceinline__ uint64_t route_key_from(uint64_t h, const uint4 (&pw)[P / 16]) {
#pragma unroll
    for (int k = 0; k < P / 16; ++k) {
        h = fin64(h ^ pack64(pw[k].x, pw[k].y));
        h = fin64(h ^ pack64(pw[k].z, pw[k].w));
    }
    return h;
}

// ---------------------------------------------------------------------------
// Persistent chain, one CTA, explicit session indices, K a multiple of 8 up
// to 256, payloads of at most 64 bytes: two steps per block barrier.
//
// The route key of step j depends on the decisions only through the state
// value x the step reads, and the state a session left in step i is
// T_{sel_i}[x_i][o_i] with sel_i = d_{i-1}.  So the keys of step j need the
// decisions up to d_{j-2}, and steps 2r and 2r + 1 can be keyed side by side
// once d_{2r-1} is known.  Region r (between two block barriers):
//   key group A (warps 0 .. ceil(K/32) - 1) takes step 2r, key group B (the
//   next ceil(K/32) warps) step 2r + 1, one member per thread.  x comes from
//   the session's previous appearance (k_link_reach, up to kPairD steps
//   back: the input state and outcome that step left in the rings X and O,
//   and that step's decision) or from its record gathered from HBM.  A
//   member of step 2r + 1 whose session is in step 2r follows that member's
//   own link one level further.  The key is a table of first rounds plus one
//   finaliser round per payload word, the payload read from a swizzled tile.
//   Two block barriers end the region; their counts are the two groups' odd
//   keys.
//   The record group (the next ceil(K/32) warps) completes the records of
//   steps 2r - 2 and 2r - 1 (a record-group barrier between the two): the
//   input record is the session's previous output (record ring, up to
//   kPairD steps back) or the gathered one; the output goes to HBM and to
//   the ring, with the effect.  It also gathers the records of steps 2r + 4
//   and 2r + 5 for members without a link: their sessions were last written
//   in step 2r - 4 or earlier, by region r - 1 at the latest, which that
//   region's barrier made visible.
//   The producer lane issues the payload tiles of steps 2r + 2 and 2r + 3,
//   stores decisions 2r - 2 and 2r - 1, issues the outcome, index and link
//   runs of steps 2r + 8 and 2r + 9 and waits (bounded) for those runs of
//   2r + 6 and 2r + 7 and for the two tiles.
// The loop runs one region past the last key step, in which only the record
// group works.  A producer wait that runs out latches RC_E_TIMEOUT; the CTA
// stops after that region, its record group first completing the two steps
// the key groups finished.  Trace points (thread 0, at step 2r): 0 region
// start, 1 x ready, 2 key done, 3 after the barrier.
// ---------------------------------------------------------------------------
constexpr uint32_t kPairRW = 16;  // word slots
constexpr uint32_t kPairRR = 16;  // record slots
constexpr uint32_t kPairRX = 16;  // input-state / outcome slots
constexpr uint32_t kPairRK = 4;   // key / flag slots
constexpr uint32_t kPairSkip = 0, kPairRejected = 1, kPairApplied = 2;  // member flags
constexpr uint32_t kPairRP = 4;   // payload tile slots

template <int SB, int P>
__global__ void __launch_bounds__(800, 1)
    k_chain_cta_pair(const __grid_constant__ CUtensorMap tmap, StepArgs a, const uint32_t *lnk, LinkShape sh) {
    constexpr int NV = SB / 16;
    constexpr int PV = P / 16;
    constexpr uint32_t RW = kPairRW, RR = kPairRR, RX = kPairRX, RK = kPairRK, RP = kPairRP;
    extern __shared__ uint8_t dsm_raw[];
    __shared__ __align__(8) uint64_t wbar[RW];
    __shared__ __align__(8) uint64_t pbar[RP];
    __shared__ uint32_t s_ab[2];
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t K = a.K;
    const uint32_t Kw = (K + 31u) & ~31u;
    const uint32_t tid = threadIdx.x;
    const uint32_t grp = tid / Kw;      // 0: key A, 1: key B, 2: records, 3: producer
    const uint32_t m = tid - grp * Kw;  // member (groups 0 .. 2)
    const uint32_t nst = a.n_steps;
    const uint32_t stride = a.tab_stride;
    const uint64_t limit = a.dev->wait_ns;
    // layout: payload tiles [RP] | records [RR][K][NV] | h0 [S][8] | keys [RK][K] |
    //         words [RW][3][K] | X [RX][K] | O [RX][K] (u8) | flags [RK][K] (u8) | tables
    uint8_t *const pay = base;
    uint4 *const rec = reinterpret_cast<uint4 *>(base + static_cast<size_t>(RP) * sh.stage_pay);
    uint64_t *const h0 = reinterpret_cast<uint64_t *>(rec + static_cast<size_t>(RR) * K * NV);
    uint64_t *const rks = h0 + static_cast<size_t>(a.S) * 8u;
    uint32_t *const words = reinterpret_cast<uint32_t *>(rks + static_cast<size_t>(RK) * K);
    uint32_t *const xs = words + static_cast<size_t>(RW) * 3 * K;
    uint8_t *const os = reinterpret_cast<uint8_t *>(xs + static_cast<size_t>(RX) * K);
    uint8_t *const fls = os + static_cast<size_t>(RX) * K;
    uint8_t *const tab = fls + static_cast<size_t>(RK) * K;
    // ring offsets stay below 2^20 elements: 32-bit arithmetic
    auto word_of = [&](uint32_t j, uint32_t which) { return words + ((j % RW) * 3u + which) * K; };
    auto rec_of = [&](uint32_t j, uint32_t q) { return rec + ((j % RR) * K + q) * NV; };
    const uint64_t stream_pol = policy_evict_first();
    long long *trace = (a.trace && tid == 0) ? a.trace : nullptr;

    // producer lane only
    auto issue_words = [&](uint32_t j) {
        if (j >= nst) return;
        const size_t e0 = static_cast<size_t>(j % a.n_sets) * K;
        uint64_t *b = &wbar[j % RW];
        mbar_arrive_expect_tx(b, 3u * K * 4u);
        bulk_load_hint(word_of(j, 0), a.outcome + e0, K * 4u, b, stream_pol);
        bulk_load_hint(word_of(j, 1), a.idx + e0, K * 4u, b, stream_pol);
        bulk_load_hint(word_of(j, 2), lnk + e0, K * 4u, b, stream_pol);
    };
    auto landed_words = [&](uint32_t j) { return j >= nst || mbar_wait_bounded(&wbar[j % RW], (j / RW) & 1u, limit); };
    auto issue_pay = [&](uint32_t j) {
        if (j >= nst) return;
        const uint32_t st = j % RP;
        mbar_arrive_expect_tx(&pbar[st], sh.box_rows * P);
        tma_load_2d_hint(pay + static_cast<size_t>(st) * sh.stage_pay, &tmap, 0,
                         static_cast<int32_t>((j % a.n_sets) * K), &pbar[st], stream_pol);
    };
    auto landed_pay = [&](uint32_t j) { return j >= nst || mbar_wait_bounded(&pbar[j % RP], (j / RP) & 1u, limit); };
    auto unlinked = [](uint32_t l, uint32_t j) {
        const uint32_t t = l >> 16;
        return t == 0u || t > j;
    };

    const uint32_t sel0 = ld_volatile_u32(&a.dev->sel) & 1u;
    uint64_t dv = 0;  // bit (i & 63): decision d_i, for the steps decided so far
    auto sel_of = [&](uint32_t j) -> uint32_t {
        return j == 0u ? sel0 : static_cast<uint32_t>((dv >> ((j - 1u) & 63u)) & 1u);
    };
    // the state member q of step j left its session in (rings X and O of step j)
    auto after = [&](uint32_t j, uint32_t q) -> uint32_t {
        const uint32_t x = xs[(j % RX) * K + q];
        const uint32_t o = os[(j % RX) * K + q];
        return (x < a.S && o < 8u) ? static_cast<uint32_t>(tab[sel_of(j) * stride + x * 8u + o]) : x;
    };

    // key thread: the outcome, index and link of its next step, loaded a
    // region ahead
    auto key_prefetch = [&](uint32_t j, uint32_t &o, uint32_t &s, uint32_t &l) {
        if (j < nst && m < K) {
            o = word_of(j, 0)[m];
            s = word_of(j, 1)[m];
            l = word_of(j, 2)[m];
        }
    };
    // key thread: x, the rings X and O, the key and the flag of its member of
    // step j; `chase` for group B (a session in step j - 1 is in this region)
    auto key_step = [&](uint32_t j, bool chase, uint32_t o, uint32_t s, uint32_t l) {
        uint32_t odd = 0;
        if (j >= nst || m >= K) return odd;
        uint4 pw[PV];
        read_payload_swizzled<P>(pw, pay + static_cast<size_t>(j % RP) * sh.stage_pay, m);
        uint32_t f = kPairSkip;
        if (s >= a.n_sessions) {
            latch_error(a.dev, DEV_E_INDEX, j, m);
        } else {
            const uint32_t t = l >> 16, q = l & 0xFFFFu;
            uint32_t x;
            if (t == 0u || t > j) {
                x = rec_of(j, m)[0].x;
            } else if (chase && t == 1u) {
                const uint32_t i = j - 1u;
                const uint32_t l2 = word_of(i, 2)[q];
                const uint32_t oi = word_of(i, 0)[q];
                const uint32_t xi = unlinked(l2, i) ? rec_of(i, q)[0].x : after(i - (l2 >> 16), l2 & 0xFFFFu);
                x = (xi < a.S && oi < 8u) ? static_cast<uint32_t>(tab[sel_of(i) * stride + xi * 8u + oi]) : xi;
            } else {
                x = after(j - t, q);
            }
            if (trace) {
                asm volatile("" ::"r"(x));
                trace[j * 8 + 1] = clock64();
            }
            xs[(j % RX) * K + m] = x;
            os[(j % RX) * K + m] = static_cast<uint8_t>(o < 8u ? o : 8u);
            if (x >= a.S || o >= 8u) {
                latch_error(a.dev, DEV_E_STATE, j, m);
                f = kPairRejected;
            } else {
                const uint64_t rk = route_key_from<P>(h0[x * 8u + o], pw);
                rks[(j % RK) * K + m] = rk;
                odd = static_cast<uint32_t>(rk & 1u);
                f = kPairApplied;
            }
        }
        fls[(j % RK) * K + m] = static_cast<uint8_t>(f);
        return odd;
    };
    // record thread: gather its member's record of step j when it has no link
    auto gather = [&](uint32_t j) {
        if (j < nst && m < K) {
            const uint32_t s = word_of(j, 1)[m];
            if (s < a.n_sessions && unlinked(word_of(j, 2)[m], j)) {
                const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s) * SB);
                uint4 *dst = rec_of(j, m);
#pragma unroll
                for (int k = 0; k < NV; ++k) cp_async16(dst + k, rp + k);
            }
        }
    };
    // record thread: complete its member's record of step j
    auto record_step = [&](uint32_t j) {
        if (j >= nst || m >= K) return;
        const uint32_t f = fls[(j % RK) * K + m];
        if (f == kPairSkip) return;
        const uint32_t l = word_of(j, 2)[m];
        uint4 *mine = rec_of(j, m);
        const uint4 *src = unlinked(l, j) ? mine : rec_of(j - (l >> 16), l & 0xFFFFu);
        uint4 r[NV];
#pragma unroll
        for (int k = 0; k < NV; ++k) r[k] = src[k];
        if (f == kPairRejected) {
            if (src != mine) {
#pragma unroll
                for (int k = 0; k < NV; ++k) mine[k] = r[k];
            }
            return;
        }
        const uint32_t o = word_of(j, 0)[m];
        const uint32_t s = word_of(j, 1)[m];
        const uint32_t x = xs[(j % RX) * K + m];
        const uint32_t sel = sel_of(j);
        const uint32_t y = tab[sel * stride + x * 8u + o];
        const uint64_t rk = rks[(j % RK) * K + m];
        r[0].x = y;
        r[0].y = r[0].y + 1u;
        mix_acc<SB>(r, rk);
        uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s) * SB);
#pragma unroll
        for (int k = 0; k < NV; ++k) {
            mine[k] = r[k];
            rp[k] = r[k];
        }
        const size_t slot = static_cast<size_t>(j) * K + m;
        if (a.effects) {
            uint4 e;
            e.x = static_cast<uint32_t>(rk);
            e.y = static_cast<uint32_t>(rk >> 32);
            e.z = s;
            e.w = y | (o << 16) | (sel << 24);
            __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
        }
        if (a.state_log) {
            uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
            for (int k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
        }
    };

    if (tid == 0) {
        for (uint32_t i = 0; i < RW; ++i) mbar_init(&wbar[i], 1);
        for (uint32_t i = 0; i < RP; ++i) mbar_init(&pbar[i], 1);
        fence_mbar_init();
        s_ab[0] = 0;
        s_ab[1] = 0;
    }
    stage_tables(tab, a.tables, stride, 2, 0);
    for (uint32_t i = tid; i < a.S * 8u; i += blockDim.x) h0[i] = fin64(pack64(i >> 3, i & 7u) ^ kGamma);
    __syncthreads();
    // prologue: runs of steps 0..7 and tiles of steps 0 and 1 go out; the
    // runs of 0..5 and the tiles are waited for; then the record group gathers
    // steps 0..3 (two copy groups) and waits for the first, and the key groups
    // load their steps 0 and 1
    const uint32_t prod_lane = 3u * Kw;
    if (tid == prod_lane) {
        for (uint32_t j = 0; j < 8u; ++j) issue_words(j);
        issue_pay(0);
        issue_pay(1);
        bool ok = landed_pay(0) && landed_pay(1);
        for (uint32_t j = 0; j < 6u; ++j) ok = ok && landed_words(j);
        if (!ok) {
            latch_error(a.dev, DEV_E_TIMEOUT, 0, tid);
            s_ab[0] = 1;
        }
    }
    __syncthreads();
    const bool started = s_ab[0] == 0u;  // false: the prologue gave up a wait, no step runs
    uint32_t o_a = 0, s_a = 0, l_a = 0, o_b = 0, s_b = 0, l_b = 0;
    if (started) {
        if (grp == 2u) {
            gather(0);
            gather(1);
            cp_async_commit();
            gather(2);
            gather(3);
            cp_async_commit();
            cp_async_wait<1>();
        } else if (grp < 2u) {
            key_prefetch(grp, o_a, s_a, l_a);
        }
    }
    __syncthreads();

    // the last region: its key steps are past the end, the record group
    // completes the last two steps
    const uint32_t r_end = nst == 0u ? 0u : (nst - 1u) / 2u + 1u;
    uint32_t r = 0;
    bool aborted = !started;
    for (; started && r <= r_end; ++r) {
        const uint32_t ja = 2u * r, jb = ja + 1u;
        uint32_t odd_a = 0, odd_b = 0;
        if (grp == 3u) {
            if (tid == prod_lane) {
                issue_pay(ja + 2u);
                issue_pay(ja + 3u);
                if (a.decisions && r > 0) {
                    if (ja - 2u < nst) a.decisions[ja - 2u] = sel_of(ja - 1u);
                    if (ja - 1u < nst) a.decisions[ja - 1u] = sel_of(ja);
                }
                issue_words(ja + 8u);
                issue_words(ja + 9u);
                if (!(landed_words(ja + 6u) && landed_words(ja + 7u) && landed_pay(ja + 2u) &&
                      landed_pay(ja + 3u))) {
                    latch_error(a.dev, DEV_E_TIMEOUT, ja, tid);
                    s_ab[r & 1u] = 1;
                }
            }
        } else if (grp < 2u) {
            const uint32_t j = ja + grp;
            if (trace && j < nst) trace[j * 8 + 0] = clock64();
            // this step's inputs are in (o_a, s_a, l_a); the next step's go to
            // the b set, and the roles swap below
            key_prefetch(j + 2u, o_b, s_b, l_b);
            const uint32_t odd = key_step(j, grp == 1u, o_a, s_a, l_a);
            if (grp == 0u)
                odd_a = odd;
            else
                odd_b = odd;
            if (trace && j < nst) {
                asm volatile("" ::"r"(odd));
                trace[j * 8 + 2] = clock64();
            }
            o_a = o_b;
            s_a = s_b;
            l_a = l_b;
        } else if (grp == 2u) {
            gather(ja + 4u);
            gather(ja + 5u);
            cp_async_commit();
            if (r > 0) record_step(ja - 2u);
            named_sync(2, Kw);
            if (r > 0) record_step(ja - 1u);
            cp_async_wait<1>();  // this thread's copies of steps 2r + 2 and 2r + 3
        }
        // the counts of the two groups' odd keys, one block barrier each; the
        // first also publishes this region's rings, records and the
        // producer's news
        const uint32_t total_a = static_cast<uint32_t>(__syncthreads_count(odd_a));
        const uint32_t total_b = static_cast<uint32_t>(__syncthreads_count(odd_b));
        if (trace && ja < nst) trace[ja * 8 + 3] = clock64();
        if (ja < nst) {
            const uint32_t da = total_a > K / 2u ? 1u : 0u;
            dv = (dv & ~(1ull << (ja & 63u))) | (static_cast<uint64_t>(da) << (ja & 63u));
        }
        if (jb < nst) {
            const uint32_t db = total_b > K / 2u ? 1u : 0u;
            dv = (dv & ~(1ull << (jb & 63u))) | (static_cast<uint64_t>(db) << (jb & 63u));
        }
        if (s_ab[r & 1u] != 0u) {
            aborted = true;
            break;
        }
    }
    // stopped early: the key groups finished steps 2r and 2r + 1, the record
    // group completes them
    if (started && aborted && grp == 2u) {
        record_step(2u * r);
        named_sync(2, Kw);
        record_step(2u * r + 1u);
    }
    cp_async_wait<0>();
    if (tid == prod_lane && aborted) {
        // wait (bounded) for the runs and tiles still in flight
        const uint32_t j0 = started ? 2u * r + 6u : 0u, j1 = started ? 2u * r + 10u : 8u;
        for (uint32_t j = j0; j < j1 && j < nst; ++j) (void)landed_words(j);
        const uint32_t p0 = started ? 2u * r + 2u : 0u, p1 = p0 + 2u;
        for (uint32_t j = p0; j < p1 && j < nst; ++j) (void)landed_pay(j);
    }
    if (tid == 0 && !aborted) {
        if (nst > 0) a.dev->sel = sel_of(nst);
        a.dev->step = nst;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, cooperative grid, split by links (explicit session
// indices, K a multiple of 8; one CTA per SM, CTA b owns the contiguous
// members [b*chunk, b*chunk + cnt) as in k_chain_grid_tma).
//
// lnk[j][m] is non-zero when member m's session also sits in cohort j - 1
// (k_mark / k_flag).  Only such a "linked" member of step n + 1 needs the
// records stored in step n; every other member's record was last stored in
// step n - 1 or earlier, which the grid barrier of step n - 1 already made
// visible.  So each step splits in two regions:
//   A(n)  after the barrier of step n - 1: gather and hash the linked members
//         of step n; then transition every member of step n with d(n - 1),
//         store the records (warp-cooperatively, NV lanes per record) and
//         stage the effects in shared memory;
//   B(n)  the control thread (lane 0 of the last warp) adds (1 << 32 | odd
//         count of step n) to the barrier word with release semantics,
//         stores the effect run of step n with one bulk copy (so the release
//         does not wait for it), issues the event copies of step n + 2 and
//         spins for all CTAs; meanwhile the member warps gather and hash the
//         unlinked members of step n + 1.
// Step 0 has no earlier step in the launch: all its members count as
// unlinked.  Every wait is bounded: a CTA that gives up latches
// RC_E_TIMEOUT, raises dev->abort and leaves after the next block barrier,
// the control thread first waiting (bounded) for its copies in flight.
// ---------------------------------------------------------------------------
struct GridLinkShape {
    TmaShape t;         // chunk, payload tiles, stage sizes (as k_chain_grid_tma)
    uint32_t members;   // member threads (a multiple of 32, >= chunk); the control warp follows
    uint32_t pad[3];
};

__device__ __forceinline__ void bulk_store(void *gdst, const void *ssrc, uint32_t bytes) {
    asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;" ::"l"(gdst), "r"(smem_addr(ssrc)),
                 "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void bulk_wait_read() {
    asm volatile("cp.async.bulk.wait_group.read %0;" ::"n"(N) : "memory");
}
template <int N>
__device__ __forceinline__ void bulk_wait_all() {
    asm volatile("cp.async.bulk.wait_group %0;" ::"n"(N) : "memory");
}

// Marks, per cohort j of the ring, its sessions in bitmap bits[j] (words of
// 32 sessions; the caller clears the bitmaps).
__global__ void k_mark(const uint32_t *idx, uint32_t n_sets, uint32_t K, uint64_t N, uint64_t words_per_set,
                       uint32_t *bits) {
    const size_t total = static_cast<size_t>(n_sets) * K;
    for (size_t e = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const uint32_t s = idx[e];
        if (s >= N) continue;
        const size_t j = e / K;
        atomicOr(bits + j * words_per_set + (s >> 5), 1u << (s & 31u));
    }
}

// lnk[j][m] = 1 when member m's session of cohort j is in cohort j - 1 (mod n_sets).
__global__ void k_flag(const uint32_t *idx, uint32_t n_sets, uint32_t K, uint64_t N, uint64_t words_per_set,
                       const uint32_t *bits, uint32_t *lnk) {
    const size_t total = static_cast<size_t>(n_sets) * K;
    for (size_t e = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const uint32_t s = idx[e];
        const size_t j = e / K;
        const size_t jp = (j + n_sets - 1) % n_sets;
        uint32_t l = 0;
        if (s < N) l = (bits[jp * words_per_set + (s >> 5)] >> (s & 31u)) & 1u;
        lnk[e] = l;
    }
}

template <int SB, int P>
__global__ void __launch_bounds__(544, 1)
    k_chain_grid_link(const __grid_constant__ CUtensorMap tmap, StepArgs a, const uint32_t *lnk, GridLinkShape gs) {
    constexpr uint32_t NV = SB / 16;
    constexpr uint32_t RPI = 32u / NV;
    const TmaShape sh = gs.t;
    extern __shared__ uint8_t dsm_raw[];
    __shared__ __align__(8) uint64_t bar[2];
    __shared__ uint32_t warp_odd[17];
    __shared__ uint32_t s_sel, s_rej;
    __shared__ uint32_t s_upd[17];  // per member warp: which lanes transitioned this step
    __shared__ uint32_t s_ab[2];  // [0]: raised in region A, read after its barrier; [1]: region B
    // layout: [pay 0][pay 1][out 0|1][idx 0|1][lnk 0|1][tables][records 0|1][effects 0|1]
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    uint32_t *const words = reinterpret_cast<uint32_t *>(base + 2 * sh.stage_pay);
    uint8_t *const tab = reinterpret_cast<uint8_t *>(words + 6 * sh.stage_words);
    uint4 *const recs = reinterpret_cast<uint4 *>(tab + ((2 * a.tab_stride + 15u) & ~15u));
    uint4 *const effs = recs + 2ull * sh.chunk * NV;
    auto pay_of = [&](uint32_t st) { return base + st * sh.stage_pay; };
    auto out_of = [&](uint32_t st) { return words + st * sh.stage_words; };
    auto idx_of = [&](uint32_t st) { return words + (2u + st) * sh.stage_words; };
    auto lnk_of = [&](uint32_t st) { return words + (4u + st) * sh.stage_words; };
    auto rec_of = [&](uint32_t st) { return recs + static_cast<size_t>(st) * sh.chunk * NV; };
    auto eff_of = [&](uint32_t st) { return effs + static_cast<size_t>(st) * sh.chunk; };

    const uint32_t tid = threadIdx.x;
    const bool ctl = tid == gs.members;
    const bool member = tid < gs.members;
    const uint32_t lane = tid & 31u, wbase = tid & ~31u;
    const uint32_t G = gridDim.x;
    const uint32_t m0 = blockIdx.x * sh.chunk;
    const uint32_t cnt = m0 < a.K ? min(sh.chunk, a.K - m0) : 0u;
    const uint32_t nst = a.n_steps;
    const uint64_t limit = a.dev->wait_ns;
    const uint64_t stream_pol = policy_evict_first();
    const uint64_t keep_pol = policy_evict_last();
    // profiling: the control thread and member thread 0 of the first and last CTA
    long long *trace = nullptr;
    if (a.trace && (tid == 0 || ctl) && (blockIdx.x == 0 || blockIdx.x == G - 1))
        trace = a.trace + (blockIdx.x == 0 ? 0 : static_cast<size_t>(nst) * 8) + (ctl ? 0 : 4);

    uint32_t issued = 0;  // control thread: steps [0, issued) have had their events issued
    auto issue = [&](uint32_t j) {  // control thread: events of step j into stage j & 1
        issued = j + 1u;
        const uint32_t st = j & 1u;
        const uint32_t row0 = (j % a.n_sets) * a.K + m0;
        mbar_arrive_expect_tx(&bar[st], sh.n_boxes * sh.box_rows * P + cnt * 12u);
        for (uint32_t b = 0; b < sh.n_boxes; ++b)
            tma_load_2d_hint(pay_of(st) + b * sh.box_rows * P, &tmap, 0,
                             static_cast<int32_t>(row0 + b * sh.box_rows), &bar[st], stream_pol);
        bulk_load_hint(out_of(st), a.outcome + row0, cnt * 4u, &bar[st], stream_pol);
        bulk_load_hint(idx_of(st), a.idx + row0, cnt * 4u, &bar[st], stream_pol);
        bulk_load_hint(lnk_of(st), lnk + row0, cnt * 4u, &bar[st], stream_pol);
    };
    auto linked = [&](uint32_t j, uint32_t t) { return j > 0u && lnk_of(j & 1u)[t] != 0u; };
    // member warps: gather the records of step j's members of this warp whose
    // linked flag equals want, NV lanes per record
    auto gather = [&](uint32_t j, bool want) {
        const uint32_t st = j & 1u;
        const uint32_t c = lane % NV;
#pragma unroll
        for (uint32_t k = 0; k < NV; ++k) {
            const uint32_t t = wbase + k * RPI + lane / NV;
            if (t < cnt && linked(j, t) == want) {
                const uint32_t s = idx_of(st)[t];
                if (s < a.n_sessions)
                    cp_async16(rec_of(st) + pay_chunk<SB>(t, c),
                               reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s) * SB) + c);
            }
        }
        cp_async_commit();
        cp_async_wait<0>();
        __syncwarp();
    };
    // this thread's member of step j (when its linked flag equals want): route key
    uint64_t rk = 0;
    uint32_t ok = 0, odd = 0;
    auto key = [&](uint32_t j, bool want) {
        if (tid >= cnt || linked(j, tid) != want) return;
        const uint32_t st = j & 1u;
        const uint32_t s = idx_of(st)[tid], o = out_of(st)[tid];
        ok = 0;
        odd = 0;
        if (s >= a.n_sessions) {
            latch_error(a.dev, DEV_E_INDEX, j, m0 + tid);
            return;
        }
        const uint32_t x = rec_of(st)[pay_chunk<SB>(tid, 0)].x;
        if (x >= a.S || o >= 8u) {
            latch_error(a.dev, DEV_E_STATE, j, m0 + tid);
            return;
        }
        uint4 pw[P / 16];
        read_payload_swizzled<P>(pw, pay_of(st), tid);
        rk = route_key<P>(x, o, pw);
        odd = static_cast<uint32_t>(rk & 1u);
        ok = 1;
    };

    if (ctl) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        fence_mbar_init();
        s_sel = ld_volatile_u32(&a.dev->sel) & 1u;
        s_ab[0] = 0;
        s_ab[1] = 0;
        s_rej = 0;
    }
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    __syncthreads();
    if (ctl && cnt > 0) {
        if (nst > 0) issue(0);
        if (nst > 1) issue(1);
    }
    uint32_t sel = s_sel;
    // prologue: step 0 (all members unlinked) gathered and hashed
    if (member && cnt > 0 && nst > 0) {
        if (!mbar_wait_bounded(&bar[0], 0u, limit)) {
            latch_error(a.dev, DEV_E_TIMEOUT, 0, blockIdx.x);
            s_ab[1] = 1;
        } else {
            gather(0, false);
            key(0, false);
        }
    }
    __syncthreads();
    const bool started = s_ab[1] == 0u;
    uint32_t n = 0;
    for (; started && n < nst; ++n) {
        const uint32_t st = n & 1u;
        // ---- region A(n): linked members, transition, stores ----
        if (member) {
            if (trace) trace[n * 8 + 0] = clock64();
            if (n > 0) {
                gather(n, true);
                key(n, true);
            }
            if (trace) trace[n * 8 + 1] = clock64();
            uint32_t v = (tid < cnt && ok) ? odd : 0u;
#pragma unroll
            for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
            if (lane == 0) warp_odd[tid >> 5] = v;
            uint32_t upd = 0;
            if (tid < cnt && ok) {
                const uint32_t s = idx_of(st)[tid], o = out_of(st)[tid];
                uint4 r[NV];
#pragma unroll
                for (uint32_t k = 0; k < NV; ++k) r[k] = rec_of(st)[pay_chunk<SB>(tid, k)];
                const uint32_t y = tab[sel * a.tab_stride + r[0].x * 8u + o];
                r[0].x = y;
                r[0].y = r[0].y + 1u;
                mix_acc<SB>(r, rk);
#pragma unroll
                for (uint32_t k = 0; k < NV; ++k) rec_of(st)[pay_chunk<SB>(tid, k)] = r[k];
                uint4 e;
                e.x = static_cast<uint32_t>(rk);
                e.y = static_cast<uint32_t>(rk >> 32);
                e.z = s;
                e.w = y | (o << 16) | (sel << 24);
                eff_of(st)[tid] = e;
                if (a.state_log) {
                    uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + (static_cast<size_t>(n) * a.K + m0 + tid) * SB);
#pragma unroll
                    for (uint32_t k = 0; k < NV; ++k) __stcs(lp + k, r[k]);
                }
                upd = 1;
            } else if (tid < cnt) {
                s_rej = 1;  // a rejected member: this step's effects go out one by one
            }
            fence_proxy_async_smem();  // the staged effects are read by the bulk copy
            const uint32_t umask = __ballot_sync(0xffffffffu, upd);
            if (lane == 0) s_upd[tid >> 5] = umask;
            __syncwarp();
            const uint32_t c = lane % NV;
#pragma unroll
            for (uint32_t k = 0; k < NV; ++k) {
                const uint32_t q = k * RPI + lane / NV;
                if ((umask >> q) & 1u) {
                    const uint32_t t = wbase + q;
                    const uint32_t s = idx_of(st)[t];
                    st_hint(reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s) * SB) + c,
                            rec_of(st)[pay_chunk<SB>(t, c)], keep_pol);
                }
            }
            ok = 0;
            if (trace) trace[n * 8 + 2] = clock64();
        }
        __syncthreads();  // region A done: stores issued, counts and effects staged
        if (s_ab[0] != 0u) break;
        // ---- region B(n): control thread publishes and waits; members run ahead ----
        if (ctl) {
            if (trace) trace[n * 8 + 0] = clock64();
            uint32_t c = 0;
            for (uint32_t w = 0; w < gs.members / 32u; ++w) c += warp_odd[w];
            unsigned long long *word = &a.dev->slot[n % 3u];
            if (blockIdx.x == 0) a.dev->slot[(n + 1u) % 3u] = 0ull;
            const bool skip = (n == 0 && blockIdx.x == 1 && ld_volatile_u32(&a.dev->skip_arrival) != 0u);
            if (!skip) red_release_add_u64(word, (1ull << 32) | c);
            if (trace) trace[n * 8 + 1] = clock64();
            if (a.effects && cnt > 0) {
                if (s_rej == 0u) {
                    bulk_store(reinterpret_cast<uint4 *>(a.effects) + static_cast<size_t>(n) * a.K + m0, eff_of(st),
                               cnt * 16u);
                } else {
                    // error path: only the transitioned members' effects
                    for (uint32_t t = 0; t < cnt; ++t)
                        if ((s_upd[t >> 5] >> (t & 31u)) & 1u)
                            reinterpret_cast<uint4 *>(a.effects)[static_cast<size_t>(n) * a.K + m0 + t] = eff_of(st)[t];
                    s_rej = 0;
                }
                bulk_commit();
                bulk_wait_read<1>();  // the staging buffer of step n - 1 is free again
            }
            if (cnt > 0 && n + 2u < nst) {
                fence_proxy_async_smem();
                issue(n + 2u);
            }
            if (trace) trace[n * 8 + 2] = clock64();
            uint64_t t0 = 0;
            unsigned long long w;
            uint32_t spins = 0;
            for (;;) {
                w = ld_acquire_u64(word);
                if ((w >> 32) >= G) break;
                if ((++spins & 63u) == 0u) {
                    if (ld_volatile_u32(&a.dev->abort) != 0u) {
                        s_ab[1] = 1;
                        break;
                    }
                    if (timed_out(t0, limit)) {
                        latch_error(a.dev, DEV_E_TIMEOUT, n, blockIdx.x);
                        atomicExch(&a.dev->abort, 1u);
                        s_ab[1] = 1;
                        break;
                    }
                }
            }
            const uint32_t d = (static_cast<uint32_t>(w & 0xffffffffull) > a.K / 2u) ? 1u : 0u;
            s_sel = d;
            if (blockIdx.x == 0 && a.decisions && s_ab[1] == 0u) a.decisions[n] = d;
            if (trace) trace[n * 8 + 3] = clock64();
        } else if (member && cnt > 0 && n + 1u < nst) {
            if (!mbar_wait_bounded(&bar[(n + 1u) & 1u], ((n + 1u) >> 1) & 1u, limit)) {
                latch_error(a.dev, DEV_E_TIMEOUT, n + 1u, blockIdx.x);
                s_ab[1] = 1;
            } else {
                gather(n + 1u, false);
                key(n + 1u, false);
            }
            if (trace) trace[n * 8 + 3] = clock64();
        }
        __syncthreads();  // region B done: decision of step n known, step n + 1 run ahead
        if (s_ab[1] != 0u) break;
        sel = s_sel;
    }
    cp_async_wait<0>();
    if (ctl) {
        bulk_wait_all<0>();
        if (n < nst) {
            // stopped early: wait (bounded) for the event copies still in flight
            for (uint32_t j = n; j < issued; ++j) (void)mbar_wait_bounded(&bar[j & 1u], (j >> 1) & 1u, limit);
        } else if (blockIdx.x == 0 && nst > 0) {
            a.dev->sel = sel;
            a.dev->step = nst;
        }
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, cooperative grid, two steps per grid barrier (explicit
// session indices, K a multiple of 8 and at most 65,536; one CTA per SM, CTA
// b owns the members [b*chunk, b*chunk + cnt) of every step).
//
// The route key of step j needs the decisions only up to d(j - 2): the state
// a session enters step j with is T_sel(i)[x_i][o_i] for its last step i < j,
// and sel(i) = d(i - 1).  So region r, which starts once the barrier has
// published d(2r - 2) and d(2r - 1), keys steps 2r and 2r + 1 together, and
// its barrier publishes both odd counts; the records of those two steps are
// completed (their transitions need d(2r - 1) and d(2r)) in region r + 1.
//
// The link pass (k_mark_pos, k_link_grid2) gives each member the nearest of
// the three earlier cohorts holding its session (distance t, position q), a
// forward bit (its session is in the next cohort) and, for t = 1, the same
// link one level further back.  Every member writes its input state and
// outcome to the ring `xo` (four steps) and, on even steps, its key to the
// ring `keyring` (two even steps); other CTAs read them after the barrier.
//  * x of an even step 2r: t in {1, 2} -> T_sel(i)[x_i][o_i] from xo, i =
//    2r - t (keyed in region r - 1); otherwise the state array (the session's
//    last step is at most 2r - 3, completed in region r - 1 at the latest).
//  * x of an odd step 2r + 1: t in {2, 3} the same way; t = 1 (the session is
//    in step 2r, keyed in this region by its owner) -> x of step 2r from the
//    second link, then T_d(2r - 1)[x][outcome of step 2r]; otherwise the
//    state array.
//  * completing steps 2r - 2 and 2r - 1 in region r: a member of the even
//    step whose session is in the odd one neither gathers nor stores: the
//    odd step's member gathers the record, applies both steps (the first
//    with the key from the ring) and stores once, writing both log rows.
//    No other CTA touches that session's record in the region.
// Region r, member threads: A1 gather the records of steps 2r - 2 and
// 2r - 1 (warp-cooperatively), load x of steps 2r and 2r + 1 and the words
// of steps 2r + 2 and 2r + 3; A3 complete, store and emit steps 2r - 2 and
// 2r - 1; A2 wait for the payload tiles, key steps 2r and 2r + 1, write the
// rings, count.  Then the control thread adds (1 << 48 | odd(2r + 1) << 24 |
// odd(2r)) to the barrier word with release semantics, issues the payload
// tiles of steps 2r + 3 and 2r + 4 (three tile stages) and spins.  Every
// wait is bounded; a CTA that gives up latches RC_E_TIMEOUT, raises
// dev->abort and leaves after the next block barrier, the control thread
// first waiting (bounded) for its tile copies in flight.
// ---------------------------------------------------------------------------
struct GridPairShape {
    TmaShape t;        // chunk, payload tiles, stage size (stage_words unused)
    uint32_t members;  // member threads (a multiple of 32, >= chunk); the control warp follows
    uint32_t pad[3];
};
constexpr uint32_t kGridPairStages = 3;  // payload tile stages
constexpr uint32_t kGridPairThreads = 480;

// bits[j] marks cohort j's sessions, pos[j][s] = the position of session s
// in cohort j (read only where the bit is set; the caller clears the bits).
__global__ void k_mark_pos(const uint32_t *idx, uint32_t n_sets, uint32_t K, uint64_t N, uint64_t words_per_set,
                           uint32_t *bits, uint16_t *pos) {
    const size_t total = static_cast<size_t>(n_sets) * K;
    for (size_t e = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const uint32_t s = idx[e];
        if (s >= N) continue;
        const size_t j = e / K;
        atomicOr(bits + j * words_per_set + (s >> 5), 1u << (s & 31u));
        pos[j * N + s] = static_cast<uint16_t>(e - j * K);
    }
}

// lnk2[j][m] = {a, b}: a = fwd << 31 | t << 16 | q, the nearest cohort j - t
// (t = 1..3, mod n_sets) holding member m's session at position q (t = 0:
// none), fwd = the session is in cohort j + 1; for t = 1, b = t' << 16 | q',
// the nearest of cohorts j - 2, j - 3 holding it, t' counted from j - 1.
__global__ void k_link_grid2(const uint32_t *idx, uint32_t n_sets, uint32_t K, uint64_t N, uint64_t words_per_set,
                             const uint32_t *bits, const uint16_t *pos, uint2 *lnk2) {
    const size_t total = static_cast<size_t>(n_sets) * K;
    for (size_t e = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < total;
         e += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const uint32_t s = idx[e];
        const uint64_t j = e / K;
        uint2 w = make_uint2(0u, 0u);
        if (s < N) {
            auto back = [&](uint32_t t) { return (j + 3ull * n_sets - t) % n_sets; };
            auto has = [&](uint64_t jj) { return ((bits[jj * words_per_set + (s >> 5)] >> (s & 31u)) & 1u) != 0u; };
            auto at = [&](uint64_t jj) { return static_cast<uint32_t>(pos[jj * N + s]); };
            for (uint32_t t = 1; t <= 3u; ++t) {
                if (has(back(t))) {
                    w.x = (t << 16) | at(back(t));
                    break;
                }
            }
            if (((w.x >> 16) & 3u) == 1u) {
                for (uint32_t t = 2; t <= 3u; ++t) {
                    if (has(back(t))) {
                        w.y = ((t - 1u) << 16) | at(back(t));
                        break;
                    }
                }
            }
            if (has((j + 1u) % n_sets)) w.x |= 1u << 31;
        }
        lnk2[e] = w;
    }
}

template <int SB, int P>
__global__ void __launch_bounds__(kGridPairThreads, 1)
    k_chain_grid_pair(const __grid_constant__ CUtensorMap tmap, StepArgs a, const uint2 *lnk, uint32_t *xo,
                      unsigned long long *keyring, GridPairShape gs) {
    constexpr uint32_t NV = SB / 16;
    constexpr uint32_t RPI = 32u / NV;
    constexpr uint32_t NS = kGridPairStages;
    constexpr uint32_t kSkip = 0, kRejected = 1, kApplied = 2;
    const TmaShape sh = gs.t;
    extern __shared__ uint8_t dsm_raw[];
    __shared__ __align__(8) uint64_t pbar[NS];
    __shared__ uint32_t warp_odd[2][16];
    __shared__ uint32_t s_dec[4];  // d(i) at i & 3
    __shared__ uint32_t s_sel0;
    __shared__ uint32_t s_ab[2];  // [0]: raised before S1, read after it; [1]: raised in the spin, read after S2
    // layout: [payload stage 0 | 1 | 2][records of the two completed steps][tables]
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    uint4 *const recs = reinterpret_cast<uint4 *>(base + NS * sh.stage_pay);
    uint8_t *const tab = reinterpret_cast<uint8_t *>(recs + 2ull * sh.chunk * NV);
    auto pay_of = [&](uint32_t j) { return base + (j % NS) * sh.stage_pay; };
    auto rec_of = [&](uint32_t i) { return recs + static_cast<size_t>(i) * sh.chunk * NV; };

    const uint32_t tid = threadIdx.x;
    const bool ctl = tid == gs.members;
    const bool member = tid < gs.members;
    const uint32_t lane = tid & 31u, wbase = tid & ~31u;
    const uint32_t G = gridDim.x;
    const uint32_t K = a.K;
    const uint32_t m0 = blockIdx.x * sh.chunk;
    const uint32_t cnt = m0 < K ? min(sh.chunk, K - m0) : 0u;
    const bool mine = tid < cnt;  // this thread owns member p of every step
    const uint32_t p = m0 + tid;
    const uint32_t nst = a.n_steps;
    const uint32_t S = a.S, stride = a.tab_stride;
    const uint64_t N = a.n_sessions;
    const uint64_t limit = a.dev->wait_ns;
    const uint64_t stream_pol = policy_evict_first();
    const uint64_t keep_pol = policy_evict_last();
    long long *trace = nullptr;
    if (a.trace && (tid == 0 || ctl) && (blockIdx.x == 0 || blockIdx.x == G - 1))
        trace = a.trace + (blockIdx.x == 0 ? 0 : static_cast<size_t>(nst) * 8) + (ctl ? 0 : 4);

    uint32_t issued = 0;  // control thread: the tiles of steps [0, issued) have been issued
    auto issue = [&](uint32_t j) {
        if (j >= nst || cnt == 0u) return;
        issued = j + 1u;
        uint64_t *b = &pbar[j % NS];
        const uint32_t row0 = (j % a.n_sets) * K + m0;
        mbar_arrive_expect_tx(b, sh.n_boxes * sh.box_rows * P);
        for (uint32_t k = 0; k < sh.n_boxes; ++k)
            tma_load_2d_hint(pay_of(j) + k * sh.box_rows * P, &tmap, 0, static_cast<int32_t>(row0 + k * sh.box_rows),
                             b, stream_pol);
    };
    // the route body of step j: d(j - 1), d(-1) being the flag the chain starts from
    auto sel_of = [&](uint32_t j) -> uint32_t { return j == 0u ? s_sel0 : s_dec[(j - 1u) & 3u]; };
    auto body = [&](uint32_t j, uint32_t x, uint32_t o) -> uint32_t {
        return (x < S && o < 8u) ? static_cast<uint32_t>(tab[sel_of(j) * stride + x * 8u + o]) : x;
    };

    if (ctl) {
        for (uint32_t i = 0; i < NS; ++i) mbar_init(&pbar[i], 1);
        fence_mbar_init();
        s_sel0 = ld_volatile_u32(&a.dev->sel) & 1u;
        for (uint32_t i = 0; i < 4u; ++i) s_dec[i] = 0;
        s_ab[0] = 0;
        s_ab[1] = 0;
        for (uint32_t j = 0; j < NS; ++j) issue(j);
    }
    stage_tables(tab, a.tables, stride, 2, 0);

    // words of this region's key steps (c*) and of the next region's (n*)
    uint32_t co0 = 0, co1 = 0, cs0 = 0, cs1 = 0;
    uint2 cl0 = make_uint2(0u, 0u), cl1 = make_uint2(0u, 0u);
    uint32_t no0 = 0, no1 = 0, ns0 = 0, ns1 = 0;
    uint2 nl0 = make_uint2(0u, 0u), nl1 = make_uint2(0u, 0u);
    auto load_words = [&](uint32_t j, uint32_t &o, uint32_t &s, uint2 &l) {
        if (mine && j < nst) {
            const size_t e = static_cast<size_t>(j % a.n_sets) * K + p;
            o = __ldcs(a.outcome + e);
            s = __ldcs(a.idx + e);
            l = __ldcs(lnk + e);
        }
    };
    if (member) {
        load_words(0, co0, cs0, cl0);
        load_words(1, co1, cs1, cl1);
    }
    // carried from the key steps to their completion a region later
    uint32_t ks0 = 0, ks1 = 0, ko0 = 0, ko1 = 0, kx0 = 0, kx1 = 0, kf0 = kSkip, kf1 = kSkip, kl0 = 0, kl1 = 0;
    uint64_t krk0 = 0, krk1 = 0;
    __syncthreads();

    const uint32_t R = (nst + 1u) / 2u;  // key regions; region R only completes
    uint32_t r = 0;
    for (; r <= R; ++r) {
        const uint32_t k0 = 2u * r, k1 = k0 + 1u;
        const bool has_keys = k0 < nst;
        long long *const tr = has_keys ? trace : nullptr;
        if (member) {
            if (tr) tr[k0 * 8 + 0] = clock64();
            // ---- A1: gathers of the completed steps, loads of the key steps' x ----
            const uint32_t c0 = k0 - 2u, c1 = k0 - 1u;  // valid when r > 0 (and < nst)
            const bool done0 = r > 0 && c0 < nst, done1 = r > 0 && c1 < nst;
            const bool fwd0 = (kl0 >> 31) != 0u && done1;     // the session goes on in step c1
            const bool need0 = done0 && kf0 == kApplied && !fwd0;
            const bool lnk1 = done1 && ((kl1 >> 16) & 3u) == 1u;  // in step c0 at position q1
            const bool need1 = done1 && kf1 != kSkip && (kf1 == kApplied || lnk1);
            uint64_t keyq = 0;
            uint32_t oq = 8;
            if (mine && need1 && lnk1) {
                const uint32_t q1 = kl1 & 0xFFFFu;
                keyq = __ldcg(keyring + static_cast<size_t>((c0 >> 1) & 1u) * K + q1);
                oq = min(__ldg(a.outcome + static_cast<size_t>(c0 % a.n_sets) * K + q1), 8u);
            }
            {
                const uint32_t c = lane % NV;
                const uint32_t m_need0 = __ballot_sync(0xffffffffu, mine && need0);
                const uint32_t m_need1 = __ballot_sync(0xffffffffu, mine && need1);
#pragma unroll
                for (uint32_t k = 0; k < NV; ++k) {
                    const uint32_t q = k * RPI + lane / NV;
                    const uint32_t s0 = __shfl_sync(0xffffffffu, ks0, q);
                    const uint32_t s1 = __shfl_sync(0xffffffffu, ks1, q);
                    if ((m_need0 >> q) & 1u)
                        cp_async16(rec_of(0) + pay_chunk<SB>(wbase + q, c),
                                   reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s0) * SB) + c);
                    if ((m_need1 >> q) & 1u)
                        cp_async16(rec_of(1) + pay_chunk<SB>(wbase + q, c),
                                   reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s1) * SB) + c);
                }
                cp_async_commit();
            }
            // x sources of the key steps: a ring entry (packed x | o << 16,
            // to pass through the body of its step) or the state array
            const bool key0 = mine && has_keys, key1 = mine && k1 < nst;
            const bool sv0 = key0 && cs0 < N, sv1 = key1 && cs1 < N;
            uint32_t v0 = 0, v1 = 0, oe = 8, i0 = 0, i1 = 0;
            bool ring0 = false, ring1 = false, chase1 = false;
            if (sv0) {
                const uint32_t t = (cl0.x >> 16) & 3u, q = cl0.x & 0xFFFFu;
                if (t >= 1u && t <= 2u && t <= k0) {
                    ring0 = true;
                    i0 = k0 - t;
                    v0 = __ldcg(xo + static_cast<size_t>(i0 & 3u) * K + q);
                } else {
                    v0 = __ldcg(reinterpret_cast<const uint32_t *>(a.state + static_cast<size_t>(cs0) * SB));
                }
            }
            if (sv1) {
                const uint32_t t = (cl1.x >> 16) & 3u, q = cl1.x & 0xFFFFu;
                if (t == 1u) {
                    chase1 = true;  // x of step k0 for this session, then step k0's body
                    oe = min(__ldg(a.outcome + static_cast<size_t>(k0 % a.n_sets) * K + q), 8u);
                    const uint32_t t2 = (cl1.y >> 16) & 3u, q2 = cl1.y & 0xFFFFu;
                    if (t2 >= 1u && t2 <= 2u && t2 <= k0) {
                        ring1 = true;
                        i1 = k0 - t2;
                        v1 = __ldcg(xo + static_cast<size_t>(i1 & 3u) * K + q2);
                    } else {
                        v1 = __ldcg(reinterpret_cast<const uint32_t *>(a.state + static_cast<size_t>(cs1) * SB));
                    }
                } else if (t >= 2u && t <= k1) {
                    ring1 = true;
                    i1 = k1 - t;
                    v1 = __ldcg(xo + static_cast<size_t>(i1 & 3u) * K + q);
                } else {
                    v1 = __ldcg(reinterpret_cast<const uint32_t *>(a.state + static_cast<size_t>(cs1) * SB));
                }
            }
            load_words(k0 + 2u, no0, ns0, nl0);
            load_words(k1 + 2u, no1, ns1, nl1);
            if (tr) tr[k0 * 8 + 1] = clock64();

            // ---- A3: complete, store and emit steps c0 and c1 ----
            cp_async_wait<0>();
            __syncwarp();
            bool st0 = false, st1 = false;
            if (mine && done0 && kf0 == kApplied) {
                const uint32_t sel = sel_of(c0);
                const uint32_t y = tab[sel * stride + kx0 * 8u + ko0];
                if (need0) {
                    uint4 rr[NV];
#pragma unroll
                    for (uint32_t k = 0; k < NV; ++k) rr[k] = rec_of(0)[pay_chunk<SB>(tid, k)];
                    rr[0].x = y;
                    rr[0].y = rr[0].y + 1u;
                    mix_acc<SB>(rr, krk0);
#pragma unroll
                    for (uint32_t k = 0; k < NV; ++k) rec_of(0)[pay_chunk<SB>(tid, k)] = rr[k];
                    if (a.state_log) {
                        uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + (static_cast<size_t>(c0) * K + p) * SB);
#pragma unroll
                        for (uint32_t k = 0; k < NV; ++k) __stcs(lp + k, rr[k]);
                    }
                    st0 = true;
                }
                if (a.effects) {
                    uint4 e;
                    e.x = static_cast<uint32_t>(krk0);
                    e.y = static_cast<uint32_t>(krk0 >> 32);
                    e.z = ks0;
                    e.w = y | (ko0 << 16) | (sel << 24);
                    __stcs(reinterpret_cast<uint4 *>(a.effects) + static_cast<size_t>(c0) * K + p, e);
                }
            }
            if (mine && need1) {
                uint4 rr[NV];
#pragma unroll
                for (uint32_t k = 0; k < NV; ++k) rr[k] = rec_of(1)[pay_chunk<SB>(tid, k)];
                if (lnk1 && rr[0].x < S && oq < 8u) {
                    // step c0 of this session, whose member left the record to this one
                    rr[0].x = tab[sel_of(c0) * stride + rr[0].x * 8u + oq];
                    rr[0].y = rr[0].y + 1u;
                    mix_acc<SB>(rr, keyq);
                    if (a.state_log) {
                        uint4 *lp = reinterpret_cast<uint4 *>(a.state_log +
                                                              (static_cast<size_t>(c0) * K + (kl1 & 0xFFFFu)) * SB);
#pragma unroll
                        for (uint32_t k = 0; k < NV; ++k) __stcs(lp + k, rr[k]);
                    }
                    st1 = true;
                }
                if (kf1 == kApplied) {
                    const uint32_t sel = sel_of(c1);
                    const uint32_t y = tab[sel * stride + kx1 * 8u + ko1];
                    rr[0].x = y;
                    rr[0].y = rr[0].y + 1u;
                    mix_acc<SB>(rr, krk1);
                    if (a.state_log) {
                        uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + (static_cast<size_t>(c1) * K + p) * SB);
#pragma unroll
                        for (uint32_t k = 0; k < NV; ++k) __stcs(lp + k, rr[k]);
                    }
                    if (a.effects) {
                        uint4 e;
                        e.x = static_cast<uint32_t>(krk1);
                        e.y = static_cast<uint32_t>(krk1 >> 32);
                        e.z = ks1;
                        e.w = y | (ko1 << 16) | (sel << 24);
                        __stcs(reinterpret_cast<uint4 *>(a.effects) + static_cast<size_t>(c1) * K + p, e);
                    }
                    st1 = true;
                }
                if (st1) {
#pragma unroll
                    for (uint32_t k = 0; k < NV; ++k) rec_of(1)[pay_chunk<SB>(tid, k)] = rr[k];
                }
            }
            {
                const uint32_t m_st0 = __ballot_sync(0xffffffffu, st0);
                const uint32_t m_st1 = __ballot_sync(0xffffffffu, st1);
                __syncwarp();
                const uint32_t c = lane % NV;
#pragma unroll
                for (uint32_t k = 0; k < NV; ++k) {
                    const uint32_t q = k * RPI + lane / NV;
                    const uint32_t s0 = __shfl_sync(0xffffffffu, ks0, q);
                    const uint32_t s1 = __shfl_sync(0xffffffffu, ks1, q);
                    if ((m_st0 >> q) & 1u)
                        st_hint(reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s0) * SB) + c,
                                rec_of(0)[pay_chunk<SB>(wbase + q, c)], keep_pol);
                    if ((m_st1 >> q) & 1u)
                        st_hint(reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s1) * SB) + c,
                                rec_of(1)[pay_chunk<SB>(wbase + q, c)], keep_pol);
                }
            }
            if (tr) tr[k0 * 8 + 2] = clock64();

            // ---- A2: key steps k0 and k1 ----
            uint32_t odd0 = 0, odd1 = 0;
            if (has_keys && cnt > 0u) {
                bool landed = mbar_wait_bounded(&pbar[k0 % NS], (k0 / NS) & 1u, limit);
                if (k1 < nst) landed = landed && mbar_wait_bounded(&pbar[k1 % NS], (k1 / NS) & 1u, limit);
                if (!landed) {
                    if (tid == 0) latch_error(a.dev, DEV_E_TIMEOUT, k0, blockIdx.x);
                    s_ab[0] = 1;
                } else {
                    const uint32_t x0 = ring0 ? body(i0, v0 & 0xFFFFu, v0 >> 16) : v0;
                    uint32_t x1 = ring1 ? body(i1, v1 & 0xFFFFu, v1 >> 16) : v1;
                    // a bad state carried from step k0 is latched by that step's member
                    const bool inherited = chase1 && x1 >= S;
                    if (chase1) x1 = body(k0, x1, oe);
                    const bool ok0 = sv0 && x0 < S && co0 < 8u, ok1 = sv1 && x1 < S && co1 < 8u;
                    if (key0 && !ok0) latch_error(a.dev, sv0 ? DEV_E_STATE : DEV_E_INDEX, k0, p);
                    if (key1 && !ok1 && !inherited) latch_error(a.dev, sv1 ? DEV_E_STATE : DEV_E_INDEX, k1, p);
                    uint4 pa[P / 16], pb[P / 16];
                    if (key0) {
                        read_payload_swizzled<P>(pa, pay_of(k0), tid);
                    } else {
#pragma unroll
                        for (int k = 0; k < P / 16; ++k) pa[k] = make_uint4(0u, 0u, 0u, 0u);
                    }
                    if (key1) {
                        read_payload_swizzled<P>(pb, pay_of(k1), tid);
                    } else {
#pragma unroll
                        for (int k = 0; k < P / 16; ++k) pb[k] = make_uint4(0u, 0u, 0u, 0u);
                    }
                    uint64_t rk0 = 0, rk1 = 0;
                    route_key_pair<P>(ok0 ? x0 : 0u, ok0 ? co0 : 0u, pa, ok1 ? x1 : 0u, ok1 ? co1 : 0u, pb, rk0, rk1);
                    odd0 = ok0 ? static_cast<uint32_t>(rk0 & 1u) : 0u;
                    odd1 = ok1 ? static_cast<uint32_t>(rk1 & 1u) : 0u;
                    if (key0) {
                        __stcg(xo + static_cast<size_t>(k0 & 3u) * K + p, min(x0, 0xFFFFu) | (min(co0, 8u) << 16));
                        __stcg(keyring + static_cast<size_t>((k0 >> 1) & 1u) * K + p,
                               static_cast<unsigned long long>(rk0));
                    }
                    if (key1) __stcg(xo + static_cast<size_t>(k1 & 3u) * K + p, min(x1, 0xFFFFu) | (min(co1, 8u) << 16));
                    ks0 = cs0;
                    ko0 = co0;
                    kx0 = x0;
                    krk0 = rk0;
                    kl0 = cl0.x;
                    kf0 = !key0 ? kSkip : (!sv0 ? kSkip : (ok0 ? kApplied : kRejected));
                    ks1 = cs1;
                    ko1 = co1;
                    kx1 = x1;
                    krk1 = rk1;
                    kl1 = cl1.x;
                    kf1 = !key1 ? kSkip : (!sv1 ? kSkip : (ok1 ? kApplied : kRejected));
                }
            }
            const uint32_t w = tid >> 5;
            const uint32_t n0 = __popc(__ballot_sync(0xffffffffu, odd0 != 0u));
            const uint32_t n1 = __popc(__ballot_sync(0xffffffffu, odd1 != 0u));
            if (lane == 0) {
                warp_odd[0][w] = n0;
                warp_odd[1][w] = n1;
            }
            co0 = no0;
            cs0 = ns0;
            cl0 = nl0;
            co1 = no1;
            cs1 = ns1;
            cl1 = nl1;
            if (tr) tr[k0 * 8 + 3] = clock64();
        }
        __syncthreads();  // S1: records stored, rings written, counts staged, tiles read
        if (s_ab[0] != 0u || !has_keys) break;
        if (ctl) {
            if (tr) tr[k0 * 8 + 0] = clock64();
            uint32_t ce = 0, cd = 0;
            for (uint32_t w = 0; w < gs.members / 32u; ++w) {
                ce += warp_odd[0][w];
                cd += warp_odd[1][w];
            }
            unsigned long long *word = &a.dev->slot[r % 3u];
            if (blockIdx.x == 0) a.dev->slot[(r + 1u) % 3u] = 0ull;
            const bool skip = (r == 0 && blockIdx.x == 1 && ld_volatile_u32(&a.dev->skip_arrival) != 0u);
            if (!skip) red_release_add_u64(word, (1ull << 48) | (static_cast<unsigned long long>(cd) << 24) | ce);
            if (tr) tr[k0 * 8 + 1] = clock64();
            fence_proxy_async_smem();
            issue(k0 + 3u);
            issue(k1 + 3u);
            if (tr) tr[k0 * 8 + 2] = clock64();
            uint64_t t0 = 0;
            unsigned long long wv;
            uint32_t spins = 0;
            for (;;) {
                wv = ld_acquire_u64(word);
                if ((wv >> 48) >= G) break;
                if ((++spins & 63u) == 0u) {
                    if (ld_volatile_u32(&a.dev->abort) != 0u) {
                        s_ab[1] = 1;
                        break;
                    }
                    if (timed_out(t0, limit)) {
                        latch_error(a.dev, DEV_E_TIMEOUT, k0, blockIdx.x);
                        atomicExch(&a.dev->abort, 1u);
                        s_ab[1] = 1;
                        break;
                    }
                }
            }
            const uint32_t d0 = (static_cast<uint32_t>(wv & 0xFFFFFFull) > K / 2u) ? 1u : 0u;
            const uint32_t d1 = (static_cast<uint32_t>((wv >> 24) & 0xFFFFFFull) > K / 2u) ? 1u : 0u;
            s_dec[k0 & 3u] = d0;
            s_dec[k1 & 3u] = d1;
            if (blockIdx.x == 0 && a.decisions && s_ab[1] == 0u) {
                a.decisions[k0] = d0;
                if (k1 < nst) a.decisions[k1] = d1;
            }
            if (tr) tr[k0 * 8 + 3] = clock64();
        }
        __syncthreads();  // S2: d(k0), d(k1) known
        if (s_ab[1] != 0u) break;
    }
    cp_async_wait<0>();
    if (ctl) {
        if (r < R) {
            // stopped early: wait (bounded) for the tile copies still in flight
            for (uint32_t j = 2u * r; j < issued; ++j) (void)mbar_wait_bounded(&pbar[j % NS], (j / NS) & 1u, limit);
        } else if (blockIdx.x == 0 && nst > 0) {
            a.dev->sel = sel_of(nst);
            a.dev->step = nst;
        }
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, one thread-block cluster (512 < K <= 8,192): C <= 16 CTAs
// of up to 512 threads, member m = rank * blockDim.x + threadIdx.x.  The step
// barrier is the cluster's hardware barrier (arrive with release, wait with
// acquire, cluster scope), not a spin on a global word: each CTA leaves its
// odd count in its own shared memory, and after the barrier every warp sums
// the C counts through distributed shared memory.  Records are read at L2
// (another CTA of the cluster may have stored them the step before; the
// barrier's release / acquire orders those stores before these loads).
// Events of the next two steps are prefetched into registers, as in
// k_chain_cta.  The hardware barrier needs no bounded wait: the CTAs of a
// cluster are co-scheduled and every one reaches every barrier.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ uint32_t cluster_size() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
    return r;
}
__device__ __forceinline__ void cluster_barrier() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// 32-bit load of the same shared variable in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t ld_cluster_u32(const uint32_t *p, uint32_t rank) {
    uint32_t remote, v;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(remote) : "r"(smem_addr(p)), "r"(rank));
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(remote) : "memory");
    return v;
}

template <int SB, int P>
__global__ void __launch_bounds__(512) k_chain_cluster(StepArgs a) {
    __shared__ __align__(16) uint8_t tab[2 * 256 * 8];
    __shared__ uint32_t cnt[2];
    const uint32_t tid = threadIdx.x;
    const uint32_t rank = cluster_rank();
    const uint32_t C = cluster_size();
    const uint32_t m = rank * blockDim.x + tid;
    const bool active = m < a.K;
    const uint32_t lane = tid & 31u;
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    uint32_t sel = ld_volatile_u32(&a.dev->sel) & 1u;
    Event<P> ev0, ev1;
    if (active && a.n_steps > 0) load_event<P>(ev0, a, 0, m);
    if (active && a.n_steps > 1) load_event<P>(ev1, a, 1 % a.n_sets, m);
    cluster_barrier();  // every CTA's tables and counters are in place
    for (uint32_t n = 0; n < a.n_steps; ++n) {
        uint32_t odd = 0;
        if (active) {
            const Event<P> ev = ev0;
            ev0 = ev1;
            if (n + 2u < a.n_steps) load_event<P>(ev1, a, (n + 2u) % a.n_sets, m);
            odd = transition<SB, P, true>(a, ev, tab + sel * a.tab_stride, sel, n, m);
        }
        const uint32_t c = static_cast<uint32_t>(__syncthreads_count(odd));
        if (tid == 0) cnt[n & 1u] = c;
        cluster_barrier();  // this step's records and counts, cluster-wide
        const uint32_t v = lane < C ? ld_cluster_u32(&cnt[n & 1u], lane) : 0u;
        const uint32_t total = __reduce_add_sync(0xffffffffu, v);
        sel = total > a.K / 2u ? 1u : 0u;
        if (rank == 0 && tid == 0 && a.decisions) a.decisions[n] = sel;
    }
    cluster_barrier();  // no CTA leaves while another may still read its counters
    if (rank == 0 && tid == 0) {
        if (a.n_steps > 0) a.dev->sel = sel;
        a.dev->step = a.n_steps;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain, split-phase (explicit session indices, K a multiple of 8,
// at most 512 members per CTA; one CTA when K <= 512, else one CTA per SM).
//
// A member whose session is not in the previous cohort ("clean") does not
// depend on that cohort's writes: its record, route key, odd bit, step and
// accumulator can be computed one step early, while the previous step's
// barrier resolves; only its next state y = T_sel[x][o] must wait for the
// decision.  A member whose session is in the previous cohort ("dirty") is
// gathered and hashed after that step's barrier.  Membership is found with
// step-tagged marks in device scratch (three arrays, one per step mod 3; a
// cohort's marks are written before the barrier that precedes any check
// against them, and a CTA can run at most one barrier ahead, so a check never
// meets a rewrite).  Iteration n (n = -1 .. n_steps - 1):
//   A  finish the clean members of step n (table lookup, stores, effect);
//      write the marks of cohort n + 1;
//   B  gather, hash and finish the dirty members of step n (compacted list);
//   -- CTA sync; thread 0 arrives at the grid barrier with the odd count of
//      step n (the early count of its clean members + the dirty ones);
//   C  early work for the clean members of step n + 1 (mark check, gather,
//      route key, accumulator), overlapping the barrier wait;
//   -- CTA sync after the barrier: the decision of step n selects the body
//      of step n + 1.
// Events arrive by TMA as in k_chain_grid_tma.  All waits are bounded.
// ---------------------------------------------------------------------------
template <int SB, int P>
__global__ void __launch_bounds__(512, 1)
    k_chain_split(const __grid_constant__ CUtensorMap tmap, StepArgs a, TmaShape sh, uint32_t *marks) {
    constexpr int NV = SB / 16;
    extern __shared__ uint8_t dsm_raw[];
    __shared__ __align__(8) uint64_t bar[2];
    __shared__ uint32_t warp_odd[16];
    __shared__ uint16_t dlist[2][512];
    __shared__ uint32_t dcount[2];
    __shared__ uint32_t s_sel, s_abort, s_pending, s_pend_step[2];
    const uint32_t raw = smem_addr(dsm_raw);
    uint8_t *const base = dsm_raw + (((raw + 1023u) & ~1023u) - raw);
    uint32_t *const words = reinterpret_cast<uint32_t *>(base + 2 * sh.stage_pay);
    uint8_t *const tab = reinterpret_cast<uint8_t *>(words + 4 * sh.stage_words);
    auto pay_of = [&](uint32_t st) { return base + st * sh.stage_pay; };
    auto out_of = [&](uint32_t st) { return words + st * sh.stage_words; };
    auto idx_of = [&](uint32_t st) { return words + (2u + st) * sh.stage_words; };

    const uint32_t tid = threadIdx.x;
    const uint32_t m0 = blockIdx.x * sh.chunk;
    const uint32_t cnt = m0 < a.K ? min(sh.chunk, a.K - m0) : 0u;
    const bool mine = tid < cnt;
    const bool single = gridDim.x == 1;
    const uint64_t limit = a.dev->wait_ns;
    const uint64_t stream_pol = policy_evict_first();
    const uint64_t keep_pol = policy_evict_last();
    const uint32_t issuer = blockDim.x > 32u ? 32u : 0u;
    const uint64_t N = a.n_sessions;
    const int nst = static_cast<int>(a.n_steps);
    long long *trace = (a.trace && tid == 0 && (blockIdx.x == 0 || blockIdx.x == gridDim.x - 1))
                           ? a.trace + (blockIdx.x == 0 ? 0 : static_cast<size_t>(a.n_steps) * 8)
                           : nullptr;
    auto mark_time = [&](int n, int k) {
        if (trace && n >= 0) trace[static_cast<size_t>(n) * 8 + k] = clock64();
    };

    auto issue = [&](uint32_t j) {
        const uint32_t st = j & 1u;
        const uint32_t row0 = (j % a.n_sets) * a.K + m0;
        const uint32_t bytes = sh.n_boxes * sh.box_rows * P + cnt * 8u;
        mbar_arrive_expect_tx(&bar[st], bytes);
        for (uint32_t b = 0; b < sh.n_boxes; ++b)
            tma_load_2d_hint(pay_of(st) + b * sh.box_rows * P, &tmap, 0,
                             static_cast<int32_t>(row0 + b * sh.box_rows), &bar[st], stream_pol);
        bulk_load_hint(out_of(st), a.outcome + row0, cnt * 4u, &bar[st], stream_pol);
        bulk_load_hint(idx_of(st), a.idx + row0, cnt * 4u, &bar[st], stream_pol);
        s_pending |= 1u << st;
        s_pend_step[st] = j;
    };
    auto wait_stage = [&](uint32_t st, uint32_t parity) -> bool { return mbar_wait_bounded(&bar[st], parity, limit); };
    auto give_up = [&](uint32_t n) {
        latch_error(a.dev, DEV_E_TIMEOUT, n, blockIdx.x);
        atomicExch(&a.dev->abort, 1u);
        s_abort = 1;
    };

    if (tid == 0) {
        mbar_init(&bar[0], 1);
        mbar_init(&bar[1], 1);
        fence_mbar_init();
        s_sel = ld_volatile_u32(&a.dev->sel) & 1u;
        s_abort = 0;
        s_pending = 0;
        dcount[0] = dcount[1] = 0;
    }
    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    __syncthreads();
    if (tid == 0 && cnt > 0) {
        if (nst > 0) issue(0);
        if (nst > 1) issue(1);
    }
    uint32_t sel = s_sel;

    // this thread's member of the next step, prepared in phase C
    bool pv = false;           // clean and prepared
    uint32_t p_s = 0, p_o = 0, p_x = 0, p_odd = 0;
    uint64_t p_rk = 0;
    uint4 p_rec[NV];
    uint32_t nx_s = 0, nx_o = 0;  // session / outcome of the next step's member

    for (int n = -1; n < nst; ++n) {
        const uint32_t un = static_cast<uint32_t>(n);
        uint32_t odd = 0;
        mark_time(n, 0);
        // ---- A: finish the clean member of step n ----
        if (n >= 0 && mine && pv) {
            const uint32_t y = tab[sel * a.tab_stride + p_x * 8u + p_o];
            p_rec[0].x = y;
            uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(p_s) * SB);
#pragma unroll
            for (int k = 0; k < NV; ++k) st_hint(rp + k, p_rec[k], keep_pol);
            const size_t slot = static_cast<size_t>(un) * a.K + m0 + tid;
            if (a.effects) {
                uint4 e;
                e.x = static_cast<uint32_t>(p_rk);
                e.y = static_cast<uint32_t>(p_rk >> 32);
                e.z = p_s;
                e.w = y | (p_o << 16) | (sel << 24);
                __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
            }
            if (a.state_log) {
                uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
                for (int k = 0; k < NV; ++k) __stcs(lp + k, p_rec[k]);
            }
            odd = p_odd;
        }
        // ---- marks of cohort n + 1 (and its session / outcome for phase C) ----
        if (n + 1 < nst && cnt > 0) {
            const uint32_t st1 = (un + 1u) & 1u;
            if (!wait_stage(st1, ((un + 1u) >> 1) & 1u)) give_up(un + 1u);
            if (mine) {
                nx_s = idx_of(st1)[tid];
                nx_o = out_of(st1)[tid];
                if (nx_s < N) marks[static_cast<size_t>((un + 1u) % 3u) * N + nx_s] = un + 1u;
            }
        }
        if (tid == 0) dcount[(un + 1u) & 1u] = 0;
        mark_time(n, 1);
        // ---- B: the dirty members of step n ----
        if (n >= 0 && tid < dcount[un & 1u]) {
            const uint32_t st = un & 1u;
            const uint32_t t = dlist[st][tid];
            Event<P> ev;
            ev.s = idx_of(st)[t];
            ev.o = out_of(st)[t];
            read_payload_swizzled<P>(ev.pw, pay_of(st), t);
            odd += transition<SB, P, true, true>(a, ev, tab + sel * a.tab_stride, sel, un, m0 + t, keep_pol);
        }
        mark_time(n, 2);
        uint32_t v = odd;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
        if ((tid & 31u) == 0) warp_odd[tid >> 5] = v;
        __syncthreads();  // (1) step n's stores issued, counts posted, stage n & 1 free
        if (s_abort) break;
        mark_time(n, 3);
        unsigned long long *word = &a.dev->slot[(un + 1u) % 3u];
        uint32_t total = 0;
        if (tid == 0) {
            for (uint32_t w = 0; w < (blockDim.x + 31u) / 32u; ++w) total += warp_odd[w];
            if (!single) {
                if (blockIdx.x == 0) a.dev->slot[(un + 2u) % 3u] = 0ull;
                const bool skip = (n == 0 && blockIdx.x == 1 && ld_volatile_u32(&a.dev->skip_arrival) != 0u);
                __threadfence();
                if (!skip) red_release_add_u64(word, (1ull << 32) | total);
            }
            mark_time(n, 4);
        }
        if (tid == issuer) {
            if (n >= 0 && cnt > 0) s_pending &= ~(1u << (un & 1u));
            if (n >= 0 && cnt > 0 && n + 2 < nst) {
                fence_proxy_async_smem();
                issue(un + 2u);
            }
        }
        // ---- C: early work for this thread's member of step n + 1 ----
        pv = false;
        p_odd = 0;
        if (n + 1 < nst && mine) {
            const uint32_t st1 = (un + 1u) & 1u;
            if (nx_s >= N) {
                latch_error(a.dev, DEV_E_INDEX, un + 1u, m0 + tid);
            } else {
                // is this session in cohort n (whose writes are not yet visible)?
                const bool dirty = n >= 0 && __ldcg(marks + static_cast<size_t>(un % 3u) * N + nx_s) == un;
                if (dirty) {
                    const uint32_t k = atomicAdd(&dcount[st1], 1u);
                    dlist[st1][k] = static_cast<uint16_t>(tid);
                } else {
                    uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(nx_s) * SB);
#pragma unroll
                    for (int k = 0; k < NV; ++k) p_rec[k] = ld_cg_hint(rp + k, keep_pol);
                    const uint32_t x = p_rec[0].x;
                    if (x >= a.S || nx_o >= 8u) {
                        latch_error(a.dev, DEV_E_STATE, un + 1u, m0 + tid);
                    } else {
                        uint4 pw[P / 16];
                        read_payload_swizzled<P>(pw, pay_of(st1), tid);
                        p_rk = route_key<P>(x, nx_o, pw);
                        p_rec[0].y = p_rec[0].y + 1u;
                        mix_acc<SB>(p_rec, p_rk);
                        p_s = nx_s;
                        p_o = nx_o;
                        p_x = x;
                        p_odd = static_cast<uint32_t>(p_rk & 1u);
                        pv = true;
                    }
                }
            }
        }
        // ---- the barrier of step n ----
        mark_time(n, 5);
        if (tid == 0) {
            if (single) {
                s_sel = total > a.K / 2u ? 1u : 0u;
            } else {
                uint64_t t0 = 0;
                unsigned long long w;
                uint32_t spins = 0;
                for (;;) {
                    w = ld_acquire_u64(word);
                    if ((w >> 32) >= gridDim.x) break;
                    if ((++spins & 63u) == 0u) {
                        if (ld_volatile_u32(&a.dev->abort) != 0u) {
                            s_abort = 1;
                            break;
                        }
                        if (timed_out(t0, limit)) {
                            give_up(un);
                            break;
                        }
                    }
                }
                __threadfence();
                s_sel = (static_cast<uint32_t>(w & 0xffffffffull) > a.K / 2u) ? 1u : 0u;
            }
            if (n >= 0 && blockIdx.x == 0 && a.decisions && !s_abort) a.decisions[un] = s_sel;
            mark_time(n, 6);
        }
        __syncthreads();  // (2) decision known; dirty list of step n + 1 complete
        mark_time(n, 7);
        if (s_abort) break;
        if (n >= 0) sel = s_sel;
    }
    if (s_abort) {
        if (tid == 0) {
            for (uint32_t st = 0; st < 2; ++st) {
                if (!(s_pending & (1u << st))) continue;
                const uint32_t parity = (s_pend_step[st] >> 1) & 1u;
                const uint64_t t0 = globaltimer_ns();
                while (!mbar_try_wait(&bar[st], parity)) {
                    if (globaltimer_ns() - t0 > limit) break;
                }
            }
        }
        __syncthreads();
        return;
    }
    if (blockIdx.x == 0 && tid == 0) {
        if (nst > 0) a.dev->sel = sel;
        a.dev->step = a.n_steps;
    }
}

// ---------------------------------------------------------------------------
// Persistent chain with session ownership (explicit session indices; G CTAs,
// CTA b owns sessions [b*per, (b+1)*per)).
//
// k_route groups every cohort's members by the CTA that owns their session:
// for cohort j it writes, contiguously per owner, the member index, the
// session and the outcome (owner b's run is [off[j][b], off[j][b+1])).
// k_chain_owned then lets each CTA transition only its own sessions, so no
// CTA ever reads a record another CTA writes: the state field of every owned
// session lives in shared memory (the whole record when RES), the per-step
// grid barrier carries nothing but the odd-key count (a relaxed atomic on a
// monotonic word per step mod 4, no fence), and a CTA arrives for step n
// before it waits for the decision of step n - 1, so that wait overlaps a
// whole step of route-key work.  Iteration n:
//   1. its payload rows (TMA-free: per-thread async copies, issued one step
//      ahead) and run of step n are ready; (non-RES) issue the record loads;
//   2. route key of every owned member from the state in shared memory;
//   3. post the odd count of step n (relaxed add);
//   4. wait for step n - 1's count: decision d_{n-1} = body of step n;
//   5. next state y = T_d[x][o] into shared memory, record and effect out.
// Four steps of barrier words suffice: a CTA can arrive for step k + 4 only
// after the barrier of step k + 2 completed, that is after every CTA has
// read the word of step k.  Waits are bounded as in the other grid kernels.
// ---------------------------------------------------------------------------
__global__ void k_route(const uint32_t *idx, const uint32_t *outcome, uint32_t n_sets, uint32_t K, uint64_t N,
                        uint32_t G, uint32_t per, uint32_t *perm_m, uint32_t *perm_s, uint32_t *perm_o,
                        uint32_t *off, DevBlock *dev) {
    extern __shared__ uint32_t hist[];  // [G + 1]
    const uint32_t j = blockIdx.x;
    for (uint32_t b = threadIdx.x; b <= G; b += blockDim.x) hist[b] = 0;
    __syncthreads();
    const size_t e0 = static_cast<size_t>(j) * K;
    for (uint32_t m = threadIdx.x; m < K; m += blockDim.x) {
        const uint32_t s = idx ? idx[e0 + m] : m;
        if (s < N) atomicAdd(&hist[s / per], 1u);
        else latch_error(dev, DEV_E_INDEX, 0xffffffffu, m);
    }
    __syncthreads();
    if (threadIdx.x == 0) {  // exclusive scan (G <= a few hundred)
        uint32_t acc = 0;
        for (uint32_t b = 0; b < G; ++b) {
            const uint32_t c = hist[b];
            hist[b] = acc;
            off[static_cast<size_t>(j) * (G + 1) + b] = acc;
            acc += c;
        }
        off[static_cast<size_t>(j) * (G + 1) + G] = acc;
    }
    __syncthreads();
    for (uint32_t m = threadIdx.x; m < K; m += blockDim.x) {
        const uint32_t s = idx ? idx[e0 + m] : m;
        if (s >= N) continue;
        const uint32_t p = atomicAdd(&hist[s / per], 1u);
        perm_m[e0 + p] = m;
        perm_s[e0 + p] = s;
        perm_o[e0 + p] = outcome[e0 + m];
    }
}

// Copies each cohort's payload rows into routed order: row i of cohort j
// becomes the payload of member perm_m[j][i], so that every CTA's run of a
// cohort is a block of consecutive rows that tensor tiles can load.  Rows
// past the cohort's routed count (invalid sessions) are left alone.
__global__ void k_permute_payload(const uint8_t *payload, const uint32_t *perm_m, const uint32_t *off,
                                  uint32_t n_sets, uint32_t K, uint32_t G, uint32_t P, uint8_t *out) {
    const uint32_t nc = P / 16u;
    const size_t total = static_cast<size_t>(n_sets) * K * nc;
    for (size_t q = static_cast<size_t>(blockIdx.x) * blockDim.x + threadIdx.x; q < total;
         q += static_cast<size_t>(gridDim.x) * blockDim.x) {
        const size_t e = q / nc;
        const uint32_t c = static_cast<uint32_t>(q % nc);
        const size_t j = e / K;
        const uint32_t i = static_cast<uint32_t>(e % K);
        if (i >= off[j * (G + 1u) + G]) continue;
        const uint32_t m = perm_m[e];
        reinterpret_cast<uint4 *>(out)[e * nc + c] =
            __ldg(reinterpret_cast<const uint4 *>(payload + (j * K + m) * P) + c);
    }
}

struct OwnedShape {
    uint32_t G;    // CTAs
    uint32_t per;  // sessions owned per CTA
    uint32_t res;  // records resident in shared memory
    uint32_t pad;
};

__device__ __forceinline__ uint32_t ld_relaxed_hi(const unsigned long long *p, uint32_t *lo) {
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    *lo = static_cast<uint32_t>(v);
    return static_cast<uint32_t>(v >> 32);
}

// One routed member: index in its cohort, session, outcome; valid when this
// thread's slot lies inside its CTA's run.
struct Routed {
    uint32_t m, s, o, valid;
};

template <int SB, int P, bool RES>
__global__ void __launch_bounds__(512, 1)
    k_chain_owned(const __grid_constant__ CUtensorMap tmap, StepArgs a, OwnedShape sh, const uint32_t *perm_m,
                  const uint32_t *perm_s, const uint32_t *perm_o, const uint32_t *off) {
    constexpr int NV = SB / 16;
    constexpr uint32_t NC = P / 16;
    constexpr uint32_t kTileRows = 256;
    extern __shared__ __align__(16) uint8_t dsm[];
    __shared__ __align__(8) uint64_t tbar[2];
    __shared__ uint32_t warp_odd[16];
    __shared__ uint32_t s_sel, s_abort;
    const uint32_t tid = threadIdx.x;
    const uint32_t T = blockDim.x;
    const uint32_t b = blockIdx.x;
    const uint32_t G = gridDim.x;
    const uint32_t nst = a.n_steps;
    const uint64_t limit = a.dev->wait_ns;
    const uint32_t base_s = b * sh.per;
    const uint64_t left = base_s < a.n_sessions ? a.n_sessions - base_s : 0ull;
    const uint32_t own = left < sh.per ? static_cast<uint32_t>(left) : sh.per;
    const size_t n_ev = static_cast<size_t>(a.n_sets) * a.K;
    long long *trace = (a.trace && tid == 0 && (b == 0 || b == G - 1))
                           ? a.trace + (b == 0 ? 0 : static_cast<size_t>(nst) * 8)
                           : nullptr;
    // shared layout: [payload tiles: 2 stages x 2 tiles of 256 rows, 1024-aligned][tables]
    // [record stage: T (not RES)][owned states (u16) or records]
    const uint32_t raw = smem_addr(dsm);
    uint8_t *const pay = dsm + (((raw + 1023u) & ~1023u) - raw);
    constexpr uint32_t kStage = 2u * kTileRows * P;
    uint8_t *tab = pay + 2u * kStage;
    uint4 *rec_st = reinterpret_cast<uint4 *>(tab + 2 * a.tab_stride);
    uint16_t *owned = reinterpret_cast<uint16_t *>(rec_st + (RES ? 0ull : static_cast<size_t>(T) * NV));
    uint4 *owned_rec = reinterpret_cast<uint4 *>(owned);  // RES: [per][NV]
    const uint64_t stream_pol = policy_evict_first();

    stage_tables(tab, a.tables, a.tab_stride, 2, 0);
    for (uint32_t ls = tid; ls < own; ls += T) {
        const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(base_s + ls) * SB);
        if constexpr (RES) {
#pragma unroll
            for (int k = 0; k < NV; ++k) owned_rec[static_cast<size_t>(ls) * NV + k] = rp[k];
        } else {
            const uint32_t x0 = __ldg(reinterpret_cast<const uint32_t *>(rp));
            owned[ls] = static_cast<uint16_t>(x0 < a.S ? x0 : 0xFFFFu);  // >= S stays >= S
        }
    }
    if (tid == 0) {
        s_sel = ld_volatile_u32(&a.dev->sel) & 1u;
        s_abort = 0;
        mbar_init(&tbar[0], 1);
        mbar_init(&tbar[1], 1);
        fence_mbar_init();
    }

    // run of step j for this CTA (two plain loads; clamped so that no branch waits on them)
    auto load_run = [&](uint32_t j, uint32_t &lo, uint32_t &hi) {
        const uint32_t jj = j < nst ? j : 0u;
        const size_t o = static_cast<size_t>(jj % a.n_sets) * (G + 1) + b;
        lo = __ldg(off + o);
        hi = __ldg(off + o + 1);
        if (j >= nst) hi = lo;  // applied when the values are used
    };
    // this thread's entry of step j's run (clamped address, validity kept apart)
    auto load_entry = [&](uint32_t j, uint32_t lo, uint32_t hi, Routed &r) {
        const bool v = j < nst && tid < hi - lo;
        size_t e = static_cast<size_t>((j < nst ? j : 0u) % a.n_sets) * a.K + lo + tid;
        e = v ? e : 0;
        e = e < n_ev ? e : 0;
        r.m = __ldg(perm_m + e);
        r.s = __ldg(perm_s + e);
        r.o = __ldg(perm_o + e);
        r.valid = v ? 1u : 0u;
    };
    // The run of step j sits in rows [j*K + lo, j*K + hi) of the routed
    // payload copy: thread 0 loads it as one or two 256-row tensor tiles
    // (rows past the run are loaded and ignored).  Records are gathered
    // warp-cooperatively: NV lanes take the 16-byte chunks of one record.
    const uint32_t lane = tid & 31u, wbase = tid & ~31u;
    uint32_t tiles_issued = 0;  // thread 0: steps [0, tiles_issued) have had their tiles issued
    auto stage_tiles = [&](uint32_t j, uint32_t lo, uint32_t hi) {  // thread 0
        if (j >= nst) return;
        tiles_issued = j + 1u;
        const uint32_t nb = (hi - lo) > kTileRows ? 2u : 1u;
        uint64_t *bb = &tbar[j & 1u];
        mbar_arrive_expect_tx(bb, nb * kTileRows * P);
        const int32_t row0 = static_cast<int32_t>((j % a.n_sets) * a.K + lo);
        for (uint32_t q = 0; q < nb; ++q)
            tma_load_2d_hint(pay + (j & 1u) * kStage + q * kTileRows * P, &tmap, 0,
                             row0 + static_cast<int32_t>(q * kTileRows), bb, stream_pol);
    };
    auto stage_record = [&](const Routed &r) {  // all lanes of the warp
        if constexpr (!RES) {
            constexpr uint32_t RPI = 32u / NV;
            const uint32_t c = lane % NV;
#pragma unroll
            for (uint32_t k = 0; k < static_cast<uint32_t>(NV); ++k) {
                const uint32_t from = k * RPI + lane / NV;
                const uint32_t s2 = __shfl_sync(0xffffffffu, r.s, from);
                const uint32_t v = __shfl_sync(0xffffffffu, r.valid, from);
                if (v) cp_async16(rec_st + static_cast<size_t>(wbase + from) * NV + c,
                                  reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s2) * SB) + c);
            }
        }
    };
    auto wait_count = [&](uint32_t k, uint32_t *low_prev) -> uint32_t {
        const uint32_t target = (k / 4u + 1u) * G;
        uint64_t t0 = 0;
        uint32_t spins = 0, low = 0;
        for (;;) {
            const uint32_t hi = ld_relaxed_hi(&a.dev->slot4[k & 3u], &low);
            if (hi >= target) break;
            __nanosleep(64);
            if ((++spins & 31u) == 0u) {
                if (ld_volatile_u32(&a.dev->abort) != 0u) {
                    s_abort = 1;
                    break;
                }
                if (timed_out(t0, limit)) {
                    latch_error(a.dev, DEV_E_TIMEOUT, k, b);
                    atomicExch(&a.dev->abort, 1u);
                    s_abort = 1;
                    break;
                }
            }
        }
        const uint32_t total = low - low_prev[k & 3u];
        low_prev[k & 3u] = low;
        return total > a.K / 2u ? 1u : 0u;
    };

    // pipeline: runs three steps ahead, entries two, rows one
    uint32_t lo0, hi0, lo1, hi1, lo2, hi2, lo3, hi3;
    Routed r0, r1, r2;
    load_run(0, lo0, hi0);
    load_run(1, lo1, hi1);
    load_run(2, lo2, hi2);
    load_entry(0, lo0, hi0, r0);
    load_entry(1, lo1, hi1, r1);
    __syncthreads();  // mbarriers initialised
    if (tid == 0) stage_tiles(0, lo0, hi0);
    uint32_t sel = s_sel;
    uint32_t low_prev[4] = {0u, 0u, 0u, 0u};

    for (uint32_t n = 0; n < nst; ++n) {
        if (trace) trace[n * 8 + 0] = clock64();
        load_run(n + 3u, lo3, hi3);
        load_entry(n + 2u, lo2, hi2, r2);
        stage_record(r0);           // records of step n (the previous step's writes are done)
        cp_async_commit();
        if (tid == 0) {             // tiles of step n + 1 into the stage step n - 1 used
            fence_proxy_async_smem();
            stage_tiles(n + 1u, lo1, (n + 1u < nst) ? hi1 : lo1);
        }
        if (!mbar_wait_bounded(&tbar[n & 1u], (n >> 1) & 1u, limit)) {  // tiles of step n
            latch_error(a.dev, DEV_E_TIMEOUT, n, b);
            atomicExch(&a.dev->abort, 1u);
            s_abort = 1;
        }
        if (trace) trace[n * 8 + 1] = clock64();
        const size_t e0 = static_cast<size_t>(n % a.n_sets) * a.K;
        const uint32_t cnt0 = hi0 - lo0;
        uint32_t odd = 0, x = 0;
        uint64_t rk = 0;
        bool ok = false;
        if (r0.valid) {
            const uint32_t ls = r0.s - base_s;
            x = RES ? owned_rec[static_cast<size_t>(ls) * NV].x : static_cast<uint32_t>(owned[ls]);
            if (x >= a.S || r0.o >= 8u) {
                latch_error(a.dev, DEV_E_STATE, n, r0.m);
            } else {
                uint4 pw[NC];
                read_payload_swizzled<P>(pw, pay + (n & 1u) * kStage, tid);
                rk = route_key<P>(x, r0.o, pw);
                odd = static_cast<uint32_t>(rk & 1u);
                ok = true;
            }
        }
        // members beyond one per thread (rare): keys now, state after the decision
        for (uint32_t p = tid + T; p < cnt0; p += T) {
            const size_t e = e0 + lo0 + p;
            const uint32_t s2 = __ldg(perm_s + e), m2 = __ldg(perm_m + e), o2 = __ldg(perm_o + e);
            const uint32_t x2 = RES ? owned_rec[static_cast<size_t>(s2 - base_s) * NV].x : owned[s2 - base_s];
            if (x2 >= a.S || o2 >= 8u) {
                latch_error(a.dev, DEV_E_STATE, n, m2);
                continue;
            }
            uint4 pw[NC];
            const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + (e0 + m2) * P);
#pragma unroll
            for (uint32_t k = 0; k < NC; ++k) pw[k] = __ldg(src + k);
            odd += static_cast<uint32_t>(route_key<P>(x2, o2, pw) & 1u);
        }
        if (trace) trace[n * 8 + 2] = clock64();
        uint32_t v = odd;
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o2);
        if ((tid & 31u) == 0) warp_odd[tid >> 5] = v;
        __syncthreads();
        if (tid == 0) {
            if (trace) trace[n * 8 + 3] = clock64();
            uint32_t c = 0;
            for (uint32_t w = 0; w < (T + 31u) / 32u; ++w) c += warp_odd[w];
            // post step n's count (nothing else crosses CTAs), then take step n - 1's decision
            const bool skip = (n == 0 && b == 1 && ld_volatile_u32(&a.dev->skip_arrival) != 0u);
            if (!skip) atomicAdd(&a.dev->slot4[n & 3u], (1ull << 32) | c);
            if (trace) trace[n * 8 + 4] = clock64();
            if (n > 0) {
                s_sel = wait_count(n - 1u, low_prev);
                if (b == 0 && a.decisions && !s_abort) a.decisions[n - 1u] = s_sel;
            }
            if (trace) trace[n * 8 + 5] = clock64();
        }
        __syncthreads();
        if (s_abort) break;
        if (n > 0) sel = s_sel;
        cp_async_wait<0>();  // the warp's records of step n are here
        __syncwarp();
        if (trace) trace[n * 8 + 6] = clock64();
        // --- next state, record and effect (body chosen by the decision of step n - 1) ---
        // coop: the record goes back to this thread's shared stage, and the warp
        // stores the stages cooperatively below
        auto finish = [&](uint32_t s2, uint32_t m2, uint32_t o2, uint32_t x2, uint64_t rk2, uint4 (&rr)[NV],
                          bool coop) {
            const uint32_t y = tab[sel * a.tab_stride + x2 * 8u + o2];
            rr[0].x = y;
            rr[0].y = rr[0].y + 1u;
            mix_acc<SB>(rr, rk2);
            const uint32_t ls = s2 - base_s;
            if constexpr (RES) {
#pragma unroll
                for (int k = 0; k < NV; ++k) owned_rec[static_cast<size_t>(ls) * NV + k] = rr[k];
            } else {
                owned[ls] = static_cast<uint16_t>(y);
                if (coop) {
#pragma unroll
                    for (int k = 0; k < NV; ++k) rec_st[static_cast<size_t>(tid) * NV + k] = rr[k];
                } else {
                    uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s2) * SB);
#pragma unroll
                    for (int k = 0; k < NV; ++k) rp[k] = rr[k];
                }
            }
            const size_t slot = static_cast<size_t>(n) * a.K + m2;
            if (a.effects) {
                uint4 e;
                e.x = static_cast<uint32_t>(rk2);
                e.y = static_cast<uint32_t>(rk2 >> 32);
                e.z = s2;
                e.w = y | (o2 << 16) | (sel << 24);
                __stcs(reinterpret_cast<uint4 *>(a.effects) + slot, e);
            }
            if (a.state_log) {
                uint4 *lp = reinterpret_cast<uint4 *>(a.state_log + slot * SB);
#pragma unroll
                for (int k = 0; k < NV; ++k) __stcs(lp + k, rr[k]);
            }
        };
        if (ok) {
            uint4 rr[NV];
            if constexpr (RES) {
#pragma unroll
                for (int k = 0; k < NV; ++k) rr[k] = owned_rec[static_cast<size_t>(r0.s - base_s) * NV + k];
            } else {
#pragma unroll
                for (int k = 0; k < NV; ++k) rr[k] = rec_st[static_cast<size_t>(tid) * NV + k];
            }
            finish(r0.s, r0.m, r0.o, x, rk, rr, true);
        }
        if constexpr (!RES) {
            // the warp's updated records, NV lanes per record
            __syncwarp();
            constexpr uint32_t RPI = 32u / NV;
            const uint32_t c = lane % NV;
#pragma unroll
            for (uint32_t k = 0; k < static_cast<uint32_t>(NV); ++k) {
                const uint32_t from = k * RPI + lane / NV;
                const uint32_t s2 = __shfl_sync(0xffffffffu, r0.s, from);
                const uint32_t v = __shfl_sync(0xffffffffu, ok ? 1u : 0u, from);
                if (v)
                    reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s2) * SB)[c] =
                        rec_st[static_cast<size_t>(wbase + from) * NV + c];
            }
        }
        for (uint32_t p = tid + T; p < cnt0; p += T) {
            const size_t e = e0 + lo0 + p;
            const uint32_t s2 = __ldg(perm_s + e), m2 = __ldg(perm_m + e), o2 = __ldg(perm_o + e);
            uint4 rr[NV];
            uint32_t x2;
            if constexpr (RES) {
#pragma unroll
                for (int k = 0; k < NV; ++k) rr[k] = owned_rec[static_cast<size_t>(s2 - base_s) * NV + k];
                x2 = rr[0].x;
            } else {
                const uint4 *rp = reinterpret_cast<const uint4 *>(a.state + static_cast<size_t>(s2) * SB);
#pragma unroll
                for (int k = 0; k < NV; ++k) rr[k] = __ldcg(rp + k);
                x2 = owned[s2 - base_s];
            }
            if (x2 >= a.S || o2 >= 8u) continue;
            uint4 pw[NC];
            const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + (e0 + m2) * P);
#pragma unroll
            for (uint32_t k = 0; k < NC; ++k) pw[k] = __ldg(src + k);
            finish(s2, m2, o2, x2, route_key<P>(x2, o2, pw), rr, false);
        }
        __syncthreads();  // owned state updated before the next step reads it; stages free
        if (trace) trace[n * 8 + 7] = clock64();
        lo0 = lo1;
        hi0 = hi1;
        r0 = r1;
        lo1 = lo2;
        hi1 = hi2;
        r1 = r2;
        lo2 = lo3;
        hi2 = hi3;
    }
    cp_async_wait<0>();
    if (tid == 0) {  // the tiles still in flight after an early stop (bounded)
        for (uint32_t j = tiles_issued >= 2u ? tiles_issued - 2u : 0u; j < tiles_issued; ++j)
            (void)mbar_wait_bounded(&tbar[j & 1u], (j >> 1) & 1u, limit);
    }
    if (tid == 0 && !s_abort && nst > 0) {
        s_sel = wait_count(nst - 1u, low_prev);
        if (b == 0 && !s_abort) {
            if (a.decisions) a.decisions[nst - 1u] = s_sel;
            a.dev->sel = s_sel;
            a.dev->step = nst;
        }
    }
    __syncthreads();
    if constexpr (RES) {
        if (!s_abort) {
            for (uint32_t ls = tid; ls < own; ls += T) {
                uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(base_s + ls) * SB);
#pragma unroll
                for (int k = 0; k < NV; ++k) rp[k] = owned_rec[static_cast<size_t>(ls) * NV + k];
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Segmented step: one launch over several route-keyed cohorts (segments),
// each with its own pair of route bodies and its own decision chain (the
// per-route compaction with variable route bodies that Section 9.1 and the
// scope paragraph of Section 10 leave to a route service).  Member m finds
// its segment by binary search over seg_off, transitions with the body its
// route's flag selects, and adds its odd key to its segment's count (warp
// lanes of one segment aggregate first); the last CTA (ticket) turns every
// count into that segment's decision, the route's next flag.  Sessions are
// distinct across the whole step (checked by the caller's contract), so the
// segments commute and the step equals their cohort steps in any order.
// ---------------------------------------------------------------------------
template <int SB, int P>
__global__ void __launch_bounds__(kStepThreads) k_seg_step(SegArgs a) {
    constexpr int NV = SB / 16;
    __shared__ uint32_t s_last;
    const uint32_t tid = threadIdx.x;
    const uint32_t lane = tid & 31u;
    const uint32_t m = blockIdx.x * blockDim.x + tid;
    const bool act = m < a.total;
    uint32_t g = 0, odd = 0;
    if (act) {
        uint32_t lo = 0, hi = a.n_seg;  // seg_off[lo] <= m < seg_off[hi]
        while (hi - lo > 1u) {
            const uint32_t mid = (lo + hi) >> 1;
            if (__ldg(a.seg_off + mid) <= m) lo = mid;
            else hi = mid;
        }
        g = lo;
        const uint32_t r = __ldg(a.seg_route + g);
        const uint32_t sel = a.flags[r] & 1u;
        const uint8_t *tab = a.tables + static_cast<size_t>(2u * r + sel) * a.tab_stride;
        const uint32_t s = a.idx ? __ldg(a.idx + m) : m;
        const uint32_t o = __ldg(a.outcome + m);
        if (s >= a.n_sessions) {
            latch_error(a.dev, DEV_E_INDEX, g, m);
        } else {
            uint4 *rp = reinterpret_cast<uint4 *>(a.state + static_cast<size_t>(s) * SB);
            uint4 rr[NV];
#pragma unroll
            for (int k = 0; k < NV; ++k) rr[k] = rp[k];
            const uint32_t x = rr[0].x;
            if (x >= a.S || o >= 8u) {
                latch_error(a.dev, DEV_E_STATE, g, m);
            } else {
                uint4 pw[P / 16];
                const uint4 *src = reinterpret_cast<const uint4 *>(a.payload + static_cast<size_t>(m) * P);
#pragma unroll
                for (int k = 0; k < P / 16; ++k) pw[k] = __ldg(src + k);
                const uint64_t rk = route_key<P>(x, o, pw);
                const uint32_t y = __ldg(tab + x * 8u + o);
                rr[0].x = y;
                rr[0].y = rr[0].y + 1u;
                mix_acc<SB>(rr, rk);
#pragma unroll
                for (int k = 0; k < NV; ++k) rp[k] = rr[k];
                if (a.effects) {
                    uint4 e;
                    e.x = static_cast<uint32_t>(rk);
                    e.y = static_cast<uint32_t>(rk >> 32);
                    e.z = s;
                    e.w = y | (o << 16) | (sel << 24);
                    __stcs(reinterpret_cast<uint4 *>(a.effects) + m, e);
                }
                odd = static_cast<uint32_t>(rk & 1u);
            }
        }
    }
    // per-segment odd counts: lanes of one segment aggregate, their first lane adds
    const uint32_t amask = __ballot_sync(0xffffffffu, act);
    if (act) {
        const uint32_t same = __match_any_sync(amask, g);
        const uint32_t c = __popc(__ballot_sync(amask, odd != 0u) & same);
        if (lane == static_cast<uint32_t>(__ffs(same) - 1) && c != 0u) atomicAdd(a.count + g, c);
    }
    __syncthreads();
    if (tid == 0) {
        __threadfence();
        s_last = atomicAdd(a.ticket, 1u) == gridDim.x - 1u ? 1u : 0u;
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (uint32_t q = tid; q < a.n_seg; q += blockDim.x) {
        const uint32_t c = atomicExch(a.count + q, 0u);
        const uint32_t size = __ldg(a.seg_off + q + 1u) - __ldg(a.seg_off + q);
        const uint32_t d = c > size / 2u ? 1u : 0u;
        a.flags[__ldg(a.seg_route + q)] = d;
        if (a.decisions) a.decisions[q] = d;
    }
    if (tid == 0) *a.ticket = 0u;
}

__global__ void k_empty_cohorts(StepArgs a) {
    for (uint32_t n = blockIdx.x * blockDim.x + threadIdx.x; n < a.n_steps; n += gridDim.x * blockDim.x)
        if (a.decisions) a.decisions[n] = 0u;
    if (blockIdx.x == 0 && threadIdx.x == 0 && a.n_steps > 0) {
        a.dev->sel = 0u;
        a.dev->step = a.n_steps;
    }
}

// Fixed-nested control: device-launches a pre-uploaded child graph that holds
// the route body the host chose.  It removes no host decision.
__global__ void k_launch_child(cudaGraphExec_t child, DevBlock *dev) {
    if (cudaGraphLaunch(child, cudaStreamGraphFireAndForget) != cudaSuccess) {
        latch_error(dev, DEV_E_STATE, 0xffffffffu, 0xffffffffu);
    }
}

// One word written in stream order (the step base of a chain run in pieces).
__global__ void k_set_word(uint32_t *p, uint32_t v) { *p = v; }

__global__ void k_empty() {}

// Launch-floor probe of the persistent grid chains: one CTA per SM runs
// n_steps empty steps, each one grid barrier exactly as the large-K chain
// keys it (block barrier, release add of (1 << 32 | count) to the step's
// word, CTA 0 clearing the word two steps back, acquire spin bounded by
// dev->wait_ns, block barrier), with no member work between barriers.
__global__ void __launch_bounds__(480, 1) k_grid_barrier_floor(DevBlock *dev, uint32_t n_steps) {
    __shared__ uint32_t s_stop;
    const uint32_t G = gridDim.x;
    const uint64_t limit = dev->wait_ns;
    if (threadIdx.x == 0) s_stop = 0;
    __syncthreads();
    for (uint32_t n = 0; n < n_steps; ++n) {
        if (threadIdx.x == 0) {
            unsigned long long *word = &dev->slot[n % 3u];
            if (blockIdx.x == 0) dev->slot[(n + 1u) % 3u] = 0ull;
            red_release_add_u64(word, (1ull << 32) | (blockIdx.x & 1u));
            uint64_t t0 = 0;
            uint32_t spins = 0;
            for (;;) {
                if ((ld_acquire_u64(word) >> 32) >= G) break;
                if ((++spins & 63u) == 0u) {
                    if (ld_volatile_u32(&dev->abort) != 0u) {
                        s_stop = 1;
                        break;
                    }
                    if (timed_out(t0, limit)) {
                        latch_error(dev, DEV_E_TIMEOUT, n, blockIdx.x);
                        atomicExch(&dev->abort, 1u);
                        s_stop = 1;
                        break;
                    }
                }
            }
        }
        __syncthreads();
        if (s_stop != 0u) break;
    }
}

__global__ void k_countdown(DevBlock *dev, cudaGraphConditionalHandle h) {
    const uint32_t left = dev->countdown - 1u;
    dev->countdown = left;
    cudaGraphSetConditional(h, left != 0u ? 1u : 0u);
}

template <int SB, int P>
const void *pick_step(bool decide) {
    return decide ? reinterpret_cast<const void *>(&k_step<SB, P, true>)
                  : reinterpret_cast<const void *>(&k_step<SB, P, false>);
}

template <int V>
using IC = std::integral_constant<int, V>;

// Calls f(IC<state_bytes>, IC<payload_bytes>) for the supported shapes.
template <typename F>
auto dispatch(int SB, int P, F &&f) {
    if (SB == 16) {
        if (P == 32) return f(IC<16>{}, IC<32>{});
        if (P == 64) return f(IC<16>{}, IC<64>{});
        return f(IC<16>{}, IC<128>{});
    }
    if (P == 32) return f(IC<64>{}, IC<32>{});
    if (P == 64) return f(IC<64>{}, IC<64>{});
    return f(IC<64>{}, IC<128>{});
}

}  // namespace

const void *step_kernel(int SB, int P, bool decide) {
    return dispatch(SB, P, [&](auto b, auto q) { return pick_step<decltype(b)::value, decltype(q)::value>(decide); });
}

dim3 step_block(uint32_t K) {
    const uint32_t b = K >= static_cast<uint32_t>(kStepThreads) ? kStepThreads : ((K + 31u) / 32u) * 32u;
    return dim3(b ? b : 32u);
}

dim3 step_grid(uint32_t K) {
    const uint32_t b = step_block(K).x;
    const uint32_t g = (K + b - 1u) / b;
    return dim3(g ? g : 1u);
}

cudaError_t launch_step(const StepArgs &a, int SB, int P, int step, int sel, uint32_t epi, bool decide,
                        cudaStream_t s) {
    const void *fn = step_kernel(SB, P, decide);
    StepArgs aa = a;
    void *args[] = {&aa, &step, &sel, &epi};
    return cudaLaunchKernel(fn, step_grid(a.K), step_block(a.K), args, 0, s);
}

namespace {
template <int SB, int P, int D>
const void *ident_fn() {
    return reinterpret_cast<const void *>(&k_chain_cta_ident<SB, P, D>);
}
const void *ident_fn_rt(int SB, int P, int D) {
    return dispatch(SB, P, [&](auto b, auto q) {
        constexpr int B = decltype(b)::value, Q = decltype(q)::value;
        return D == 4 ? ident_fn<B, Q, 4>() : D == 2 ? ident_fn<B, Q, 2>() : ident_fn<B, Q, 1>();
    });
}
size_t ident_smem(uint32_t K, int P, int D, uint32_t tab_stride) {
    const size_t Kp = (K + 3u) & ~3u, RD = D + 1;
    return 2 * tab_stride + RD * Kp * 4 + RD * Kp * P;
}
const void *ident2_fn_rt(int SB, int P, int D) {
    return dispatch(SB, P, [&](auto b, auto q) {
        constexpr int B = decltype(b)::value, Q = decltype(q)::value;
        return D == 4 ? reinterpret_cast<const void *>(&k_chain_cta_ident2<B, Q, 4>)
                      : reinterpret_cast<const void *>(&k_chain_cta_ident2<B, Q, 2>);
    });
}
const void *warp_fn_rt(int SB, int P, int D) {
    return dispatch(SB, P, [&](auto b, auto q) {
        constexpr int B = decltype(b)::value, Q = decltype(q)::value;
        return D == 4 ? reinterpret_cast<const void *>(&k_chain_warp_ident<B, Q, 4>)
                      : reinterpret_cast<const void *>(&k_chain_warp_ident<B, Q, 2>);
    });
}
size_t ident2_smem(uint32_t K, int P, int D, uint32_t tab_stride) {
    const size_t Kp = (K + 3u) & ~3u, RD = D + 2;
    return 2 * tab_stride + RD * Kp * 4 + RD * Kp * P;
}
int max_optin_smem() {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return 0;
    return v;
}
}  // namespace

cudaError_t launch_chain_cta_fast(const StepArgs &a, int SB, int P, cudaStream_t s, bool *launched,
                                  bool two_steps) {
    *launched = false;
    const uint32_t K = a.K;
    if (K == 0 || K > 1024u) return cudaSuccess;
    const size_t cap = static_cast<size_t>(max_optin_smem());
    const uint32_t threads = ((K + 31u) / 32u) * 32u;
    StepArgs aa = a;
    if (!a.idx && two_steps && K <= 32u) {
        for (int D : {4, 2}) {
            const size_t smem = ident2_smem(K, P, D, a.tab_stride);
            if (smem > cap) continue;
            const void *fn = warp_fn_rt(SB, P, D);
            cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            void *args[] = {&aa};
            *launched = true;
            return cudaLaunchKernel(fn, dim3(1), dim3(32), args, smem, s);
        }
    }
    if (!a.idx && two_steps && K <= 512u) {
        for (int D : {4, 2}) {
            const size_t smem = ident2_smem(K, P, D, a.tab_stride);
            if (smem > cap) continue;
            const void *fn = ident2_fn_rt(SB, P, D);
            cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            void *args[] = {&aa};
            *launched = true;
            return cudaLaunchKernel(fn, dim3(1), dim3(threads), args, smem, s);
        }
    }
    if (!a.idx) {
        for (int D : {4, 2, 1}) {
            const size_t smem = ident_smem(K, P, D, a.tab_stride);
            if (smem > cap) continue;
            const void *fn = ident_fn_rt(SB, P, D);
            cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
            if (e != cudaSuccess) return e;
            void *args[] = {&aa};
            *launched = true;
            return cudaLaunchKernel(fn, dim3(1), dim3(threads), args, smem, s);
        }
        return cudaSuccess;
    }
    return cudaSuccess;
}

cudaError_t launch_chain_cta(const StepArgs &a, int SB, int P, cudaStream_t s) {
    const void *fn = dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_cta<decltype(b)::value, decltype(q)::value>);
    });
    StepArgs aa = a;
    void *args[] = {&aa};
    const uint32_t threads = ((a.K + 31u) / 32u) * 32u;
    return cudaLaunchKernel(fn, dim3(1), dim3(threads ? threads : 32u), args, 0, s);
}

static const void *grid_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_grid<decltype(b)::value, decltype(q)::value>);
    });
}

cudaError_t chain_grid_size(int SB, int P, uint32_t K, int *grid) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, grid_fn(SB, P), kGridThreads, 0);
    if (e != cudaSuccess) return e;
    const long long cap = static_cast<long long>(sms) * per_sm;
    const long long need = (static_cast<long long>(K) + kGridThreads - 1) / kGridThreads;
    long long g = need < cap ? need : cap;
    if (g < 1) g = 1;
    *grid = static_cast<int>(g);
    return cudaSuccess;
}

cudaError_t launch_chain_grid(const StepArgs &a, int SB, int P, int grid, cudaStream_t s) {
    StepArgs aa = a;
    void *args[] = {&aa};
    return cudaLaunchCooperativeKernel(grid_fn(SB, P), dim3(grid), dim3(kGridThreads), args, 0, s);
}

static const void *grid_tma_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_grid_tma<decltype(b)::value, decltype(q)::value>);
    });
}

namespace {
using EncodeTiled = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                 const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiled encode_fn() {
    static EncodeTiled fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiled>(p);
    }
    return fn;
}

size_t tma_smem_bytes(const TmaShape &sh, uint32_t tab_stride) {
    return 1024 + 2ull * sh.stage_pay + 4ull * sh.stage_words * 4 + 2ull * tab_stride;
}
}  // namespace

// Chooses the TMA grid shape for K members, or returns false when the TMA
// kernel does not apply (K not a multiple of 8, or a stage would not fit).
bool chain_grid_tma_plan(int SB, int P, uint32_t K, uint32_t tab_stride, int *grid, uint32_t *threads,
                         size_t *smem, void *shape_out) {
    if (K == 0 || K % 8u != 0u || !encode_fn()) return false;
    int dev = 0, sms = 0, max_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return false;
    TmaShape sh;
    uint32_t per = (K + static_cast<uint32_t>(sms) - 1u) / static_cast<uint32_t>(sms);
    sh.chunk = (per + 7u) & ~7u;
    const uint32_t g = (K + sh.chunk - 1u) / sh.chunk;
    sh.n_boxes = (sh.chunk + 255u) / 256u;
    sh.box_rows = (((sh.chunk + sh.n_boxes - 1u) / sh.n_boxes) + 7u) & ~7u;
    sh.stage_pay = ((sh.n_boxes * sh.box_rows * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
    sh.stage_words = (sh.chunk + 3u) & ~3u;
    const uint32_t thr = sh.chunk >= 512u ? 512u : ((sh.chunk + 31u) / 32u) * 32u;
    const size_t rec_stage = SB >= 64 ? static_cast<size_t>(thr) * SB + 16 : 0;
    const size_t bytes = tma_smem_bytes(sh, tab_stride) + rec_stage;
    if (bytes + 2048 > static_cast<size_t>(max_optin)) return false;
    const void *fn = grid_tma_fn(SB, P);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes)) !=
        cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, static_cast<int>(thr), bytes) != cudaSuccess ||
        per_sm < 1 || static_cast<long long>(per_sm) * sms < g)
        return false;
    *grid = static_cast<int>(g);
    *threads = thr;
    *smem = bytes;
    *static_cast<TmaShape *>(shape_out) = sh;
    return true;
}

cudaError_t launch_chain_grid_tma(const StepArgs &a, int SB, int P, int grid, uint32_t threads, size_t smem,
                                  const void *shape, cudaStream_t s) {
    const TmaShape &sh = *static_cast<const TmaShape *>(shape);
    EncodeTiled enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    alignas(64) CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(P), static_cast<cuuint64_t>(a.n_sets) * a.K};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(P)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(P), sh.box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz = P == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                   : P == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                             : CU_TENSOR_MAP_SWIZZLE_32B;
    CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.payload), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    StepArgs aa = a;
    TmaShape shc = sh;
    void *args[] = {&map, &aa, &shc};
    return cudaLaunchCooperativeKernel(grid_tma_fn(SB, P), dim3(grid), dim3(threads), args, smem, s);
}

namespace {
const void *link_fn_rt(int SB, int P, bool prod) {
    return dispatch(SB, P, [&](auto b, auto q) {
        constexpr int B = decltype(b)::value, Q = decltype(q)::value;
        return prod ? reinterpret_cast<const void *>(&k_chain_cta_prod<B, Q>)
                    : reinterpret_cast<const void *>(&k_chain_cta_link<B, Q>);
    });
}
size_t link_smem(const LinkShape &sh, uint32_t K, int SB, uint32_t tab_stride) {
    const size_t Kp = (K + 3u) & ~3u;
    if (sh.prod)
        return 1024 + kProdRP * static_cast<size_t>(sh.stage_pay) + kProdRR * static_cast<size_t>(K) * SB +
               kProdRW * 3ull * K * 4 + 2ull * tab_stride;
    return 1024 + kLinkRP * static_cast<size_t>(sh.stage_pay) + kLinkRR * Kp * SB + 2ull * kLinkRI * Kp * 4 +
           kLinkRP * Kp * 4 + 2ull * tab_stride;
}
}  // namespace

bool chain_cta_link_plan(int SB, int P, uint32_t K, uint64_t n_sessions, uint32_t tab_stride, bool allow_prod,
                         size_t *smem, void *shape_out) {
    if (K == 0 || K > 512u || n_sessions > 0xFFFFFFFFull) return false;
    const size_t cap = static_cast<size_t>(max_optin_smem());
    LinkShape sh{};
    if (allow_prod && K % 8u == 0u && encode_fn()) {
        sh.prod = 1;
        sh.n_boxes = K <= 256u ? 1u : 2u;
        sh.box_rows = (((K + sh.n_boxes - 1u) / sh.n_boxes) + 7u) & ~7u;
        sh.stage_pay = ((sh.n_boxes * sh.box_rows * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
        const size_t bytes = link_smem(sh, K, SB, tab_stride);
        if (bytes <= cap) {
            *smem = bytes;
            *static_cast<LinkShape *>(shape_out) = sh;
            return true;
        }
    }
    sh = LinkShape{};
    const uint32_t Kp = (K + 3u) & ~3u;
    sh.stage_pay = ((Kp * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
    const size_t bytes = link_smem(sh, K, SB, tab_stride);
    if (bytes > cap) return false;
    *smem = bytes;
    *static_cast<LinkShape *>(shape_out) = sh;
    return true;
}

cudaError_t launch_link(const StepArgs &a, uint32_t *lnk, cudaStream_t s) {
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const uint32_t cap = static_cast<uint32_t>(sms) * 4u;
    const uint32_t grid = a.n_sets < cap ? a.n_sets : cap;
    const uint32_t threads = a.K >= 512u ? 512u : ((a.K + 31u) / 32u) * 32u;
    k_link<<<grid ? grid : 1u, threads ? threads : 32u, 0, s>>>(a.idx, a.n_sets, a.K, a.n_sessions, lnk);
    return cudaGetLastError();
}

namespace {
// Tensor map of the payload rows (P bytes each, n_sets * K rows) in tiles of
// box_rows rows, swizzled to the row length, as the producer warps load them.
bool payload_map(const StepArgs &a, int P, uint32_t box_rows, CUtensorMap *map) {
    EncodeTiled enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(P), static_cast<cuuint64_t>(a.n_sets) * a.K};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(P)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(P), box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz = P == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                   : P == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                             : CU_TENSOR_MAP_SWIZZLE_32B;
    return enc(map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.payload), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}
}  // namespace

namespace {
const void *pair_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) -> const void * {
        constexpr int B = decltype(b)::value, Q = decltype(q)::value;
        if constexpr (Q <= 64) return reinterpret_cast<const void *>(&k_chain_cta_pair<B, Q>);
        return nullptr;
    });
}
size_t pair_smem(uint32_t K, int SB, uint32_t S, uint32_t tab_stride, uint32_t stage_pay) {
    return 1024 + kPairRP * static_cast<size_t>(stage_pay) + kPairRR * static_cast<size_t>(K) * SB + static_cast<size_t>(S) * 64u + kPairRK * 8ull * K +
           kPairRW * 12ull * K + kPairRX * 4ull * K + kPairRX * static_cast<size_t>(K) + kPairRK * static_cast<size_t>(K) +
           2ull * tab_stride;
}
}  // namespace

bool chain_cta_pair_plan(int SB, int P, uint32_t K, uint32_t S, uint64_t n_sessions, uint32_t tab_stride,
                         size_t *smem, void *shape_out) {
    if (K == 0 || K > 256u || K % 8u != 0u || P > 64 || n_sessions > 0xFFFFFFFFull || S == 0 || S > 256u ||
        !encode_fn())
        return false;
    LinkShape sh{};
    sh.prod = 3;
    sh.n_boxes = 1;
    sh.box_rows = K;
    sh.stage_pay = ((K * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
    const size_t bytes = pair_smem(K, SB, S, tab_stride, sh.stage_pay);
    if (bytes > static_cast<size_t>(max_optin_smem())) return false;
    *smem = bytes;
    *static_cast<LinkShape *>(shape_out) = sh;
    return true;
}

cudaError_t launch_link_pair(const StepArgs &a, uint32_t *lnk, cudaStream_t s) {
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    if (a.K > 256u) return cudaErrorInvalidValue;  // the table holds 8 x 256 keys in 4,096 slots
    const uint32_t cap = static_cast<uint32_t>(sms) * 4u;
    const uint32_t grid = a.n_sets < cap ? a.n_sets : cap;
    const uint32_t threads = ((a.K + 31u) / 32u) * 32u;
    k_link_reach<kPairD, 4096><<<grid ? grid : 1u, threads ? threads : 32u, 0, s>>>(a.idx, a.n_sets, a.K,
                                                                                    a.n_sessions, lnk);
    return cudaGetLastError();
}

cudaError_t launch_chain_cta_pair(const StepArgs &a, int SB, int P, size_t smem, const void *shape,
                                  const uint32_t *lnk, cudaStream_t s) {
    const LinkShape &sh = *static_cast<const LinkShape *>(shape);
    const void *fn = pair_fn(SB, P);
    if (!fn) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    alignas(64) CUtensorMap map;
    if (!payload_map(a, P, sh.box_rows, &map)) return cudaErrorInvalidValue;
    StepArgs aa = a;
    const uint32_t *l = lnk;
    LinkShape shc = sh;
    void *args[] = {&map, &aa, &l, &shc};
    const uint32_t member_threads = ((a.K + 31u) / 32u) * 32u;
    return cudaLaunchKernel(fn, dim3(1), dim3(3u * member_threads + 32u), args, smem, s);
}

cudaError_t launch_chain_cta_link(const StepArgs &a, int SB, int P, size_t smem, const void *shape,
                                  const uint32_t *lnk, cudaStream_t s) {
    const LinkShape &sh = *static_cast<const LinkShape *>(shape);
    const void *fn = link_fn_rt(SB, P, sh.prod != 0u);
    cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    StepArgs aa = a;
    const uint32_t *l = lnk;
    LinkShape shc = sh;
    const uint32_t member_threads = ((a.K + 31u) / 32u) * 32u;
    if (!sh.prod) {
        void *args[] = {&aa, &l, &shc};
        return cudaLaunchKernel(fn, dim3(1), dim3(member_threads), args, smem, s);
    }
    EncodeTiled enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    alignas(64) CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(P), static_cast<cuuint64_t>(a.n_sets) * a.K};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(P)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(P), sh.box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz = P == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                   : P == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                             : CU_TENSOR_MAP_SWIZZLE_32B;
    CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.payload), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    void *args[] = {&map, &aa, &l, &shc};
    return cudaLaunchKernel(fn, dim3(1), dim3(member_threads + 32u), args, smem, s);
}

static const void *grid_link_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_grid_link<decltype(b)::value, decltype(q)::value>);
    });
}

bool chain_grid_link_plan(int SB, int P, uint32_t K, uint64_t n_sessions, uint32_t n_sets, uint32_t tab_stride,
                          int *grid, uint32_t *threads, size_t *smem, void *shape_out, size_t *scratch) {
    if (K == 0 || K % 8u != 0u || n_sessions > 0xFFFFFFFFull || !encode_fn()) return false;
    int dev = 0, sms = 0, max_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return false;
    GridLinkShape gs{};
    TmaShape &sh = gs.t;
    const uint32_t per = (K + static_cast<uint32_t>(sms) - 1u) / static_cast<uint32_t>(sms);
    sh.chunk = (per + 7u) & ~7u;
    const uint32_t g = (K + sh.chunk - 1u) / sh.chunk;
    sh.n_boxes = (sh.chunk + 255u) / 256u;
    sh.box_rows = (((sh.chunk + sh.n_boxes - 1u) / sh.n_boxes) + 7u) & ~7u;
    sh.stage_pay = ((sh.n_boxes * sh.box_rows * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
    sh.stage_words = (sh.chunk + 3u) & ~3u;
    gs.members = ((sh.chunk + 31u) / 32u) * 32u;
    if (gs.members + 32u > 544u) return false;
    const size_t bytes = 1024 + 2ull * sh.stage_pay + 6ull * sh.stage_words * 4 + ((2ull * tab_stride + 15u) & ~15ull) +
                         2ull * sh.chunk * SB + 2ull * sh.chunk * 16 + 64;
    if (bytes > static_cast<size_t>(max_optin)) return false;
    const uint64_t words_per_set = (n_sessions + 31u) / 32u;
    const size_t bits_bytes = (static_cast<size_t>(n_sets) * words_per_set * 4 + 255u) & ~static_cast<size_t>(255u);
    const size_t need = bits_bytes + static_cast<size_t>(n_sets) * K * 4;
    if (need > (1ull << 30)) return false;
    const void *fn = grid_link_fn(SB, P);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes)) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, static_cast<int>(gs.members + 32u), bytes) !=
            cudaSuccess ||
        per_sm < 1 || static_cast<long long>(per_sm) * sms < g)
        return false;
    *grid = static_cast<int>(g);
    *threads = gs.members + 32u;
    *smem = bytes;
    *scratch = need;
    static_assert(sizeof(GridLinkShape) <= 48, "shape buffer");
    std::memcpy(shape_out, &gs, sizeof(gs));
    return true;
}

cudaError_t launch_chain_grid_link(const StepArgs &a, int SB, int P, int grid, uint32_t threads, size_t smem,
                                   const void *shape, void *scratch, cudaStream_t s) {
    GridLinkShape gs;
    std::memcpy(&gs, shape, sizeof(gs));
    // [bitmaps, padded to 256 bytes][link words]: the link runs are read by
    // 16-byte-aligned bulk copies
    const uint64_t words_per_set = (a.n_sessions + 31u) / 32u;
    const size_t bits_bytes = (static_cast<size_t>(a.n_sets) * words_per_set * 4 + 255u) & ~static_cast<size_t>(255u);
    uint32_t *bits = static_cast<uint32_t *>(scratch);
    uint32_t *lnk = reinterpret_cast<uint32_t *>(static_cast<uint8_t *>(scratch) + bits_bytes);
    cudaError_t e = cudaMemsetAsync(bits, 0, static_cast<size_t>(a.n_sets) * words_per_set * 4, s);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const size_t total = static_cast<size_t>(a.n_sets) * a.K;
    const size_t want = (total + 255u) / 256u;
    const unsigned blocks = static_cast<unsigned>(want < static_cast<size_t>(sms) * 8u ? want : static_cast<size_t>(sms) * 8u);
    k_mark<<<blocks ? blocks : 1u, 256, 0, s>>>(a.idx, a.n_sets, a.K, a.n_sessions, words_per_set, bits);
    k_flag<<<blocks ? blocks : 1u, 256, 0, s>>>(a.idx, a.n_sets, a.K, a.n_sessions, words_per_set, bits, lnk);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const TmaShape &sh = gs.t;
    EncodeTiled enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    alignas(64) CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(P), static_cast<cuuint64_t>(a.n_sets) * a.K};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(P)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(P), sh.box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz = P == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                   : P == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                             : CU_TENSOR_MAP_SWIZZLE_32B;
    CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.payload), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    StepArgs aa = a;
    const uint32_t *l = lnk;
    void *args[] = {&map, &aa, &l, &gs};
    return cudaLaunchCooperativeKernel(grid_link_fn(SB, P), dim3(grid), dim3(threads), args, smem, s);
}

namespace {
const void *grid_pair_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_grid_pair<decltype(b)::value, decltype(q)::value>);
    });
}
// Byte offsets of the two-step grid chain's scratch: cohort bitmaps, session
// positions per cohort, link words, the input-state ring and the key ring
// (each part 256-byte aligned).
struct GridPairScratch {
    size_t pos, lnk, xo, keys, total;
};
GridPairScratch grid_pair_scratch(uint32_t K, uint64_t N, uint32_t n_sets) {
    auto up = [](size_t v) { return (v + 255u) & ~static_cast<size_t>(255u); };
    const uint64_t words_per_set = (N + 31u) / 32u;
    GridPairScratch o{};
    o.pos = up(static_cast<size_t>(n_sets) * words_per_set * 4);
    o.lnk = o.pos + up(static_cast<size_t>(n_sets) * N * 2);
    o.xo = o.lnk + up(static_cast<size_t>(n_sets) * K * 8);
    o.keys = o.xo + up(4ull * K * 4);
    o.total = o.keys + up(2ull * K * 8);
    return o;
}
}  // namespace

bool chain_grid_pair_plan(int SB, int P, uint32_t K, uint64_t n_sessions, uint32_t n_sets, uint32_t tab_stride,
                          int *grid, uint32_t *threads, size_t *smem, void *shape_out, size_t *scratch) {
    if (K == 0 || K % 8u != 0u || K > 65536u || n_sessions > 0xFFFFFFFFull || !encode_fn()) return false;
    int dev = 0, sms = 0, max_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return false;
    GridPairShape gs{};
    TmaShape &sh = gs.t;
    const uint32_t per = (K + static_cast<uint32_t>(sms) - 1u) / static_cast<uint32_t>(sms);
    sh.chunk = (per + 7u) & ~7u;
    const uint32_t g = (K + sh.chunk - 1u) / sh.chunk;
    sh.n_boxes = (sh.chunk + 255u) / 256u;
    sh.box_rows = (((sh.chunk + sh.n_boxes - 1u) / sh.n_boxes) + 7u) & ~7u;
    sh.stage_pay = ((sh.n_boxes * sh.box_rows * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
    sh.stage_words = 0;
    gs.members = ((sh.chunk + 31u) / 32u) * 32u;
    if (gs.members + 32u > kGridPairThreads) return false;
    const size_t bytes = 1024 + static_cast<size_t>(kGridPairStages) * sh.stage_pay + 2ull * sh.chunk * SB +
                         ((2ull * tab_stride + 15u) & ~15ull);
    if (bytes > static_cast<size_t>(max_optin)) return false;
    const GridPairScratch o = grid_pair_scratch(K, n_sessions, n_sets);
    if (o.total > (1ull << 30)) return false;
    const void *fn = grid_pair_fn(SB, P);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes)) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, static_cast<int>(gs.members + 32u), bytes) !=
            cudaSuccess ||
        per_sm < 1 || static_cast<long long>(per_sm) * sms < g)
        return false;
    *grid = static_cast<int>(g);
    *threads = gs.members + 32u;
    *smem = bytes;
    *scratch = o.total;
    static_assert(sizeof(GridPairShape) <= 48, "shape buffer");
    std::memcpy(shape_out, &gs, sizeof(gs));
    return true;
}

cudaError_t launch_chain_grid_pair(const StepArgs &a, int SB, int P, int grid, uint32_t threads, size_t smem,
                                   const void *shape, void *scratch, cudaStream_t s) {
    GridPairShape gs;
    std::memcpy(&gs, shape, sizeof(gs));
    const GridPairScratch o = grid_pair_scratch(a.K, a.n_sessions, a.n_sets);
    uint8_t *const base = static_cast<uint8_t *>(scratch);
    uint32_t *bits = reinterpret_cast<uint32_t *>(base);
    uint16_t *pos = reinterpret_cast<uint16_t *>(base + o.pos);
    uint2 *lnk = reinterpret_cast<uint2 *>(base + o.lnk);
    uint32_t *xo = reinterpret_cast<uint32_t *>(base + o.xo);
    unsigned long long *keys = reinterpret_cast<unsigned long long *>(base + o.keys);
    const uint64_t words_per_set = (a.n_sessions + 31u) / 32u;
    cudaError_t e = cudaMemsetAsync(bits, 0, static_cast<size_t>(a.n_sets) * words_per_set * 4, s);
    if (e != cudaSuccess) return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const size_t total = static_cast<size_t>(a.n_sets) * a.K;
    const size_t want = (total + 255u) / 256u;
    const unsigned blocks = static_cast<unsigned>(want < static_cast<size_t>(sms) * 8u ? want : static_cast<size_t>(sms) * 8u);
    k_mark_pos<<<blocks ? blocks : 1u, 256, 0, s>>>(a.idx, a.n_sets, a.K, a.n_sessions, words_per_set, bits, pos);
    k_link_grid2<<<blocks ? blocks : 1u, 256, 0, s>>>(a.idx, a.n_sets, a.K, a.n_sessions, words_per_set, bits, pos,
                                                      lnk);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    alignas(64) CUtensorMap map;
    if (!payload_map(a, P, gs.t.box_rows, &map)) return cudaErrorInvalidValue;
    StepArgs aa = a;
    const uint2 *l = lnk;
    void *args[] = {&map, &aa, &l, &xo, &keys, &gs};
    return cudaLaunchCooperativeKernel(grid_pair_fn(SB, P), dim3(grid), dim3(threads), args, smem, s);
}

namespace {
const void *cluster_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_cluster<decltype(b)::value, decltype(q)::value>);
    });
}
cudaLaunchConfig_t cluster_cfg(uint32_t cluster, uint32_t threads, cudaStream_t s, cudaLaunchAttribute *attr) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(cluster);
    cfg.blockDim = dim3(threads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = cluster;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cfg;
}
}  // namespace

// One cluster of C = ceil(K / 512) CTAs (at most 16, a non-portable size
// above 8); false when the device cannot place such a cluster.
bool chain_cluster_plan(int SB, int P, uint32_t K, uint32_t *cluster, uint32_t *threads) {
    if (K <= 512u || K > 8192u) return false;
    const uint32_t C = (K + 511u) / 512u;
    const uint32_t T = ((K + C - 1u) / C + 31u) / 32u * 32u;
    const void *fn = cluster_fn(SB, P);
    if (C > 8u && cudaFuncSetAttribute(fn, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t cfg = cluster_cfg(C, T, nullptr, attr);
    int n_clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&n_clusters, fn, &cfg) != cudaSuccess || n_clusters < 1) {
        cudaGetLastError();
        return false;
    }
    *cluster = C;
    *threads = T;
    return true;
}

cudaError_t launch_chain_cluster(const StepArgs &a, int SB, int P, uint32_t cluster, uint32_t threads,
                                 cudaStream_t s) {
    cudaLaunchAttribute attr[1];
    cudaLaunchConfig_t cfg = cluster_cfg(cluster, threads, s, attr);
    StepArgs aa = a;
    void *args[] = {&aa};
    return cudaLaunchKernelExC(&cfg, cluster_fn(SB, P), args);
}

static const void *split_fn(int SB, int P) {
    return dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_chain_split<decltype(b)::value, decltype(q)::value>);
    });
}

bool chain_split_plan(int SB, int P, uint32_t K, uint32_t tab_stride, int *grid, uint32_t *threads, size_t *smem,
                      void *shape_out) {
    if (K == 0 || K % 8u != 0u || !encode_fn()) return false;
    int dev = 0, sms = 0, max_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return false;
    TmaShape sh;
    if (K <= 512u) {
        sh.chunk = K;  // one CTA
    } else {
        const uint32_t per = (K + static_cast<uint32_t>(sms) - 1u) / static_cast<uint32_t>(sms);
        sh.chunk = (per + 7u) & ~7u;
        if (sh.chunk > 512u) return false;
    }
    const uint32_t g = (K + sh.chunk - 1u) / sh.chunk;
    sh.n_boxes = (sh.chunk + 255u) / 256u;
    sh.box_rows = (((sh.chunk + sh.n_boxes - 1u) / sh.n_boxes) + 7u) & ~7u;
    sh.stage_pay = ((sh.n_boxes * sh.box_rows * static_cast<uint32_t>(P)) + 1023u) & ~1023u;
    sh.stage_words = (sh.chunk + 3u) & ~3u;
    const size_t bytes = tma_smem_bytes(sh, tab_stride);
    if (bytes + 4096 > static_cast<size_t>(max_optin)) return false;
    const void *fn = split_fn(SB, P);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes)) !=
        cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    const uint32_t thr = ((sh.chunk + 31u) / 32u) * 32u;
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, static_cast<int>(thr), bytes) != cudaSuccess ||
        per_sm < 1 || static_cast<long long>(per_sm) * sms < g)
        return false;
    *grid = static_cast<int>(g);
    *threads = thr;
    *smem = bytes;
    *static_cast<TmaShape *>(shape_out) = sh;
    return true;
}

cudaError_t launch_chain_split(const StepArgs &a, int SB, int P, int grid, uint32_t threads, size_t smem,
                               const void *shape, uint32_t *marks, cudaStream_t s) {
    const TmaShape &sh = *static_cast<const TmaShape *>(shape);
    EncodeTiled enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    alignas(64) CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(P), static_cast<cuuint64_t>(a.n_sets) * a.K};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(P)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(P), sh.box_rows};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz = P == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                   : P == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                             : CU_TENSOR_MAP_SWIZZLE_32B;
    CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(a.payload), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    StepArgs aa = a;
    TmaShape shc = sh;
    uint32_t *mk = marks;
    void *args[] = {&map, &aa, &shc, &mk};
    if (grid == 1) return cudaLaunchKernel(split_fn(SB, P), dim3(1), dim3(threads), args, smem, s);
    return cudaLaunchCooperativeKernel(split_fn(SB, P), dim3(grid), dim3(threads), args, smem, s);
}

static const void *owned_fn(int SB, int P, bool res) {
    return dispatch(SB, P, [&](auto b, auto q) {
        constexpr int B = decltype(b)::value, Q = decltype(q)::value;
        return res ? reinterpret_cast<const void *>(&k_chain_owned<B, Q, true>)
                   : reinterpret_cast<const void *>(&k_chain_owned<B, Q, false>);
    });
}

bool chain_owned_plan(int SB, int P, uint32_t K, uint64_t N, uint32_t tab_stride, int *grid, uint32_t *threads,
                      size_t *smem, void *shape_out) {
    if (K == 0 || !encode_fn()) return false;
    int dev = 0, sms = 0, max_optin = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return false;
    if (cudaDeviceGetAttribute(&max_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess)
        return false;
    OwnedShape sh;
    sh.G = static_cast<uint32_t>(sms);
    sh.per = static_cast<uint32_t>((N + sh.G - 1) / sh.G);
    sh.pad = 0;
    // one member per thread in the common case: room for a quarter more than the mean run
    const uint32_t want = (K + sh.G - 1) / sh.G;
    uint32_t thr = ((want + want / 4u + 31u) / 32u) * 32u;
    if (thr < 32u) thr = 32u;
    if (thr > 512u) thr = 512u;
    // [1024-aligned payload tiles: 2 stages x 2 x 256 rows][tables][record stage][owned states]
    const size_t base = 1024 + 4ull * 256 * P + 2 * static_cast<size_t>(tab_stride);
    const size_t res_bytes = base + static_cast<size_t>(sh.per) * SB;
    const size_t x_bytes = base + static_cast<size_t>(thr) * SB + ((static_cast<size_t>(sh.per) * 2 + 15u) & ~size_t(15));
    sh.res = res_bytes + 2048 <= static_cast<size_t>(max_optin) ? 1u : 0u;
    const size_t bytes = sh.res ? res_bytes : x_bytes;
    if (bytes + 2048 > static_cast<size_t>(max_optin)) return false;
    const void *fn = owned_fn(SB, P, sh.res != 0);
    if (cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes)) !=
        cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, static_cast<int>(thr), bytes) != cudaSuccess ||
        per_sm < 1)
        return false;
    *grid = static_cast<int>(sh.G);
    *threads = thr;
    *smem = bytes;
    *static_cast<OwnedShape *>(shape_out) = sh;
    return true;
}

cudaError_t launch_route(const StepArgs &a, const void *shape, uint32_t *perm_m, uint32_t *perm_s, uint32_t *perm_o,
                         uint32_t *off, cudaStream_t s) {
    const OwnedShape &sh = *static_cast<const OwnedShape *>(shape);
    const size_t smem = (sh.G + 1) * sizeof(uint32_t);
    k_route<<<a.n_sets, 1024, smem, s>>>(a.idx, a.outcome, a.n_sets, a.K, a.n_sessions, sh.G, sh.per, perm_m,
                                          perm_s, perm_o, off, a.dev);
    return cudaGetLastError();
}

cudaError_t launch_permute_payload(const StepArgs &a, int P, const void *shape, const uint32_t *perm_m,
                                   const uint32_t *off, uint8_t *pay_routed, cudaStream_t s) {
    const OwnedShape &sh = *static_cast<const OwnedShape *>(shape);
    int dev = 0, sms = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    k_permute_payload<<<static_cast<unsigned>(sms) * 8u, 256, 0, s>>>(a.payload, perm_m, off, a.n_sets, a.K, sh.G,
                                                                      static_cast<uint32_t>(P), pay_routed);
    return cudaGetLastError();
}

cudaError_t launch_chain_owned(const StepArgs &a, int SB, int P, int grid, uint32_t threads, size_t smem,
                               const void *shape, const uint32_t *perm_m, const uint32_t *perm_s,
                               const uint32_t *perm_o, const uint32_t *off, const uint8_t *pay_routed,
                               cudaStream_t s) {
    const OwnedShape &sh = *static_cast<const OwnedShape *>(shape);
    EncodeTiled enc = encode_fn();
    if (!enc) return cudaErrorNotSupported;
    alignas(64) CUtensorMap map;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(P), static_cast<cuuint64_t>(a.n_sets) * a.K};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(P)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(P), 256u};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle swz = P == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                                   : P == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                             : CU_TENSOR_MAP_SWIZZLE_32B;
    CUresult r = enc(&map, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<uint8_t *>(pay_routed), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, swz, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                     CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cudaErrorInvalidValue;
    StepArgs aa = a;
    OwnedShape shc = sh;
    void *args[] = {&map, &aa, &shc, &perm_m, &perm_s, &perm_o, &off};
    return cudaLaunchCooperativeKernel(owned_fn(SB, P, sh.res != 0), dim3(grid), dim3(threads), args, smem, s);
}

cudaError_t launch_seg_step(const SegArgs &a, int SB, int P, cudaStream_t s) {
    const void *fn = dispatch(SB, P, [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_seg_step<decltype(b)::value, decltype(q)::value>);
    });
    SegArgs aa = a;
    void *args[] = {&aa};
    const uint32_t grid = a.total == 0u ? 1u : (a.total + kStepThreads - 1u) / kStepThreads;
    return cudaLaunchKernel(fn, dim3(grid), dim3(kStepThreads), args, 0, s);
}

cudaError_t launch_empty_cohorts(const StepArgs &a, cudaStream_t s) {
    StepArgs aa = a;
    void *args[] = {&aa};
    return cudaLaunchKernel(reinterpret_cast<const void *>(&k_empty_cohorts), dim3(1), dim3(256), args, 0, s);
}

cudaError_t launch_set_word(uint32_t *p, uint32_t v, cudaStream_t s) {
    k_set_word<<<1, 1, 0, s>>>(p, v);
    return cudaGetLastError();
}

const void *launcher_kernel() { return reinterpret_cast<const void *>(&k_launch_child); }
const void *empty_kernel() { return reinterpret_cast<const void *>(&k_empty); }
const void *countdown_kernel() { return reinterpret_cast<const void *>(&k_countdown); }

cudaError_t launch_grid_barrier_floor(DevBlock *dev, uint32_t n_steps, cudaStream_t s) {
    int d = 0, sms = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&d);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, d);
    const void *fn = reinterpret_cast<const void *>(&k_grid_barrier_floor);
    if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, 480, 0);
    if (e != cudaSuccess) return e;
    if (per_sm < 1) return cudaErrorCooperativeLaunchTooLarge;
    void *args[] = {&dev, &n_steps};
    return cudaLaunchCooperativeKernel(fn, dim3(sms), dim3(480), args, 0, s);
}

// ---------------------------------------------------------------------------
// Allocation-free cohort step (rc_cohort_step_noalloc in include/rc.h).
//
// For callers that must not allocate device memory (the allocator belongs to
// someone else, or allocation is not allowed once the process is serving).
// The only scratch is a file-scope device array: an error latch and a
// last-CTA ticket (a DevBlock) plus one odd count per CTA, summed by the last
// CTA in CTA order.  The array is shared by every call in the process and
// keeps the previous call's contents: the entry point clears the latch words
// on the stream before each launch, and calls that overlap on the GPU race.
// ---------------------------------------------------------------------------
namespace {

constexpr uint32_t kNoAllocMaxCtas = 4096;  // at most 4096 * 256 = 1,048,576 members per call

struct NoAllocScratch {
    DevBlock dev;                       // error latch, ticket (256 bytes)
    uint32_t partial[kNoAllocMaxCtas];  // odd count of each CTA
};

static __device__ __align__(256) NoAllocScratch g_noalloc_scratch;

template <int SB, int P>
__global__ void __launch_bounds__(kStepThreads) k_step_noalloc(StepArgs a, uint32_t *flag, uint32_t *status,
                                                              NoAllocScratch *scr) {
    __shared__ __align__(16) uint8_t tab[256 * 8];
    __shared__ uint32_t warp_odd[kStepThreads / 32];
    __shared__ uint32_t s_sel;
    const uint32_t tid = threadIdx.x;
    if (tid == 0) s_sel = ld_volatile_u32(flag) & 1u;
    __syncthreads();
    const uint32_t sel = s_sel;
    stage_tables(tab, a.tables, a.tab_stride, 1, sel);
    __syncthreads();
    const uint32_t m = blockIdx.x * blockDim.x + tid;
    uint32_t odd = 0;
    if (m < a.K) {
        Event<P> ev;
        load_event<P>(ev, a, 0, m);
        odd = transition<SB, P, false>(a, ev, tab, sel, 0, m);
    }
    const uint32_t ball = __ballot_sync(0xffffffffu, odd);
    if ((tid & 31u) == 0) warp_odd[tid >> 5] = __popc(ball);
    __syncthreads();
    if (tid != 0) return;
    uint32_t c = 0;
    for (uint32_t w = 0; w < (blockDim.x + 31u) / 32u; ++w) c += warp_odd[w];
    scr->partial[blockIdx.x] = c;
    __threadfence();
    const uint32_t ticket = atomicAdd(&scr->dev.ticket, 1u);
    if (ticket != gridDim.x - 1) return;
    __threadfence();
    uint32_t total = 0;
    for (uint32_t b = 0; b < gridDim.x; ++b) total += ld_volatile_u32(&scr->partial[b]);
    scr->dev.ticket = 0u;
    *flag = total > a.K / 2u ? 1u : 0u;
    if (status) *status = ld_volatile_u32(&scr->dev.err);
}

}  // namespace

namespace {
std::mutex g_noalloc_mu;
void *g_noalloc_addr[64];  // device address of g_noalloc_scratch, per device (set-up on first call)
}  // namespace

}  // namespace rc

extern "C" int rc_cohort_step_noalloc(const uint8_t *tables, uint32_t S, uint32_t state_bytes,
                                      uint32_t payload_bytes, void *state, uint64_t n_sessions,
                                      const rc_events *events, uint32_t K, uint32_t *flag, void *effects_out,
                                      uint32_t *status_out, void *cuda_stream) {
    using namespace rc;
    auto a16 = [](const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    if (!tables || !a16(tables) || S < 2 || S > 256 || (S & (S - 1)) != 0) return RC_E_INVAL;
    if ((state_bytes != 16 && state_bytes != 64) || (payload_bytes != 32 && payload_bytes != 64 &&
                                                     payload_bytes != 128))
        return RC_E_INVAL;
    if (!state || !a16(state) || n_sessions < 1 || n_sessions > 0xffffffffull) return RC_E_INVAL;
    if (!flag || (reinterpret_cast<uintptr_t>(flag) & 3u) != 0 || !events || events->payload_bytes != payload_bytes)
        return RC_E_INVAL;
    if (!a16(effects_out) || (reinterpret_cast<uintptr_t>(status_out) & 3u) != 0) return RC_E_INVAL;
    // the scratch array holds one count per CTA: larger cohorts do not fit
    if (K > kNoAllocMaxCtas * static_cast<uint32_t>(kStepThreads)) return RC_E_SIZE;
    if (K > 0 && (!events->outcome || !events->payload || !a16(events->outcome) || !a16(events->payload) ||
                  !a16(events->session_idx)))
        return RC_E_INVAL;
    cudaStream_t stream = static_cast<cudaStream_t>(cuda_stream);
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return RC_E_CUDA;
    void *scr = nullptr;
    {
        std::lock_guard<std::mutex> lock(g_noalloc_mu);
        if (!g_noalloc_addr[dev]) {
            // set-up, once per device, with that device current: the host-side
            // name of a __device__ array is not its device address
            void *p = nullptr;
            if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return RC_E_CUDA;
            g_noalloc_addr[dev] = p;
        }
        scr = g_noalloc_addr[dev];
    }
    NoAllocScratch *ns = static_cast<NoAllocScratch *>(scr);
    // the latch and the ticket must start at zero; the array keeps the last call's contents
    if (cudaMemsetAsync(&ns->dev, 0, sizeof(DevBlock), stream) != cudaSuccess) return RC_E_CUDA;
    if (K == 0) {
        if (cudaMemsetAsync(flag, 0, sizeof(uint32_t), stream) != cudaSuccess) return RC_E_CUDA;
        if (status_out && cudaMemsetAsync(status_out, 0, sizeof(uint32_t), stream) != cudaSuccess) return RC_E_CUDA;
        return RC_OK;
    }
    StepArgs a;
    std::memset(&a, 0, sizeof(a));
    a.state = static_cast<uint8_t *>(state);
    a.n_sessions = n_sessions;
    a.outcome = events->outcome;
    a.payload = events->payload;
    a.idx = events->session_idx;
    a.n_sets = 1;
    a.K = K;
    a.tables = tables;
    a.S = S;
    a.tab_stride = S * 8u;
    a.effects = static_cast<uint8_t *>(effects_out);
    a.n_steps = 1;
    a.dev = &ns->dev;
    const void *fn = dispatch(static_cast<int>(state_bytes), static_cast<int>(payload_bytes), [](auto b, auto q) {
        return reinterpret_cast<const void *>(&k_step_noalloc<decltype(b)::value, decltype(q)::value>);
    });
    void *args[] = {&a, &flag, &status_out, &ns};
    if (cudaLaunchKernel(fn, step_grid(K), step_block(K), args, 0, stream) != cudaSuccess) return RC_E_CUDA;
    return RC_OK;
}
