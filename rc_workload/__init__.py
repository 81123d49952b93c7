"""Seeded synthetic inputs for the ready-cohort transition path.

This module is the one piece of code that both the CPU oracle (``oracle/``) and
the CUDA path (``paper_2608_12123_gb300``) consume.  It draws numbers and lays
them out; it holds none of the method's arithmetic (no route key, no
transition, no decision, no cohort forming, no F / P* / U).

Random numbers come from the SplitMix64 generator of Steele, Lea and Flood
("Fast splittable pseudorandom number generators", OOPSLA 2014), used in its
counter form: the n-th output (n = 1, 2, ...) of the stream seeded with ``s`` is
``fin(s + n * gamma)`` with gamma = 0x9E3779B97F4A7C15 and ``fin`` the
generator's output finaliser.  Every array below is a pure function of
(config id, purpose, index) through :func:`stream_seed`, so any part can be
regenerated without the rest.

Workload shapes follow the paper's two studies:

* cohort events (Section 7.1): a per-session state record, an outcome code per
  event and a random payload; tables of an S-state automaton, one per route body;
* Poisson replay (Section 5.2): sessions arrive as a homogeneous Poisson process,
  each session copies a template drawn uniformly from a fixed panel, the arrival
  rate is the target active population C divided by the mean template duration,
  arrivals start one maximum template duration before the retained interval,
  and the retained interval is [0, 60 s) on an integer-nanosecond clock
  (Section 4, "Exact clock").  The public trace panel the paper replays is not
  available; templates are drawn here from the stated distributions instead
  (geometric span count with mean 10.6, log-normal gaps with median 200 ms and
  sigma 1.5, 70 route labels with Zipf(1) frequencies).
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

__all__ = [
    "GAMMA", "ROOT_SEED", "Purpose", "stream_seed", "splitmix64", "uniform01",
    "make_tables", "make_state", "make_cohort_events", "sample_without_replacement",
    "Panel", "make_panel", "Arrivals", "make_arrivals", "payload_for_events",
    "CONFIGS", "STATE_FIELDS",
]

GAMMA = 0x9E3779B97F4A7C15
ROOT_SEED = 20260811            # the replay root seed of Section 5.2
_M64 = (1 << 64) - 1
_U64 = np.uint64


class Purpose:
    """Stream tags: each kind of draw has a stream of its own."""
    TABLE = 1
    STATE = 2
    OUTCOME = 3
    PAYLOAD = 4
    INDEX = 5
    PANEL_SPANS = 6
    PANEL_GAPS = 7
    PANEL_LABELS = 8
    ARRIVALS = 9
    TEMPLATE_PICK = 10
    EVENT_PAYLOAD = 11


def stream_seed(config_id: int, purpose: int, index: int = 0, root: int = ROOT_SEED) -> int:
    """Seed of the stream for (config, purpose, index); distinct tuples give
    distinct seeds that are far apart in the gamma-lattice."""
    return (root ^ (config_id << 56) ^ (purpose << 48) ^ (index * 0x100000001)) & _M64


def _fin(z: np.ndarray) -> np.ndarray:
    # SplitMix64 output finaliser (Steele, Lea and Flood 2014), on uint64 lanes.
    z = z ^ (z >> _U64(30))
    z = z * _U64(0xBF58476D1CE4E5B9)
    z = z ^ (z >> _U64(27))
    z = z * _U64(0x94D049BB133111EB)
    return z ^ (z >> _U64(31))


def splitmix64(seed: int, n: int, offset: int = 0) -> np.ndarray:
    """Outputs offset+1 .. offset+n of the SplitMix64 stream seeded ``seed``."""
    with np.errstate(over="ignore"):
        k = np.arange(offset + 1, offset + n + 1, dtype=np.uint64)
        return _fin(_U64(seed & _M64) + k * _U64(GAMMA))


def uniform01(words: np.ndarray) -> np.ndarray:
    """Doubles in [0, 1) from the top 53 bits of each word."""
    return (words >> _U64(11)).astype(np.float64) * (1.0 / 9007199254740992.0)


def _uniform_open0(words: np.ndarray) -> np.ndarray:
    """Doubles in (0, 1]: safe arguments for log."""
    return ((words >> _U64(11)).astype(np.float64) + 1.0) * (1.0 / 9007199254740992.0)


def _round_half_up(x: np.ndarray) -> np.ndarray:
    return np.floor(x + 0.5).astype(np.int64)


# ----------------------------------------------------------------------------
# Cohort-step inputs
# ----------------------------------------------------------------------------

#: byte layout of the per-session state record for each record size
STATE_FIELDS = {
    16: (("state", "<i4", 0), ("step", "<u4", 4), ("acc", "<u8", 8)),
    64: (("state", "<i4", 0), ("step", "<u4", 4), ("acc", "<u8", 8, 7)),
}


def make_tables(S: int, seed: int) -> np.ndarray:
    """Two transition tables (route bodies A then B) of an S-state automaton
    over 8 outcome classes: uint8 [2][S][8], entries drawn as ``word & (S-1)``.
    S must be a power of two no larger than 256."""
    if S < 1 or S > 256 or (S & (S - 1)) != 0:
        raise ValueError("S must be a power of two in [1, 256]")
    w = splitmix64(seed, 2 * S * 8)
    return (w & _U64(S - 1)).astype(np.uint8).reshape(2, S, 8)


def make_state(N: int, S: int, state_bytes: int, seed: int) -> np.ndarray:
    """N initial state records (uint8 [N][state_bytes]), little-endian.

    Each record draws its state (``word & (S-1)``) and then its accumulator
    word(s) from one stream, in session order; the step counter starts at 0."""
    if state_bytes not in STATE_FIELDS:
        raise ValueError("state_bytes must be 16 or 64")
    n_acc = 1 if state_bytes == 16 else 7
    w = splitmix64(seed, N * (1 + n_acc)).reshape(N, 1 + n_acc)
    rec = np.zeros((N, state_bytes // 4), dtype=np.uint32)
    rec[:, 0] = (w[:, 0] & _U64(S - 1)).astype(np.uint32)
    acc = np.ascontiguousarray(w[:, 1:])
    rec[:, 2:2 + 2 * n_acc] = acc.view(np.uint32).reshape(N, 2 * n_acc)
    return rec.view(np.uint8).reshape(N, state_bytes)


def sample_without_replacement(N: int, K: int, seed: int) -> np.ndarray:
    """K distinct session indices out of N, uniformly, in random order.

    Each index gets a random sort key whose low 20+ bits hold the index itself,
    so keys are distinct and the order is a pure function of the seed; the K
    smallest keys are taken in key order."""
    if K > N:
        raise ValueError("K > N")
    bits = max(1, int(N - 1).bit_length())
    w = splitmix64(seed, N)
    keys = ((w >> _U64(bits)) << _U64(bits)) | np.arange(N, dtype=np.uint64)
    if K == N:
        part = np.arange(N)
    else:
        part = np.argpartition(keys, K - 1)[:K]
    order = np.argsort(keys[part], kind="stable")
    return part[order].astype(np.uint32)


def make_cohort_events(config_id: int, n_sets: int, K: int, payload_bytes: int,
                       n_sessions: int | None = None, set_offset: int = 0):
    """Event sets for ``n_sets`` cohorts of K members.

    Returns (outcome uint32 [n_sets][K], payload uint8 [n_sets][K][P],
    session_idx uint32 [n_sets][K] or None).  Outcomes are uniform over the 8
    classes; payloads are little-endian random words.  With ``n_sessions``
    given, each cohort draws K distinct sessions out of n_sessions; without it
    member m is session m."""
    if payload_bytes % 8:
        raise ValueError("payload_bytes must be a multiple of 8")
    outc = np.empty((n_sets, K), dtype=np.uint32)
    pay = np.empty((n_sets, K, payload_bytes), dtype=np.uint8)
    idx = None if n_sessions is None else np.empty((n_sets, K), dtype=np.uint32)
    nw = payload_bytes // 8
    for j in range(n_sets):
        g = set_offset + j
        outc[j] = (splitmix64(stream_seed(config_id, Purpose.OUTCOME, g), K) & _U64(7)).astype(np.uint32)
        if nw:
            pay[j] = splitmix64(stream_seed(config_id, Purpose.PAYLOAD, g), K * nw).view(np.uint8).reshape(K, payload_bytes)
        if idx is not None:
            idx[j] = sample_without_replacement(n_sessions, K, stream_seed(config_id, Purpose.INDEX, g))
    return outc, pay, idx


# ----------------------------------------------------------------------------
# Poisson replay of a template panel (Section 5.2)
# ----------------------------------------------------------------------------

@dataclasses.dataclass
class Panel:
    """Session templates: template j has spans span_start[j]..span_start[j+1]-1,
    with completion offsets (ns after the session's arrival) and route labels."""
    span_start: np.ndarray   # int64 [n_templates + 1]
    offset_ns: np.ndarray    # int64 [n_spans], non-decreasing within a template
    label: np.ndarray        # uint32 [n_spans]
    n_labels: int

    @property
    def n_templates(self) -> int:
        return len(self.span_start) - 1

    @property
    def duration_ns(self) -> np.ndarray:
        return self.offset_ns[self.span_start[1:] - 1]


def make_panel(n_templates: int = 851, mean_spans: float = 10.6, median_gap_s: float = 0.2,
               sigma: float = 1.5, n_labels: int = 70, zipf_s: float = 1.0,
               config_id: int = 2) -> Panel:
    """A synthetic panel shaped like the paper's (851 sessions, about 9,000 spans,
    70 route labels).  Span counts are geometric on {1, 2, ...} with the given
    mean (inverse CDF); gaps are log-normal (Box-Muller); labels follow Zipf(s)
    over n_labels values (inverse CDF).  A session with n spans has n gaps: the
    first span completes one gap after the arrival."""
    p = 1.0 / mean_spans
    u = _uniform_open0(splitmix64(stream_seed(config_id, Purpose.PANEL_SPANS), n_templates))
    n_spans = 1 + np.floor(np.log(u) / math.log1p(-p)).astype(np.int64)
    total = int(n_spans.sum())
    gw = splitmix64(stream_seed(config_id, Purpose.PANEL_GAPS), 2 * total).reshape(total, 2)
    u1 = _uniform_open0(gw[:, 0])
    u2 = uniform01(gw[:, 1])
    z = np.sqrt(-2.0 * np.log(u1)) * np.cos(2.0 * math.pi * u2)
    gaps_s = np.exp(math.log(median_gap_s) + sigma * z)
    span_start = np.zeros(n_templates + 1, dtype=np.int64)
    np.cumsum(n_spans, out=span_start[1:])
    cum = np.cumsum(gaps_s)
    base = np.repeat(np.concatenate(([0.0], cum[span_start[1:-1] - 1])), n_spans)
    offset_ns = _round_half_up((cum - base) * 1e9)
    w = 1.0 / np.power(np.arange(1, n_labels + 1, dtype=np.float64), zipf_s)
    cdf = np.cumsum(w) / w.sum()
    ul = uniform01(splitmix64(stream_seed(config_id, Purpose.PANEL_LABELS), total))
    label = np.minimum(np.searchsorted(cdf, ul, side="right"), n_labels - 1).astype(np.uint32)
    return Panel(span_start, offset_ns, label, n_labels)


@dataclasses.dataclass
class Arrivals:
    """Retained events E on the integer-ns clock, in (t, event_id) order.

    event_id is the position in this order; session is a compact index over the
    sessions that own at least one retained event."""
    t_ns: np.ndarray        # int64 [n]
    route: np.ndarray       # uint32 [n]  (template label)
    session: np.ndarray     # uint32 [n]
    n_sessions: int
    horizon_ns: int
    lam_per_s: float
    warmup_ns: int

    @property
    def n(self) -> int:
        return len(self.t_ns)


def make_arrivals(C: float, panel: Panel, horizon_s: float = 60.0, config_id: int = 2,
                  seed_index: int = 0) -> Arrivals:
    """Stationary Poisson replay: rate C / mean template duration, arrivals from
    -max template duration to the horizon, every span completion is an event,
    events with t in [0, horizon) are retained."""
    dur = panel.duration_ns.astype(np.float64) * 1e-9
    lam = C / float(dur.mean())
    warm = float(dur.max())
    t0 = -warm
    span = horizon_s + warm
    n_exp = int(lam * span * 1.05 + 10 * math.sqrt(lam * span) + 64)
    seed = stream_seed(config_id, Purpose.ARRIVALS, seed_index)
    arr = np.empty(0, dtype=np.float64)
    drawn = 0
    last = t0
    chunks = []
    while last < horizon_s:
        u = _uniform_open0(splitmix64(seed, n_exp, offset=drawn))
        drawn += n_exp
        a = last + np.cumsum(-np.log(u) / lam)
        chunks.append(a)
        last = float(a[-1])
    arr = np.concatenate(chunks)
    arr = arr[arr < horizon_s]
    n_sess = len(arr)
    pick = splitmix64(stream_seed(config_id, Purpose.TEMPLATE_PICK, seed_index), n_sess)
    tmpl = ((pick >> _U64(11)).astype(np.float64) * (1.0 / 9007199254740992.0) * panel.n_templates).astype(np.int64)
    tmpl = np.minimum(tmpl, panel.n_templates - 1)
    arr_ns = _round_half_up(arr * 1e9)
    counts = panel.span_start[tmpl + 1] - panel.span_start[tmpl]
    total = int(counts.sum())
    sess_of = np.repeat(np.arange(n_sess, dtype=np.int64), counts)
    first = np.repeat(panel.span_start[tmpl], counts)
    within = np.arange(total, dtype=np.int64) - np.repeat(np.cumsum(counts) - counts, counts)
    span_ix = first + within
    t = arr_ns[sess_of] + panel.offset_ns[span_ix]
    horizon_ns = int(round(horizon_s * 1e9))
    keep = (t >= 0) & (t < horizon_ns)
    t = t[keep]
    sess_of = sess_of[keep]
    route = panel.label[span_ix[keep]]
    # (t, generation order) is a strict order: stable sort on t keeps generation order on ties.
    order = np.argsort(t, kind="stable")
    t = t[order]
    route = route[order]
    sess_of = sess_of[order]
    present = np.zeros(n_sess, dtype=np.int64)
    present[sess_of] = 1
    remap = np.cumsum(present) - 1
    compact = remap[sess_of]
    return Arrivals(t.astype(np.int64), route.astype(np.uint32), compact.astype(np.uint32),
                    int(present.sum()), horizon_ns, lam, int(round(warm * 1e9)))


def payload_for_events(event_ids: np.ndarray, payload_bytes: int, config_id: int = 2,
                       seed_index: int = 0) -> np.ndarray:
    """Payload bytes of the given retained events: event e owns words
    e*P/8 .. (e+1)*P/8-1 of its stream, so any subset is drawn directly."""
    nw = payload_bytes // 8
    seed = stream_seed(config_id, Purpose.EVENT_PAYLOAD, seed_index)
    ev = np.asarray(event_ids, dtype=np.uint64).reshape(-1)
    with np.errstate(over="ignore"):
        k = (ev[:, None] * _U64(nw) + np.arange(1, nw + 1, dtype=np.uint64)[None, :])
        words = _fin(_U64(seed) + k * _U64(GAMMA))
    return np.ascontiguousarray(words).view(np.uint8).reshape(len(ev), payload_bytes)


# ----------------------------------------------------------------------------
# The five workloads (shapes of the paper's studies, at the sizes measured here)
# ----------------------------------------------------------------------------

CONFIGS = {
    1: dict(name="tiny chain", K=32, S=16, state_bytes=16, payload_bytes=32, n_steps=1000,
            identity=True),
    2: dict(name="primary cohort replay", C=100_000, K=256, delta_ns=50_000_000, S=64,
            state_bytes=16, payload_bytes=64, horizon_s=60.0),
    3: dict(name="deadline and capacity sweep", C=(10_000, 100_000), K=(32, 64, 128, 256),
            delta_ns=50_000_000, S=64, state_bytes=16, payload_bytes=64, n_invocations=1000,
            reps=100),
    4: dict(name="bandwidth-bound large cohort", N=1_048_576, K=65_536, S=256, state_bytes=64,
            payload_bytes=128, n_steps=1000, n_sets=64),
    5: dict(name="long decision chain", K=256, S=128, state_bytes=16, payload_bytes=32,
            n_steps=10_000, seeds=50, identity=True),
}
