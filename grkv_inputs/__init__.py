"""Seeded synthetic KV caches for the GRKV prefill compression path.

This module only draws random inputs.  It holds none of the method's
arithmetic: no attention, no pooling, no selection and no regression.  Both
the fp64 CPU oracle (through the tests and the bench's CPU baseline) and the
CUDA library consume the arrays produced here.

Layout of one *unit* (one layer x KV head of one sequence):

    q : [g][w][d]   the window queries of the g query heads sharing this KV head
    k : [n][d]      full key cache
    v : [n][d]      full value cache

Every unit has its own Philox4x32-10 stream keyed by (workload seed, unit), so
any unit can be regenerated alone.  Values are drawn in fp32 and rounded once
to the workload dtype (round-to-nearest-even); the queries are built from the
*rounded* keys.  `unit_arrays` returns the rounded values as float32 arrays,
which hold bf16 values exactly when the dtype is bf16.

Recipes (the paper's workloads, LongBench and RULER, are not available; these
stand in for them with the cache shapes of the models the paper evaluates):

* ``lowrank``   K = (A[n x 16] @ G[16 x d]) / 4 + 0.1 E,  V ~ N(0, 1),
                 each window query row = 2 * K[r] + 0.5 N(0, 1) with r uniform.
* ``outlier``   ``lowrank`` keys with 4 channels per unit scaled x10 after
                 construction (the outlier channels of real key caches).
* ``spans``     ``lowrank`` keys plus 16 non-overlapping spans of 256 tokens
                 whose keys are rotated to cosine 0.8 with a per-unit topic
                 vector t; window queries are 2 sqrt(d) t + 0.5 N(0, 1).
"""
from __future__ import annotations

import concurrent.futures as _cf
import dataclasses
import os

import numpy as np

__all__ = [
    "Workload", "workload", "WORKLOADS", "sweep_points", "unit_arrays",
    "fill_units", "bf16_bits", "bf16_value", "seed_for", "heldout_queries",
]

BASE_SEED = 0x47524B56  # "GRKV"


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    units: int          # U: batch x layers x KV heads
    group: int          # g: query heads per KV head
    n: int              # context tokens, window included
    d: int              # head dimension
    window: int         # w
    budget: int         # B, window included
    pool_kernel: int
    lambda_v: float
    dtype: str          # "f32" or "bf16"
    recipe: str         # "lowrank" | "outlier" | "spans"
    seed: int

    @property
    def m(self) -> int:
        return self.group * self.window

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


def seed_for(base: int, *mix: int) -> int:
    s = int(base) & 0xFFFFFFFFFFFF
    for x in mix:
        s = (s * 1000003 + int(x)) & 0xFFFFFFFFFFFFFFFF
    return s


# The five synthetic workloads.  Shapes: Llama-3.1-8B (32 layers, 32 query
# heads over 8 KV heads, d = 128) and Mistral-7B (same head layout).
WORKLOADS = {
    "c0_single_head_f32": Workload("c0_single_head_f32", 1, 1, 2048, 128, 32, 256, 7, 1e-2,
                                   "f32", "lowrank", BASE_SEED + 0),
    "c1_llama_layer_bf16": Workload("c1_llama_layer_bf16", 8, 4, 8192, 128, 32, 512, 7, 1e-2,
                                    "bf16", "lowrank", BASE_SEED + 1),
    "c2_llama_32k_bf16": Workload("c2_llama_32k_bf16", 256, 4, 32768, 128, 32, 2048, 7, 1e-2,
                                  "bf16", "outlier", BASE_SEED + 2),
    "c3_mistral_128k_bf16": Workload("c3_mistral_128k_bf16", 256, 4, 131072, 128, 64, 1024, 7,
                                     1e-1, "bf16", "spans", BASE_SEED + 3),
    "c4_sweep_bf16": Workload("c4_sweep_bf16", 32, 4, 16384, 128, 32, 2048, 7, 1e-2,
                              "bf16", "outlier", BASE_SEED + 4),
}
_ORDER = list(WORKLOADS)

SWEEP_N = (4096, 16384, 65536, 131072)
SWEEP_B = (128, 256, 512, 1024, 2048)


def workload(i_or_name) -> Workload:
    if isinstance(i_or_name, int):
        return WORKLOADS[_ORDER[i_or_name]]
    return WORKLOADS[i_or_name]


def sweep_points():
    """The (n, budget) grid of the batch-4 sweep, each with its own seed."""
    base = WORKLOADS["c4_sweep_bf16"]
    for n in SWEEP_N:
        for b in SWEEP_B:
            yield base.replace(name=f"c4_sweep_bf16_n{n}_b{b}", n=n, budget=b,
                               seed=seed_for(base.seed, n, b))


# ---------------------------------------------------------------- rounding --
def bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = (b + (np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1)))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_value(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> the exact fp32 values."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def _round(x: np.ndarray, dtype: str) -> np.ndarray:
    x = np.asarray(x, dtype=np.float32)
    if dtype == "bf16":
        return bf16_value(bf16_bits(x))
    return x


# ---------------------------------------------------------------- recipes --
def _rng(wl: Workload, unit: int) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(np.random.SeedSequence([wl.seed, unit])))


def _lowrank_keys(g: np.random.Generator, n: int, d: int) -> np.ndarray:
    a = g.standard_normal((n, 16), dtype=np.float32)
    b = g.standard_normal((16, d), dtype=np.float32)
    k = a @ b
    k *= np.float32(0.25)
    e = g.standard_normal((n, d), dtype=np.float32)
    e *= np.float32(0.1)
    k += e
    return k


def unit_arrays(wl: Workload, unit: int):
    """(q [g][w][d], k [n][d], v [n][d]) of one unit as float32 arrays whose
    values are exactly representable in the workload dtype."""
    return _unit_draw(wl, unit)[:3]


def heldout_queries(wl: Workload, unit: int, count: int) -> np.ndarray:
    """count held-out decoding queries per query head of one unit, [g][count][d]
    float32 (dtype-exact): drawn like the window queries (noisy copies of
    random keys, or of the unit's topic direction for the span recipe) from
    a stream of their own, so that they are not the surrogate window."""
    _, k, _, topic = _unit_draw(wl, unit)
    g = np.random.Generator(np.random.Philox(np.random.SeedSequence([wl.seed, unit, 0x484F4C44])))
    noise = g.standard_normal((wl.group, count, wl.d), dtype=np.float32) * np.float32(0.5)
    if topic is not None:
        q = (2.0 * np.sqrt(wl.d) * topic).astype(np.float32)[None, None, :] + noise
    else:
        rows = g.integers(0, wl.n, size=(wl.group, count))
        q = np.float32(2.0) * k[rows] + noise
    return _round(q, wl.dtype)


def _unit_draw(wl: Workload, unit: int):
    g = _rng(wl, unit)
    n, d, w, grp = wl.n, wl.d, wl.window, wl.group
    k = _lowrank_keys(g, n, d)
    if wl.recipe == "outlier":
        ch = g.choice(d, size=4, replace=False)
        k[:, ch] *= np.float32(10.0)
    topic = None
    if wl.recipe == "spans":
        topic = g.standard_normal(d).astype(np.float64)
        topic /= np.linalg.norm(topic)
        span, nspan = 256, 16
        room = n - w - span - (nspan - 1) * span
        if room > nspan:
            starts = np.sort(g.choice(room, size=nspan, replace=False)) + np.arange(nspan) * span
            for s0 in starts:
                blk = k[s0:s0 + span].astype(np.float64)
                norm = np.linalg.norm(blk, axis=1, keepdims=True)
                orth = blk - (blk @ topic)[:, None] * topic[None, :]
                orth /= np.maximum(np.linalg.norm(orth, axis=1, keepdims=True), 1e-30)
                k[s0:s0 + span] = (norm * (0.8 * topic[None, :] + 0.6 * orth)).astype(np.float32)
    k = _round(k, wl.dtype)
    v = _round(g.standard_normal((n, d), dtype=np.float32), wl.dtype)
    noise = g.standard_normal((grp, w, d), dtype=np.float32) * np.float32(0.5)
    if wl.recipe == "spans":
        q = (2.0 * np.sqrt(d) * topic).astype(np.float32)[None, None, :] + noise
    else:
        rows = g.integers(0, n, size=(grp, w))
        q = np.float32(2.0) * k[rows] + noise
    q = _round(q, wl.dtype)
    return q, k, v, topic


def _store(dst: np.ndarray, x: np.ndarray, dtype: str):
    if dtype == "bf16":
        dst[...] = bf16_bits(x)
    else:
        dst[...] = x


def fill_units(wl: Workload, q_out, k_out, v_out, units=None, threads=None):
    """Write units into caller buffers shaped [U][g][w][d] and [U][n][d].

    The buffers hold bf16 bit patterns (uint16) for bf16 workloads and
    float32 otherwise.  `units` selects which unit indices to fill (default
    all); unit i of the selection is written to slot i of the buffers.
    """
    units = list(range(wl.units)) if units is None else list(units)
    threads = threads or min(32, os.cpu_count() or 1)

    def one(slot_u):
        slot, u = slot_u
        q, k, v = unit_arrays(wl, u)
        _store(q_out[slot], q, wl.dtype)
        _store(k_out[slot], k, wl.dtype)
        _store(v_out[slot], v, wl.dtype)

    with _cf.ThreadPoolExecutor(max_workers=threads) as ex:
        list(ex.map(one, enumerate(units)))
