"""Seeded synthetic workloads for the MeanField joint-configuration scorer.

This module only draws inputs.  It holds none of the method's arithmetic (no
decode, no aggregate, no predictor, no objective), so both the CUDA path and the
CPU oracle can take their inputs from it without sharing any computation.

Every number is drawn from a counter-based SplitMix64 stream (Steele, Lea and
Flood, "Fast splittable pseudorandom number generators", OOPSLA 2014): output j
of a stream with key s is the SplitMix64 finaliser applied to
s + (j + 1) * 0x9E3779B97F4A7C15.  A stream's key is derived from
(seed, purpose, model), so every array is reproducible bit for bit on any
machine.  A uniform draw on [lo, hi) takes the top 24 bits of the 64-bit
output, u = (z >> 40) * 2**-24, computes lo + (hi - lo) * u in float64 and
rounds to float32.

The shapes and distributions follow the paper's setting (Sec. II: per-model
discrete option spaces, Eq. 1 joint space; Sec. III-B, Eq. 6: one predictor
per model on local configuration plus aggregate GPU state; Sec. IV-C: N = 5
with 78,732 joint configurations) with the synthetic parameters below standing
in for the profiled LLM/YOLO landscape, which is not available:

* local features ~ U(0, 1), d_local per model;
* demand per option: SM share ~ U(0.05, 0.6), VRAM GB ~ U(1, 20),
  bandwidth GB/s ~ U(50, 1500);
* predictor weights: Xavier/Glorot uniform U(+-sqrt(6 / (fan_in + fan_out)));
  biases ~ U(+-1 / sqrt(fan_in)); one distinct MLP per model;
* SLA latency ceilings ~ U(0.5, 2.0); objective weights ~ U(0.5, 1.5);
* the "tight" variant draws SLA ~ U(0.1, 0.9) (TIGHT_SLA) so that the latency mask binds
  on part of the space (the synthetic predictors' latencies are of order 0-0.7; which
  scenario seeds leave a feasible fraction strictly between 0 and 1 is checked by the
  tests that use them).

Predictor weights of model i are packed, PyTorch ``Linear`` convention
(weight[out][in]), as W1[h1][d_in], b1[h1], (W2[h2][h1], b2[h2] if h2 > 0),
W3[2][h_last], b3[2], with d_in = d_local + 4.
"""
from __future__ import annotations

import numpy as np

_M64 = (1 << 64) - 1
GAMMA = 0x9E3779B97F4A7C15

# stream purposes (part of the key derivation; changing them changes every input)
P_LOCAL, P_SM, P_VRAM, P_BW, P_W1, P_B1, P_W2, P_B2, P_W3, P_B3, P_SLA, P_OBJW = range(1, 13)


def _mix_np(z: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser on a uint64 array (wrapping arithmetic)."""
    z = z.astype(np.uint64, copy=True)
    with np.errstate(over="ignore"):
        z ^= z >> np.uint64(30)
        z *= np.uint64(0xBF58476D1CE4E5B9)
        z ^= z >> np.uint64(27)
        z *= np.uint64(0x94D049BB133111EB)
        z ^= z >> np.uint64(31)
    return z


def _mix_int(x: int) -> int:
    return int(_mix_np(np.array([x & _M64], dtype=np.uint64))[0])


def stream_key(seed: int, purpose: int, model: int) -> int:
    """Key of the stream for (seed, purpose, model)."""
    return _mix_int(_mix_int(seed) ^ ((purpose << 32) | model))


def stream_u64(key: int, n: int) -> np.ndarray:
    """Outputs 0..n-1 of the SplitMix64 sequence whose state starts at ``key``."""
    ctr = np.arange(1, n + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        state = np.uint64(key) + ctr * np.uint64(GAMMA)
    return _mix_np(state)


def uniform(seed: int, purpose: int, model: int, n: int, lo: float, hi: float) -> np.ndarray:
    z = stream_u64(stream_key(seed, purpose, model), n)
    u = (z >> np.uint64(40)).astype(np.float64) * (2.0 ** -24)
    return (lo + (hi - lo) * u).astype(np.float32)


def param_count(d_local: int, h1: int, h2: int) -> int:
    d_in = d_local + 4
    n = h1 * d_in + h1
    last = h1
    if h2 > 0:
        n += h2 * h1 + h2
        last = h2
    return n + 2 * last + 2


def _xavier(seed, purpose, model, fan_out, fan_in):
    lim = np.sqrt(6.0 / (fan_in + fan_out))
    return uniform(seed, purpose, model, fan_out * fan_in, -lim, lim)


def _bias(seed, purpose, model, fan_out, fan_in):
    lim = 1.0 / np.sqrt(fan_in)
    return uniform(seed, purpose, model, fan_out, -lim, lim)


def draw_weights(seed: int, model: int, d_local: int, h1: int, h2: int) -> np.ndarray:
    d_in = d_local + 4
    parts = [_xavier(seed, P_W1, model, h1, d_in), _bias(seed, P_B1, model, h1, d_in)]
    last = h1
    if h2 > 0:
        parts += [_xavier(seed, P_W2, model, h2, h1), _bias(seed, P_B2, model, h2, h1)]
        last = h2
    parts += [_xavier(seed, P_W3, model, 2, last), _bias(seed, P_B3, model, 2, last)]
    w = np.concatenate(parts).astype(np.float32)
    assert w.size == param_count(d_local, h1, h2)
    return w


def default_agg_scale(n_models: int) -> np.ndarray:
    """Feature scaling of the aggregate (Sigma SM, Sigma VRAM, Sigma BW, N): each ~[0, 1]."""
    n = float(n_models)
    return np.array([1.0 / (0.6 * n), 1.0 / (20.0 * n), 1.0 / (1500.0 * n), 1.0 / 8.0],
                    dtype=np.float32)


def make_problem(n_options, d_local, h1, h2, seed, vram_cap, objective="weighted_thr",
                 soft_penalty=0.0, out_act="identity", precision="fp32",
                 sla_range=(0.5, 2.0), scenario_seed=None) -> dict:
    """Draw a full problem.  ``scenario_seed`` (default ``seed``) drives SLA and weights w_i."""
    n_options = np.asarray(n_options, dtype=np.int32)
    n = int(n_options.size)
    locs, dems, ws = [], [], []
    for i in range(n):
        k = int(n_options[i])
        locs.append(uniform(seed, P_LOCAL, i, k * d_local, 0.0, 1.0).reshape(k, d_local))
        dem = np.stack([uniform(seed, P_SM, i, k, 0.05, 0.6),
                        uniform(seed, P_VRAM, i, k, 1.0, 20.0),
                        uniform(seed, P_BW, i, k, 50.0, 1500.0)], axis=1)
        dems.append(dem.astype(np.float32))
        ws.append(draw_weights(seed, i, d_local, h1, h2))
    prob = dict(
        n_options=n_options, d_local=int(d_local), hidden1=int(h1), hidden2=int(h2),
        local_feats=np.ascontiguousarray(np.concatenate(locs, axis=0), dtype=np.float32),
        demand=np.ascontiguousarray(np.concatenate(dems, axis=0), dtype=np.float32),
        weights=np.ascontiguousarray(np.concatenate(ws), dtype=np.float32),
        agg_scale=default_agg_scale(n),
        vram_cap=float(vram_cap), soft_penalty=float(soft_penalty),
        objective=objective, out_act=out_act, precision=precision,
    )
    set_scenario(prob, seed if scenario_seed is None else scenario_seed, sla_range)
    return prob


# SLA ceilings under which the latency mask binds on part of a space.
TIGHT_SLA = (0.1, 0.9)


def set_scenario(prob: dict, scenario_seed: int, sla_range=(0.5, 2.0)) -> dict:
    """Redraw the SLA ceilings and objective weights (the per-scenario inputs)."""
    n = int(prob["n_options"].size)
    prob["sla"] = uniform(scenario_seed, P_SLA, 0, n, sla_range[0], sla_range[1])
    prob["obj_w"] = uniform(scenario_seed, P_OBJW, 0, n, 0.5, 1.5)
    prob["scenario_seed"] = int(scenario_seed)
    return prob


# ---------------------------------------------------------------------------
# Named workloads (shapes of the benchmark configurations).
# ---------------------------------------------------------------------------

def tiny(seed: int = 1, **kw) -> dict:
    """N = 2, options (12, 18) -> 216 joint configs, 12->32->2, VRAM cap 24 GB."""
    return make_problem([12, 18], 8, 32, 0, seed, 24.0, **kw)


def paper_scale(seed: int = 2, **kw) -> dict:
    """N = 5, options (12, 9, 9, 9, 9) -> 78,732 joint configs, 12->64->64->2, cap 180 GB."""
    return make_problem([12, 9, 9, 9, 9], 8, 64, 64, seed, 180.0, **kw)


def large(seed: int = 3, precision="bf16", **kw) -> dict:
    """N = 6, 24 options each -> 24**6 = 191,102,976 joint configs, 12->64->64->2."""
    return make_problem([24] * 6, 8, 64, 64, seed, 180.0, precision=precision, **kw)


def stress(seed: int = 4, precision="bf16", **kw) -> dict:
    """N = 8, 16 options each -> 16**8 = 2**32 joint configs, 20->128->128->2, soft latency."""
    return make_problem([16] * 8, 16, 128, 128, seed, 180.0, objective="soft_lat",
                        soft_penalty=0.1, precision=precision, **kw)


def _ints(seed: int, purpose: int, model: int, n: int, lo: int, hi: int) -> np.ndarray:
    """n integers uniform on [lo, hi] (multiply-shift on the top 32 bits), as float32."""
    z = stream_u64(stream_key(seed, purpose, model), n) >> np.uint64(32)
    span = np.uint64(hi - lo + 1)
    return ((z * span) >> np.uint64(32)).astype(np.int64).astype(np.float32) + np.float32(lo)


def integer_landscape(n_options, seed: int, vram_cap: float, objective="weighted_thr",
                      soft_penalty=0.0, coupled: bool = False) -> dict:
    """A d_L = 8, 12->64->64->2 problem whose every input is a small integer.

    Local features in [-2, 2], demands in [1, 9] (three columns), W1 in [-1, 1]
    with zero columns for the four aggregate inputs, W2 and W3 in [-1, 1], biases
    in [-2, 2], SLA ceilings and objective weights small integers.  Every
    intermediate value of the predictor and the objective is then an integer
    below 2**24 in magnitude, so fp32 and fp64 evaluation in any summation order
    give the same number and a GA run is reproducible bit for bit across
    implementations.

    coupled: keep W1's four aggregate columns (integers in [-1, 1]) and feed the
    aggregate unscaled (agg_scale = 1), so each predictor sees the candidate's
    summed demands and N; the values stay integers (below 2**24 for N <= 5).
    """
    n_options = np.asarray(n_options, dtype=np.int32)
    n = int(n_options.size)
    d, h, d_in = 8, 64, 12
    locs, dems, ws = [], [], []
    for i in range(n):
        k = int(n_options[i])
        locs.append(_ints(seed, P_LOCAL, i, k * d, -2, 2).reshape(k, d))
        dems.append(np.stack([_ints(seed, P_SM, i, k, 1, 9), _ints(seed, P_VRAM, i, k, 1, 9),
                              _ints(seed, P_BW, i, k, 1, 9)], axis=1))
        w1 = _ints(seed, P_W1, i, h * d_in, -1, 1).reshape(h, d_in)
        if not coupled:
            w1[:, d:] = 0.0
        ws.append(np.concatenate([w1.ravel(), _ints(seed, P_B1, i, h, -2, 2),
                                  _ints(seed, P_W2, i, h * h, -1, 1), _ints(seed, P_B2, i, h, -2, 2),
                                  _ints(seed, P_W3, i, 2 * h, -1, 1), _ints(seed, P_B3, i, 2, -2, 2)]))
    return dict(
        n_options=n_options, d_local=d, hidden1=h, hidden2=h,
        local_feats=np.ascontiguousarray(np.concatenate(locs, axis=0), dtype=np.float32),
        demand=np.ascontiguousarray(np.concatenate(dems, axis=0), dtype=np.float32),
        weights=np.ascontiguousarray(np.concatenate(ws), dtype=np.float32),
        agg_scale=np.ones(4, dtype=np.float32) if coupled else default_agg_scale(n), vram_cap=float(vram_cap),
        soft_penalty=float(soft_penalty), objective=objective, out_act="identity", precision="fp32",
        sla=_ints(seed, P_SLA, 0, n, 40, 120) * (4 if coupled else 1), obj_w=_ints(seed, P_OBJW, 0, n, 1, 3),
        scenario_seed=int(seed),
    )


# stream purposes of the fixed-context inputs
P_OBS, P_FMIN, P_FMAX, P_TAU, P_PREV = range(13, 18)


def fc_scenario(prob: dict, seed: int) -> dict:
    """Inputs of the fixed-context mode (observed state, per-option variant data, the
    utility constants of Eq. 3) for a problem drawn by make_problem.

    Model i alternates between an LLM-like model (two variants, FP16 / AWQ, quality
    1.000 / 0.979, reload cost 30 s) and a vision-like one (three variants, n / s / m,
    quality 0.73 / 0.96 / 1.00, reload cost 5 s) -- the paper's values (Sec. II).
    Option o of model i belongs to variant o mod V_i.  The per-variant throughput
    extrema stand in for the profiling extrema: f_min ~ U(-1, -0.2), f_max ~
    U(0.2, 1) (the synthetic predictors' outputs are of order 0.3).  The observed
    state is the aggregate of a typical configuration: SM share U(0.2, 0.4) N, VRAM
    U(5, 15) N GB, BW U(500, 1000) N GB/s.  Floors tau_i ~ U(-0.1, 0.15); the variant
    in use is uniform, or none (-1) with probability 1/4.  omega_i = 1, alpha = 1/60,
    beta = 5, delta = 0.05 (Sec. II)."""
    k = np.asarray(prob["n_options"], dtype=np.int64)
    n = int(k.size)
    llm = np.arange(n) % 2 == 0
    nv = np.where(llm, 2, 3)
    variant = np.concatenate([np.arange(int(k[i])) % nv[i] for i in range(n)]).astype(np.int32)
    qual = [np.array([1.000, 0.979]) if llm[i] else np.array([0.73, 0.96, 1.00]) for i in range(n)]
    quality = np.concatenate([qual[i][np.arange(int(k[i])) % nv[i]] for i in range(n)]).astype(np.float32)
    fmin_v = [uniform(seed, P_FMIN, i, int(nv[i]), -1.0, -0.2) for i in range(n)]
    fmax_v = [uniform(seed, P_FMAX, i, int(nv[i]), 0.2, 1.0) for i in range(n)]
    f_min = np.concatenate([fmin_v[i][np.arange(int(k[i])) % nv[i]] for i in range(n)]).astype(np.float32)
    f_max = np.concatenate([fmax_v[i][np.arange(int(k[i])) % nv[i]] for i in range(n)]).astype(np.float32)
    o = uniform(seed, P_OBS, 0, 3, 0.0, 1.0).astype(np.float64)
    obs = np.array([(0.2 + 0.2 * o[0]) * n, (5.0 + 10.0 * o[1]) * n, (500.0 + 500.0 * o[2]) * n, n],
                   dtype=np.float32)
    pz = stream_u64(stream_key(seed, P_PREV, 0), 2 * n)
    prev = np.array([-1 if (pz[2 * i] >> np.uint64(62)) == 0 else int((pz[2 * i + 1] >> np.uint64(32)) % np.uint64(nv[i]))
                     for i in range(n)], dtype=np.int32)
    return dict(obs=obs, variant=variant, quality=quality, f_min=f_min, f_max=f_max,
                omega=np.ones(n, dtype=np.float32), tau=uniform(seed, P_TAU, 0, n, -0.1, 0.15),
                reload_cost=np.where(llm, 30.0, 5.0).astype(np.float32), prev_variant=prev,
                alpha=1.0 / 60.0, beta=5.0, delta=0.05)


# The paper's GA at N = 5 (Sec. IV-C): 100 candidates, crossover probability 0.7,
# mutation probability 0.1, tournament of 3, elitism, 30 generations; infeasible
# offspring are repaired.
PAPER_GA_PARAMS = dict(pop=100, gens=30, tournament=3, crossover_p=0.7, mutation_p=0.1, elitism=1, repair=1)

GA_SCENARIO_SEEDS = tuple(range(100, 108))
GA_RUN_SEEDS = tuple(range(1000, 1050))

# GA parameters of the online-decision workload: population 1024, 100 generations,
# tournament of 4, uniform crossover, per-gene mutation 0.05, one elite.
GA_PARAMS = dict(pop=1024, gens=100, tournament=4, mutation_p=0.05, elitism=1)


def ga_scenario(scenario_seed: int, **kw) -> dict:
    """The N = 5 paper-scale problem with SLA and objective weights redrawn per scenario."""
    prob = paper_scale(**kw)
    return set_scenario(prob, scenario_seed)


def hand_example() -> dict:
    """Two models, two options each, one input feature and one hidden unit per layer.

    Small enough to evaluate by hand; the expected values are written out in the tests.
    """
    local = np.array([[0.5], [1.0], [0.25], [0.75]], dtype=np.float32)
    demand = np.array([[0.2, 4.0, 100.0], [0.4, 10.0, 300.0],
                       [0.1, 6.0, 200.0], [0.3, 16.0, 400.0]], dtype=np.float32)
    # d_in = 5: (x, Sigma SM, Sigma VRAM, Sigma BW, N)
    wa = [1, 0, -0.01, 0, 0, 0,   1, 0,   2, 1, 0, 0]
    wb = [1, -1, 0, 0, 0, 0,      1, 0,   1, 2, 0, 0]
    return dict(
        n_options=np.array([2, 2], dtype=np.int32), d_local=1, hidden1=1, hidden2=1,
        local_feats=local, demand=demand,
        weights=np.array(wa + wb, dtype=np.float32),
        agg_scale=np.ones(4, dtype=np.float32),
        sla=np.array([0.8, 0.6], dtype=np.float32), obj_w=np.ones(2, dtype=np.float32),
        vram_cap=24.0, soft_penalty=0.0, objective="weighted_thr", out_act="identity",
        precision="fp32", scenario_seed=-1,
    )


def random_small(seed: int, n_models: int, max_options: int = 6, d_local: int = 8,
                 h1: int = 32, h2: int = 0, vram_cap: float = 40.0, **kw) -> dict:
    """A small random grid (used for brute-force checks); option counts ~ U{1..max_options}."""
    z = stream_u64(stream_key(seed, 99, 0), n_models)
    ks = [1 + int(v % np.uint64(max_options)) for v in z]
    return make_problem(ks, d_local, h1, h2, seed, vram_cap, **kw)
