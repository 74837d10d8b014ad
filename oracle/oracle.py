"""ctypes wrapper of the C oracle (oracle/mf_oracle.c) -- TEST INFRASTRUCTURE.

Only tests/, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` import this module.  It never imports the CUDA package, and the
CUDA package never imports it.  Problems are the plain dicts drawn by
``paper_2609_02109_gb300.workload`` (numpy arrays only).
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
import threading

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "mf_oracle.c")
LIB = os.path.join(HERE, "_build", "liboracle.so")

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when available).  Returns the .so path."""
    os.makedirs(os.path.dirname(LIB), exist_ok=True)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= max(
            os.path.getmtime(SRC), os.path.getmtime(os.path.join(HERE, "mf_oracle.h"))):
        return LIB
    tmp = LIB + f".tmp{os.getpid()}"
    base = ["gcc", "-std=c99", "-O2", "-fPIC", "-shared", SRC, "-o", tmp, "-lm"]
    r = subprocess.run(base[:3] + ["-fopenmp"] + base[3:], capture_output=True, text=True)
    if r.returncode != 0:  # no OpenMP runtime: build single-threaded
        r = subprocess.run(base, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError("oracle build failed:\n" + r.stderr)
    os.replace(tmp, LIB)
    return LIB


class _Problem(C.Structure):
    _fields_ = [
        ("n_models", C.c_int32), ("n_options", C.c_void_p), ("d_local", C.c_int32),
        ("hidden1", C.c_int32), ("hidden2", C.c_int32),
        ("local_feats", C.c_void_p), ("demand", C.c_void_p), ("weights", C.c_void_p),
        ("agg_scale", C.c_void_p), ("sla", C.c_void_p), ("obj_w", C.c_void_p),
        ("vram_cap", C.c_float), ("soft_penalty", C.c_float),
        ("out_act", C.c_int32), ("objective", C.c_int32),
    ]


class _FC(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("variant", C.c_void_p), ("quality", C.c_void_p),
                ("f_min", C.c_void_p), ("f_max", C.c_void_p), ("omega", C.c_void_p),
                ("tau", C.c_void_p), ("reload_cost", C.c_void_p), ("prev_variant", C.c_void_p),
                ("alpha", C.c_float), ("beta", C.c_float), ("delta", C.c_float)]


class _FcGAParams(C.Structure):
    _fields_ = [("pop", C.c_int32), ("gens", C.c_int32), ("tournament", C.c_int32),
                ("crossover_p", C.c_double), ("mutation_p", C.c_double), ("elitism", C.c_int32),
                ("repair", C.c_int32)]


class _GAParams(C.Structure):
    _fields_ = [("pop", C.c_int32), ("gens", C.c_int32), ("tournament", C.c_int32),
                ("mutation_p", C.c_double), ("elitism", C.c_int32)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = C.CDLL(build())
            P = C.POINTER(_Problem)
            G = C.POINTER(_GAParams)
            vp, u64, i32, dbl = C.c_void_p, C.c_uint64, C.c_int32, C.c_double
            lib.orc_space_size.argtypes = [P]; lib.orc_space_size.restype = u64
            lib.orc_decode.argtypes = [P, u64, vp]; lib.orc_decode.restype = None
            lib.orc_score_digits.argtypes = [P, vp, vp, vp, vp]; lib.orc_score_digits.restype = dbl
            lib.orc_score_list.argtypes = [P, vp, u64, vp, vp, vp, vp, i32]
            lib.orc_score_list.restype = None
            lib.orc_pred_scale_list.argtypes = [P, vp, u64, vp, i32]
            lib.orc_pred_scale_list.restype = None
            lib.orc_exhaustive.argtypes = [P, u64, u64, i32, vp, vp, vp, i32]
            lib.orc_exhaustive.restype = None
            lib.orc_splitmix64.argtypes = [u64, u64]; lib.orc_splitmix64.restype = u64
            lib.orc_rng.argtypes = [u64, C.c_uint32, C.c_uint32, C.c_uint32, C.c_uint32]
            lib.orc_rng.restype = u64
            lib.orc_ga_init.argtypes = [P, G, u64, vp]; lib.orc_ga_init.restype = None
            lib.orc_ga_step.argtypes = [P, G, u64, i32, vp, vp, vp]; lib.orc_ga_step.restype = None
            lib.orc_ga_run.argtypes = [P, G, u64, vp, i32]; lib.orc_ga_run.restype = dbl
            F = C.POINTER(_FC)
            lib.orc_fc_local.argtypes = [P, F, vp, vp, vp, vp]; lib.orc_fc_local.restype = None
            lib.orc_fc_score_digits.argtypes = [P, F, vp, vp]; lib.orc_fc_score_digits.restype = dbl
            lib.orc_fc_exhaustive.argtypes = [P, F, u64, u64, i32, vp, vp, vp, i32]
            lib.orc_fc_exhaustive.restype = None
            lib.orc_vram_feasible.argtypes = [P, u64, u64, vp, u64]; lib.orc_vram_feasible.restype = u64
            lib.orc_util_score_digits.argtypes = [P, F, vp, vp, vp, vp]; lib.orc_util_score_digits.restype = dbl
            lib.orc_util_score_list.argtypes = [P, F, vp, u64, vp, vp, vp, vp, i32]
            lib.orc_util_score_list.restype = None
            lib.orc_util_exhaustive.argtypes = [P, F, u64, u64, i32, vp, vp, vp, i32]
            lib.orc_util_exhaustive.restype = None
            lib.orc_fc_ga_run.argtypes = [P, F, C.POINTER(_FcGAParams), u64, vp]
            lib.orc_fc_ga_run.restype = dbl
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


class Oracle:
    """Binds one problem dict; keeps its arrays alive for the C calls."""

    def __init__(self, prob: dict, nthreads: int | None = None):
        self.lib = _load()
        self.nthreads = int(nthreads or os.cpu_count() or 1)
        self._arr = {
            "n_options": np.ascontiguousarray(prob["n_options"], dtype=np.int32),
            "local_feats": np.ascontiguousarray(prob["local_feats"], dtype=np.float32),
            "demand": np.ascontiguousarray(prob["demand"], dtype=np.float32),
            "weights": np.ascontiguousarray(prob["weights"], dtype=np.float32),
            "agg_scale": None if prob.get("agg_scale") is None else
            np.ascontiguousarray(prob["agg_scale"], dtype=np.float32),
            "sla": np.ascontiguousarray(prob["sla"], dtype=np.float32),
            "obj_w": np.ascontiguousarray(prob["obj_w"], dtype=np.float32),
        }
        a = self._arr
        self.n = int(a["n_options"].size)
        self.p = _Problem(
            self.n, _ptr(a["n_options"]), int(prob["d_local"]), int(prob["hidden1"]),
            int(prob["hidden2"]), _ptr(a["local_feats"]), _ptr(a["demand"]), _ptr(a["weights"]),
            _ptr(a["agg_scale"]), _ptr(a["sla"]), _ptr(a["obj_w"]),
            float(prob["vram_cap"]), float(prob.get("soft_penalty", 0.0)),
            1 if prob.get("out_act", "identity") == "sigmoid" else 0,
            1 if prob.get("objective", "weighted_thr") == "soft_lat" else 0)

    # -- Eq. 1 ---------------------------------------------------------------
    def space_size(self) -> int:
        return int(self.lib.orc_space_size(C.byref(self.p)))

    def decode(self, idx: int) -> np.ndarray:
        o = np.zeros(self.n, dtype=np.int32)
        self.lib.orc_decode(C.byref(self.p), int(idx), _ptr(o))
        return o

    # -- Eqs. 2-6, one candidate ----------------------------------------------
    def score_digits(self, digits):
        o = np.ascontiguousarray(digits, dtype=np.int32)
        f = np.zeros(1, dtype=np.int32)
        pred = np.zeros((self.n, 2), dtype=np.float64)
        agg = np.zeros(4, dtype=np.float64)
        J = self.lib.orc_score_digits(C.byref(self.p), _ptr(o), _ptr(f), _ptr(pred), _ptr(agg))
        return float(J), bool(f[0]), pred, agg

    def score_list(self, idx, with_pred: bool = False):
        idx = np.ascontiguousarray(idx, dtype=np.uint64)
        n = idx.size
        score = np.empty(n, dtype=np.float64)
        feas = np.empty(n, dtype=np.int32)
        pred = np.empty((n, self.n, 2), dtype=np.float64) if with_pred else None
        agg = np.empty((n, 4), dtype=np.float64) if with_pred else None
        self.lib.orc_score_list(C.byref(self.p), _ptr(idx), n, _ptr(score), _ptr(feas),
                                _ptr(pred), _ptr(agg), self.nthreads)
        if with_pred:
            return score, feas.astype(bool), pred, agg
        return score, feas.astype(bool)

    def pred_scale(self, idx) -> np.ndarray:
        """[n][N][2] condition scales |b3| + sum_k |W3_k||h_k| of the outputs."""
        idx = np.ascontiguousarray(idx, dtype=np.uint64)
        out = np.empty((idx.size, self.n, 2), dtype=np.float64)
        self.lib.orc_pred_scale_list(C.byref(self.p), _ptr(idx), idx.size, _ptr(out), self.nthreads)
        return out

    def exhaustive(self, k: int, lo: int = 0, hi: int | None = None, nthreads: int | None = None):
        hi = self.space_size() if hi is None else hi
        ti = np.empty(k, dtype=np.uint64)
        ts = np.empty(k, dtype=np.float64)
        cnt = np.zeros(1, dtype=np.uint64)
        self.lib.orc_exhaustive(C.byref(self.p), int(lo), int(hi), int(k), _ptr(ti), _ptr(ts),
                                _ptr(cnt), int(nthreads or self.nthreads))
        return ti, ts, int(cnt[0])

    # -- GA ---------------------------------------------------------------------
    @staticmethod
    def _ga(params: dict) -> _GAParams:
        return _GAParams(int(params["pop"]), int(params["gens"]), int(params["tournament"]),
                         float(params["mutation_p"]), int(params.get("elitism", 1)))

    def ga_init(self, params: dict, seed: int) -> np.ndarray:
        g = self._ga(params)
        pop = np.zeros((g.pop, self.n), dtype=np.int32)
        self.lib.orc_ga_init(C.byref(self.p), C.byref(g), int(seed), _ptr(pop))
        return pop

    def ga_step(self, params: dict, seed: int, gen: int, pop, fitness) -> np.ndarray:
        g = self._ga(params)
        pop = np.ascontiguousarray(pop, dtype=np.int32)
        fit = np.ascontiguousarray(fitness, dtype=np.float64)
        nxt = np.zeros_like(pop)
        self.lib.orc_ga_step(C.byref(self.p), C.byref(g), int(seed), int(gen), _ptr(pop),
                             _ptr(fit), _ptr(nxt))
        return nxt

    def ga_run(self, params: dict, seed: int):
        g = self._ga(params)
        best = np.zeros(self.n, dtype=np.int32)
        J = self.lib.orc_ga_run(C.byref(self.p), C.byref(g), int(seed), _ptr(best), self.nthreads)
        return float(J), best


    # -- fixed-context mode (Sec. III-B, Eq. 3, Eq. 4) ---------------------------
    def _fc(self, fc: dict) -> _FC:
        keep = {
            "obs": np.ascontiguousarray(fc["obs"], dtype=np.float32),
            "variant": np.ascontiguousarray(fc["variant"], dtype=np.int32),
            "quality": np.ascontiguousarray(fc["quality"], dtype=np.float32),
            "f_min": np.ascontiguousarray(fc["f_min"], dtype=np.float32),
            "f_max": np.ascontiguousarray(fc["f_max"], dtype=np.float32),
            "omega": np.ascontiguousarray(fc["omega"], dtype=np.float32),
            "tau": np.ascontiguousarray(fc["tau"], dtype=np.float32),
            "reload_cost": np.ascontiguousarray(fc["reload_cost"], dtype=np.float32),
            "prev_variant": np.ascontiguousarray(fc["prev_variant"], dtype=np.int32),
        }
        self._fc_keep = keep
        return _FC(*(_ptr(keep[k]) for k in ("obs", "variant", "quality", "f_min", "f_max", "omega", "tau",
                                             "reload_cost", "prev_variant")),
                   float(fc["alpha"]), float(fc["beta"]), float(fc["delta"]))

    def fc_local(self, fc: dict):
        """Per option row: (fhat, f, ok, u)."""
        f_ = self._fc(fc)
        rows = int(np.asarray(self._arr["n_options"]).sum())
        fhat, f, u = (np.empty(rows) for _ in range(3))
        ok = np.empty(rows, dtype=np.int32)
        self.lib.orc_fc_local(C.byref(self.p), C.byref(f_), _ptr(fhat), _ptr(f), _ptr(ok), _ptr(u))
        return fhat, f, ok.astype(bool), u

    def fc_score_digits(self, fc: dict, digits):
        f_ = self._fc(fc)
        o = np.ascontiguousarray(digits, dtype=np.int32)
        feas = np.zeros(1, dtype=np.int32)
        J = self.lib.orc_fc_score_digits(C.byref(self.p), C.byref(f_), _ptr(o), _ptr(feas))
        return float(J), bool(feas[0])

    def fc_exhaustive(self, fc: dict, k: int, lo: int = 0, hi: int | None = None):
        f_ = self._fc(fc)
        hi = self.space_size() if hi is None else int(hi)
        ti = np.empty(k, dtype=np.uint64)
        ts = np.empty(k, dtype=np.float64)
        cnt = np.zeros(1, dtype=np.uint64)
        self.lib.orc_fc_exhaustive(C.byref(self.p), C.byref(f_), int(lo), hi, int(k), _ptr(ti), _ptr(ts),
                                   _ptr(cnt), self.nthreads)
        return ti, ts, int(cnt[0])

    # -- Eq. 3 utility on the coupled aggregate -----------------------------------
    def util_score_digits(self, fc: dict, digits):
        f_ = self._fc(fc)
        o = np.ascontiguousarray(digits, dtype=np.int32)
        feas = np.zeros(1, dtype=np.int32)
        pred = np.empty((self.n, 2))
        J = self.lib.orc_util_score_digits(C.byref(self.p), C.byref(f_), _ptr(o), _ptr(feas), _ptr(pred), None)
        return float(J), bool(feas[0]), pred

    def util_score_list(self, fc: dict, idx, with_pred: bool = False):
        f_ = self._fc(fc)
        idx = np.ascontiguousarray(idx, dtype=np.uint64)
        n = idx.size
        score = np.empty(n)
        feas = np.empty(n, dtype=np.int32)
        pred = np.empty((n, self.n, 2)) if with_pred else None
        agg = np.empty((n, 4)) if with_pred else None
        self.lib.orc_util_score_list(C.byref(self.p), C.byref(f_), _ptr(idx), n, _ptr(score), _ptr(feas),
                                     _ptr(pred), _ptr(agg), self.nthreads)
        if with_pred:
            return score, feas.astype(bool), pred, agg
        return score, feas.astype(bool)

    def util_exhaustive(self, fc: dict, k: int, lo: int = 0, hi: int | None = None):
        f_ = self._fc(fc)
        hi = self.space_size() if hi is None else int(hi)
        ti = np.empty(k, dtype=np.uint64)
        ts = np.empty(k, dtype=np.float64)
        cnt = np.zeros(1, dtype=np.uint64)
        self.lib.orc_util_exhaustive(C.byref(self.p), C.byref(f_), int(lo), hi, int(k), _ptr(ti), _ptr(ts),
                                     _ptr(cnt), self.nthreads)
        return ti, ts, int(cnt[0])

    def fc_ga_run(self, fc: dict, params: dict, seed: int):
        """The paper's GA on the fixed-context landscape: (best J, genome)."""
        f_ = self._fc(fc)
        g = _FcGAParams(int(params["pop"]), int(params["gens"]), int(params["tournament"]),
                        float(params["crossover_p"]), float(params["mutation_p"]), int(params["elitism"]),
                        int(params["repair"]))
        best = np.zeros(self.n, dtype=np.int32)
        J = self.lib.orc_fc_ga_run(C.byref(self.p), C.byref(f_), C.byref(g), int(seed), _ptr(best))
        return float(J), best

    def vram_feasible(self, lo: int = 0, hi: int | None = None, cap: int | None = None):
        """(count, ascending list of the first min(count, cap) VRAM-feasible indices)."""
        hi = self.space_size() if hi is None else int(hi)
        cap = (hi - int(lo)) if cap is None else int(cap)
        out = np.empty(max(cap, 1), dtype=np.uint64)
        c = int(self.lib.orc_vram_feasible(C.byref(self.p), int(lo), hi, _ptr(out), cap))
        return c, out[:min(c, cap)]


def splitmix64(seed: int, ctr: int) -> int:
    return int(_load().orc_splitmix64(int(seed), int(ctr)))


def rng(seed: int, gen: int, slot: int, purpose: int, j: int) -> int:
    return int(_load().orc_rng(int(seed), gen, slot, purpose, j))
