"""Thin ctypes binding of the C ABI in include/mf.h.

Argument marshalling only: every step of the scoring path runs in the CUDA
library.  Device buffers are torch tensors (their ``data_ptr()``) and calls run
on torch's current CUDA stream.  Importing this module loads the compiled
library and raises if it is missing; there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np
import torch

from . import build as _build

LIB_PATH = _build.LIB_PATH

MF_OK, MF_EINVAL, MF_ENOMEM, MF_ECUDA, MF_EUNSUPPORTED, MF_ETIMEOUT, MF_EDEVICE = range(7)
MF_FP32, MF_BF16, MF_FP32_SIMT = 0, 1, 2
_PRECISIONS = {"fp32": MF_FP32, "bf16": MF_BF16, "fp32_simt": MF_FP32_SIMT}
EMPTY = (1 << 64) - 1

_EXPORTS = ["mf_status_string", "mf_last_error", "mf_create", "mf_destroy", "mf_space_size",
            "mf_set_objective", "mf_score_batch", "mf_search_range", "mf_search_exhaustive",
            "mf_ga_generation", "mf_ga_init", "mf_ga_step", "mf_ga_run", "mf_check_device_status",
            "mf_get_stats", "mf_search_exhaustive_noalloc", "mf_fc_set", "mf_fc_table", "mf_fc_search",
            "mf_vram_feasible", "mf_set_utility", "mf_fc_ga_run", "mf_debug_wait_test"]


class MFError(RuntimeError):
    def __init__(self, status: int, where: str, detail: str):
        self.status = status
        super().__init__(f"{where}: {_lib.mf_status_string(status).decode()} ({detail})")


class _Problem(C.Structure):
    _fields_ = [
        ("n_models", C.c_int32), ("n_options", C.c_void_p), ("d_local", C.c_int32),
        ("hidden1", C.c_int32), ("hidden2", C.c_int32),
        ("local_feats", C.c_void_p), ("demand", C.c_void_p), ("weights", C.c_void_p),
        ("agg_scale", C.c_void_p), ("sla", C.c_void_p), ("obj_w", C.c_void_p),
        ("vram_cap", C.c_float), ("soft_penalty", C.c_float),
        ("out_act", C.c_int32), ("objective", C.c_int32), ("precision", C.c_int32),
        ("device", C.c_int32),
    ]


class _Result(C.Structure):
    _fields_ = [("best_idx", C.c_uint64), ("best_score", C.c_float), ("feasible_count", C.c_uint64),
                ("k", C.c_int32), ("topk_idx", C.c_void_p), ("topk_score", C.c_void_p)]


class _Stats(C.Structure):
    _fields_ = [("h2d_bytes_create", C.c_uint64), ("d2h_bytes_last", C.c_uint64),
                ("kernel_launches_last", C.c_int32), ("score_launches_last", C.c_int32),
                ("score_ms_last", C.c_float), ("total_ms_last", C.c_float), ("scoring_path", C.c_int32)]


class _GAParams(C.Structure):
    _fields_ = [("pop", C.c_int32), ("gens", C.c_int32), ("tournament", C.c_int32),
                ("mutation_p", C.c_double), ("elitism", C.c_int32)]


class _FcParams(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("variant", C.c_void_p), ("quality", C.c_void_p),
                ("f_min", C.c_void_p), ("f_max", C.c_void_p), ("omega", C.c_void_p), ("tau", C.c_void_p),
                ("reload_cost", C.c_void_p), ("prev_variant", C.c_void_p),
                ("alpha", C.c_float), ("beta", C.c_float), ("delta", C.c_float)]


class _FcGAParams(C.Structure):
    _fields_ = [("pop", C.c_int32), ("gens", C.c_int32), ("tournament", C.c_int32),
                ("crossover_p", C.c_double), ("mutation_p", C.c_double), ("elitism", C.c_int32),
                ("repair", C.c_int32)]


def _load() -> C.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with paper_2609_02109_gb300.build.build()")
    lib = C.CDLL(LIB_PATH)
    vp, u64, i32, st = C.c_void_p, C.c_uint64, C.c_int32, C.c_int
    lib.mf_status_string.argtypes = [st]; lib.mf_status_string.restype = C.c_char_p
    lib.mf_last_error.argtypes = []; lib.mf_last_error.restype = C.c_char_p
    lib.mf_create.argtypes = [C.POINTER(_Problem), C.POINTER(vp)]
    lib.mf_destroy.argtypes = [vp]
    lib.mf_space_size.argtypes = [vp, C.POINTER(u64)]
    lib.mf_set_objective.argtypes = [vp, vp, vp]
    lib.mf_score_batch.argtypes = [vp, vp, u64, vp, vp, vp, vp]
    lib.mf_search_range.argtypes = [vp, u64, u64, i32, u64, C.POINTER(_Result), vp]
    lib.mf_search_exhaustive.argtypes = [vp, i32, u64, C.POINTER(_Result), vp]
    lib.mf_ga_generation.argtypes = [vp, vp, i32, vp, vp]
    lib.mf_ga_init.argtypes = [vp, C.POINTER(_GAParams), u64, vp, vp]
    lib.mf_ga_step.argtypes = [vp, C.POINTER(_GAParams), u64, i32, vp, vp, vp, vp]
    lib.mf_ga_run.argtypes = [vp, C.POINTER(_GAParams), u64, vp, vp, vp]
    lib.mf_check_device_status.argtypes = [vp, vp]
    lib.mf_debug_wait_test.argtypes = [vp, C.c_uint32]
    lib.mf_get_stats.argtypes = [vp, C.POINTER(_Stats)]
    lib.mf_search_exhaustive_noalloc.argtypes = [C.POINTER(_Problem), i32, u64, C.POINTER(_Result), vp]
    lib.mf_fc_set.argtypes = [vp, C.POINTER(_FcParams), vp]
    lib.mf_fc_table.argtypes = [vp, vp, vp, vp, vp, vp]
    lib.mf_fc_search.argtypes = [vp, u64, u64, i32, u64, C.POINTER(_Result), vp]
    lib.mf_vram_feasible.argtypes = [vp, u64, u64, vp, u64, C.POINTER(u64), vp]
    lib.mf_set_utility.argtypes = [vp, C.POINTER(_FcParams)]
    lib.mf_fc_ga_run.argtypes = [vp, C.POINTER(_FcGAParams), u64, vp, vp, vp]
    for name in _EXPORTS[2:]:
        getattr(lib, name).restype = st
    return lib


_lib = _load()


def lib() -> C.CDLL:
    return _lib


def _check(status: int, where: str):
    if status != MF_OK:
        raise MFError(status, where, _lib.mf_last_error().decode())


def _stream(device) -> C.c_void_p:
    return C.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _ga(params: dict) -> _GAParams:
    return _GAParams(int(params["pop"]), int(params["gens"]), int(params["tournament"]),
                     float(params["mutation_p"]), int(params.get("elitism", 1)))


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32)


def _problem_struct(prob: dict, device: int, prec: str):
    """mf_problem for a workload dict; returns (struct, arrays kept alive)."""
    keep = {
        "n_options": np.ascontiguousarray(prob["n_options"], dtype=np.int32),
        "local_feats": _f32(prob["local_feats"]), "demand": _f32(prob["demand"]),
        "weights": _f32(prob["weights"]),
        "agg_scale": None if prob.get("agg_scale") is None else _f32(prob["agg_scale"]),
        "sla": _f32(prob["sla"]), "obj_w": _f32(prob["obj_w"]),
    }
    ptr = lambda a: None if a is None else a.ctypes.data  # noqa: E731
    k = keep
    p = _Problem(int(k["n_options"].size), ptr(k["n_options"]), int(prob["d_local"]),
                 int(prob["hidden1"]), int(prob["hidden2"]), ptr(k["local_feats"]), ptr(k["demand"]),
                 ptr(k["weights"]), ptr(k["agg_scale"]), ptr(k["sla"]), ptr(k["obj_w"]),
                 float(prob["vram_cap"]), float(prob.get("soft_penalty", 0.0)),
                 1 if prob.get("out_act", "identity") == "sigmoid" else 0,
                 1 if prob.get("objective", "weighted_thr") == "soft_lat" else 0,
                 _PRECISIONS[prec], int(device))
    return p, keep


def search_exhaustive_noalloc(prob: dict, k: int, chunk: int = 0, device: int | None = None) -> dict:
    """mf_search_exhaustive_noalloc: the exact fp32 search with no device allocation
    (all device memory in the library's fixed array); same result fields as
    Context.search."""
    device = torch.cuda.current_device() if device is None else int(device)
    p, _keep = _problem_struct(prob, device, "fp32")
    ti = np.empty(k, dtype=np.uint64)
    ts = np.empty(k, dtype=np.float32)
    r = _Result(0, 0.0, 0, k, ti.ctypes.data, ts.ctypes.data)
    _check(_lib.mf_search_exhaustive_noalloc(C.byref(p), int(k), int(chunk), C.byref(r),
                                              _stream(device)), "mf_search_exhaustive_noalloc")
    return dict(best_idx=int(r.best_idx), best_score=float(r.best_score),
                count=int(r.feasible_count), topk_idx=ti, topk_score=ts)


class Context:
    """An mf_ctx bound to one problem (a dict as drawn by ``workload``)."""

    def __init__(self, prob: dict, device: int | None = None, precision: str | None = None):
        self.device = torch.cuda.current_device() if device is None else int(device)
        prec = precision or prob.get("precision", "fp32")
        p, self._keep = _problem_struct(prob, self.device, prec)
        self.n_models = int(p.n_models)
        h = C.c_void_p()
        with torch.cuda.device(self.device):
            _check(_lib.mf_create(C.byref(p), C.byref(h)), "mf_create")
        self._h = h
        self.precision = prec

    # -- lifetime -----------------------------------------------------------------
    def close(self):
        if getattr(self, "_h", None):
            _lib.mf_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # -- calls ----------------------------------------------------------------------
    @property
    def space_size(self) -> int:
        v = C.c_uint64()
        _check(_lib.mf_space_size(self._h, C.byref(v)), "mf_space_size")
        return int(v.value)

    def set_objective(self, sla=None, obj_w=None):
        s = None if sla is None else _f32(sla)
        w = None if obj_w is None else _f32(obj_w)
        _check(_lib.mf_set_objective(self._h, None if s is None else s.ctypes.data,
                                     None if w is None else w.ctypes.data), "mf_set_objective")

    def score_batch(self, idx: torch.Tensor, with_pred: bool = False, score=None, feasible=None,
                    pred=None):
        """idx: int64/uint64 CUDA tensor of joint indices -> (score f32, feasible u8[, pred])."""
        assert idx.is_cuda and idx.dtype in (torch.int64, torch.uint64) and idx.is_contiguous()
        n = idx.numel()
        dev = idx.device
        score = torch.empty(n, dtype=torch.float32, device=dev) if score is None else score
        feasible = torch.empty(n, dtype=torch.uint8, device=dev) if feasible is None else feasible
        if with_pred and pred is None:
            pred = torch.empty((n, self.n_models, 2), dtype=torch.float32, device=dev)
        _check(_lib.mf_score_batch(self._h, idx.data_ptr(), n, score.data_ptr(), feasible.data_ptr(),
                                   pred.data_ptr() if pred is not None else None, _stream(dev)),
               "mf_score_batch")
        return (score, feasible, pred) if with_pred else (score, feasible)

    def search(self, k: int, lo: int = 0, hi: int | None = None, chunk: int = 0) -> dict:
        hi = self.space_size if hi is None else int(hi)
        ti = np.empty(k, dtype=np.uint64)
        ts = np.empty(k, dtype=np.float32)
        r = _Result(0, 0.0, 0, k, ti.ctypes.data, ts.ctypes.data)
        _check(_lib.mf_search_range(self._h, int(lo), hi, int(k), int(chunk), C.byref(r),
                                    _stream(self.device)), "mf_search_range")
        return dict(best_idx=int(r.best_idx), best_score=float(r.best_score),
                    count=int(r.feasible_count), topk_idx=ti, topk_score=ts)

    def ga_generation(self, pop: torch.Tensor, fitness: torch.Tensor | None = None) -> torch.Tensor:
        assert pop.is_cuda and pop.dtype == torch.int32 and pop.is_contiguous()
        P = pop.shape[0]
        fitness = torch.empty(P, dtype=torch.float32, device=pop.device) if fitness is None else fitness
        _check(_lib.mf_ga_generation(self._h, pop.data_ptr(), P, fitness.data_ptr(), _stream(pop.device)),
               "mf_ga_generation")
        return fitness

    def ga_init(self, params: dict, seed: int) -> torch.Tensor:
        g = _ga(params)
        pop = torch.empty((g.pop, self.n_models), dtype=torch.int32, device=f"cuda:{self.device}")
        _check(_lib.mf_ga_init(self._h, C.byref(g), int(seed), pop.data_ptr(), _stream(pop.device)),
               "mf_ga_init")
        return pop

    def ga_step(self, params: dict, seed: int, gen: int, pop: torch.Tensor,
                fitness: torch.Tensor) -> torch.Tensor:
        g = _ga(params)
        nxt = torch.empty_like(pop)
        _check(_lib.mf_ga_step(self._h, C.byref(g), int(seed), int(gen), pop.data_ptr(),
                               fitness.data_ptr(), nxt.data_ptr(), _stream(pop.device)), "mf_ga_step")
        return nxt

    def ga_run(self, params: dict, seed: int):
        g = _ga(params)
        genome = np.zeros(self.n_models, dtype=np.int32)
        fit = C.c_float()
        _check(_lib.mf_ga_run(self._h, C.byref(g), int(seed), genome.ctypes.data, C.byref(fit),
                              _stream(self.device)), "mf_ga_run")
        return float(fit.value), genome

    # -- fixed-context mode ---------------------------------------------------
    @staticmethod
    def _fc_params(fc: dict):
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
        p = _FcParams(*(keep[k].ctypes.data for k in ("obs", "variant", "quality", "f_min", "f_max", "omega",
                                                       "tau", "reload_cost", "prev_variant")),
                      float(fc["alpha"]), float(fc["beta"]), float(fc["delta"]))
        return p, keep

    def fc_set(self, fc: dict) -> None:
        """Evaluate the local predictions under fc["obs"] and build the utility table."""
        p, keep = self._fc_params(fc)
        _check(_lib.mf_fc_set(self._h, C.byref(p), _stream(self.device)), "mf_fc_set")

    def set_utility(self, fc: dict | None) -> None:
        """Score with the Eq. 3 utility on the coupled aggregate (None: the problem's objective)."""
        if fc is None:
            _check(_lib.mf_set_utility(self._h, None), "mf_set_utility")
            return
        p, keep = self._fc_params(dict(fc, obs=np.zeros(4, np.float32)))
        _check(_lib.mf_set_utility(self._h, C.byref(p)), "mf_set_utility")

    def fc_table(self):
        """(fhat, f, u, ok) of every option row, as numpy arrays."""
        rows = int(self._keep["n_options"].sum())
        dev = f"cuda:{self.device}"
        fhat, f, u = (torch.empty(rows, dtype=torch.float32, device=dev) for _ in range(3))
        ok = torch.empty(rows, dtype=torch.uint8, device=dev)
        _check(_lib.mf_fc_table(self._h, fhat.data_ptr(), f.data_ptr(), u.data_ptr(), ok.data_ptr(),
                                _stream(self.device)), "mf_fc_table")
        torch.cuda.current_stream(self.device).synchronize()
        return fhat.cpu().numpy(), f.cpu().numpy(), u.cpu().numpy(), ok.cpu().numpy().astype(bool)

    def fc_search(self, k: int, lo: int = 0, hi: int | None = None, chunk: int = 0) -> dict:
        hi = self.space_size if hi is None else int(hi)
        ti = np.empty(k, dtype=np.uint64)
        ts = np.empty(k, dtype=np.float32)
        r = _Result(0, 0.0, 0, k, ti.ctypes.data, ts.ctypes.data)
        _check(_lib.mf_fc_search(self._h, int(lo), hi, int(k), int(chunk), C.byref(r), _stream(self.device)),
               "mf_fc_search")
        return dict(best_idx=int(r.best_idx), best_score=float(r.best_score), count=int(r.feasible_count),
                    topk_idx=ti, topk_score=ts)

    def fc_ga_run(self, params: dict, seed: int):
        """The paper's GA on the fixed-context landscape: (best J, genome)."""
        g = _FcGAParams(int(params["pop"]), int(params["gens"]), int(params["tournament"]),
                        float(params["crossover_p"]), float(params["mutation_p"]), int(params["elitism"]),
                        int(params["repair"]))
        genome = np.zeros(self.n_models, dtype=np.int32)
        fit = C.c_float()
        _check(_lib.mf_fc_ga_run(self._h, C.byref(g), int(seed), genome.ctypes.data, C.byref(fit),
                                 _stream(self.device)), "mf_fc_ga_run")
        return float(fit.value), genome

    def vram_feasible(self, lo: int = 0, hi: int | None = None, cap: int | None = None):
        """(count, device tensor of the first min(count, cap) VRAM-feasible indices)."""
        hi = self.space_size if hi is None else int(hi)
        cap = (hi - int(lo)) if cap is None else int(cap)
        out = torch.empty(max(cap, 1), dtype=torch.int64, device=f"cuda:{self.device}")
        cnt = C.c_uint64(0)
        _check(_lib.mf_vram_feasible(self._h, int(lo), hi, out.data_ptr(), cap, C.byref(cnt),
                                     _stream(self.device)), "mf_vram_feasible")
        c = int(cnt.value)
        return c, out[:min(c, cap)]

    def stats(self) -> dict:
        st = _Stats()
        _check(_lib.mf_get_stats(self._h, C.byref(st)), "mf_get_stats")
        return {f: getattr(st, f) for f, _ in _Stats._fields_}

    def check_status(self) -> int:
        """MF_OK, or the status of the first device-reported problem (clears it)."""
        return int(_lib.mf_check_device_status(self._h, _stream(self.device)))

    def debug_wait_test(self, polls: int) -> None:
        """mf_debug_wait_test: with polls > 0 the context's waiting kernels first wait on
        a flag that nothing sets and give up (tests of the timeout path); 0 restores."""
        _check(_lib.mf_debug_wait_test(self._h, int(polls)), "mf_debug_wait_test")
