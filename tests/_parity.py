"""Comparison helpers of the GPU path against the CPU oracle.

Tolerances (from the accuracy contract of the scorer):
  * fp32 path: per-candidate J within 1e-5 relative; bf16 path within 2e-2.
    Relative to scale = max(|J_ref|, sum_i w_i |thr_i|) (plus lambda * sum_i
    |lat_i - SLA_i| for the soft-latency objective), so a J that cancels to
    ~0 is compared against the size of its terms.
  * feasibility bit-exact except for candidates near a threshold: within 1e-4
    relative of the VRAM cap or of an SLA (bf16: an SLA band of 2e-2 relative).
  * the GPU's chosen configuration scores (by the oracle) within 1e-5 relative
    of the oracle's optimum.
"""
from __future__ import annotations

import numpy as np

RTOL = {"fp32": 1e-5, "bf16": 2e-2}
NEAR_REL = 1e-4
NEAR_SLA = {"fp32": 1e-4, "bf16": 2e-2}


def score_scale(prob, ref_score, ref_pred):
    w = np.asarray(prob["obj_w"], dtype=np.float64)
    sc = np.abs(ref_pred[..., 0]) @ w
    if prob.get("objective") == "soft_lat":
        sla = np.asarray(prob["sla"], dtype=np.float64)
        sc = sc + float(prob["soft_penalty"]) * np.abs(ref_pred[..., 1] - sla).sum(axis=-1)
    fin = np.isfinite(ref_score)
    return np.maximum(np.where(fin, np.abs(np.where(fin, ref_score, 0.0)), 0.0), sc)


def near_threshold(prob, ref_pred, ref_agg, prec="fp32"):
    cap = float(prob["vram_cap"])
    near = np.abs(ref_agg[:, 1] - cap) <= NEAR_REL * max(abs(cap), 1e-30)
    if prob.get("objective", "weighted_thr") != "soft_lat":
        sla = np.asarray(prob["sla"], dtype=np.float64)[None, :]
        lat = ref_pred[..., 1]
        band = NEAR_SLA[prec] * np.maximum(np.abs(sla), np.abs(lat))
        near |= (np.abs(lat - sla) <= band).any(axis=1)
    return near


def check_scores(prob, got_score, got_feas, ref_score, ref_feas, ref_pred, ref_agg, prec="fp32",
                 got_pred=None, pred_scale=None):
    """Element-wise parity of a score batch.  Returns the number of near-threshold
    candidates excluded from the exact feasibility comparison.

    Per-model outputs: fp32 within 1e-5 of max(|y|, RMS of the head over the batch);
    bf16 within 2e-2 of max(|y|, c), c = the oracle's condition scale of the head,
    |b3| + sum_k |W3_k| |h_k| (bf16 rounding errors scale with the magnitude of the
    terms of the final dot product, which can cancel to a much smaller |y|)."""
    got_score = np.asarray(got_score, dtype=np.float64)
    got_feas = np.asarray(got_feas).astype(bool)
    near = near_threshold(prob, ref_pred, ref_agg, prec)
    bad = (got_feas != ref_feas) & ~near
    assert not bad.any(), f"{bad.sum()} feasibility mismatches away from thresholds, e.g. {np.where(bad)[0][:5]}"
    both = got_feas & ref_feas
    scale = score_scale(prob, ref_score, ref_pred)
    err = np.abs(got_score[both] - ref_score[both]) / np.maximum(scale[both], 1e-30)
    if err.size:
        assert err.max() <= RTOL[prec], f"score error {err.max():.3g} > {RTOL[prec]} at {np.argmax(err)}"
    assert np.all(got_score[~got_feas] == -np.inf)
    if got_pred is not None:
        gp = np.asarray(got_pred, dtype=np.float64)
        for h in range(2):
            if pred_scale is not None:
                den = np.maximum(np.abs(ref_pred[..., h]), pred_scale[..., h])
            else:
                rms = np.sqrt(np.mean(ref_pred[..., h] ** 2, axis=0, keepdims=True))
                den = np.maximum(np.abs(ref_pred[..., h]), rms)
            d = np.abs(gp[..., h] - ref_pred[..., h]) / np.maximum(den, 1e-30)
            assert d.max() <= RTOL[prec], f"head {h} error {d.max():.3g}"
    return int(near.sum())


def check_search(o, prob, res, k, ref_topk, ref_count, near_count_bound=0, prec="fp32"):
    """Parity of an exhaustive search result against the oracle's."""
    ti_ref, ts_ref = ref_topk
    n_valid = int(min(k, ref_count))
    assert abs(res["count"] - ref_count) <= near_count_bound, (res["count"], ref_count)
    gi = res["topk_idx"].astype(np.uint64)
    gs = res["topk_score"].astype(np.float64)
    if n_valid == 0:
        assert res["best_idx"] == 2 ** 64 - 1 and res["best_score"] == -np.inf
        return
    # GPU top-k entries rescored by the oracle
    valid = gi != np.uint64(2 ** 64 - 1)
    s_o, f_o, pred_o, agg_o = o.score_list(gi[valid], with_pred=True)
    near = near_threshold(prob, pred_o, agg_o, prec)
    assert np.all(f_o | near), "a reported top-k entry is infeasible for the oracle"
    scale = score_scale(prob, s_o, pred_o)
    rt = RTOL["fp32"]  # reported scores are fp32 (re-scored on the bf16 path)
    ok = f_o
    assert np.all(np.abs(gs[valid][ok] - s_o[ok]) <= rt * np.maximum(scale[ok], 1e-30))
    # sorted score sequences agree
    m = min(int(valid.sum()), n_valid)
    _, _, pred_r, _ = o.score_list(np.asarray(ti_ref[:m], dtype=np.uint64), with_pred=True)
    ref_scale = np.maximum(score_scale(prob, ts_ref[:m], pred_r), 1e-30)
    assert np.all(np.abs(gs[:m] - ts_ref[:m]) <= 2 * rt * ref_scale), (gs[:m], ts_ref[:m])
    # where the oracle's scores are well separated, the indices match exactly
    for j in range(m):
        gap_prev = ts_ref[j - 1] - ts_ref[j] if j > 0 else np.inf
        gap_next = ts_ref[j] - ts_ref[j + 1] if j + 1 < len(ts_ref) and np.isfinite(ts_ref[j + 1]) else np.inf
        if min(gap_prev, gap_next) > 4 * rt * ref_scale[j] and not near[j]:
            assert int(gi[j]) == int(ti_ref[j]), (j, int(gi[j]), int(ti_ref[j]))
    # the chosen configuration is optimal within 1e-5 relative
    best_ref = ts_ref[0]
    assert s_o[0] >= best_ref - 1e-5 * max(abs(best_ref), 1e-30) or near[0]
    # order: (J desc, idx asc) on the GPU's own scores
    for j in range(int(valid.sum()) - 1):
        assert gs[j] > gs[j + 1] or (gs[j] == gs[j + 1] and gi[j] < gi[j + 1])
    assert np.all(~valid[int(valid.sum()):])
