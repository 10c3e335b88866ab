"""Shared test helpers (inputs come from synth; expectations from oracle/)."""
import numpy as np

from oracle import decoder as D


def oracle_model(shape, seed=0):
    from paper_2602_20217_gb300 import synth
    return D.OracleConfig.like(shape), D.as_f64(synth.np_model_weights(shape, seed=seed))


def token_ok(gpu_tok, ref_logits_row, tol):
    """A greedy token is correct if it is the oracle's argmax, or the oracle
    ranks it within ``tol`` of the maximum (a near-tie both sides may break
    differently at different precisions)."""
    ref = int(np.argmax(ref_logits_row))
    if int(gpu_tok) == ref:
        return True
    return ref_logits_row[ref] - ref_logits_row[int(gpu_tok)] <= tol


def rel_err(got, ref):
    """Largest per-row ||got - ref||_inf / ||ref||_inf (the logits tolerance is
    stated per row, so a row of small values cannot hide behind a large one).
    A 1-D input is one row."""
    g = np.atleast_2d(np.asarray(got, np.float64))
    r = np.atleast_2d(np.asarray(ref, np.float64))
    assert g.shape == r.shape, (g.shape, r.shape)
    g = g.reshape(-1, g.shape[-1])
    r = r.reshape(-1, r.shape[-1])
    return float(np.max(np.max(np.abs(g - r), axis=1) / np.max(np.abs(r), axis=1)))


def token_within_tolerance(gpu_tok, ref_logits_row, rel_tol):
    """The greedy token is the oracle's argmax, or its oracle logit lies within
    the row's logit tolerance (rel_tol x max |logit|) of the maximum."""
    return token_ok(gpu_tok, ref_logits_row, rel_tol * float(np.max(np.abs(ref_logits_row))))


def need_gpu():
    import pytest
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2602_20217_gb300 import build
    build.build()
