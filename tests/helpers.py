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
    """||got - ref||_inf / ||ref||_inf (per the logits tolerance)."""
    return float(np.max(np.abs(np.asarray(got, np.float64) - ref)) / np.max(np.abs(ref)))


def need_gpu():
    import pytest
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2602_20217_gb300 import build
    build.build()
