"""Python face of libknapspec: a model handle whose device memory (weights,
workspace) is allocated by torch.  Marshalling only - the work runs in the
library's CUDA kernels."""
from __future__ import annotations

import numpy as np

from . import knapspec as ks
from . import synth


class Model:
    def __init__(self, shape, max_seq: int, weights: dict | None = None, seed: int = 0,
                 max_rows: int = 16, hist_steps: int = 5, hist_init_rows: int = 8,
                 device: str = "cuda", stream=None):
        import torch
        if not torch.cuda.is_available():
            raise RuntimeError("paper_2602_20217_gb300.Model needs a CUDA device")
        ks.load()
        self.shape = shape
        self.cfg = ks.make_config(shape, max_seq, max_rows, hist_steps, hist_init_rows)
        self.weights = weights if weights is not None else synth.torch_model_weights(shape, seed, device)
        self.kw, self._keep = ks.make_weights(self.weights, shape.n_layers)
        self.ws_bytes = ks.ks_workspace_bytes(self.cfg)
        if self.ws_bytes == 0:
            raise ks.KsError(ks.KS_ERR_INVALID_ARG, "Model", "config rejected by ks_workspace_bytes")
        self.workspace = torch.empty(self.ws_bytes, dtype=torch.uint8, device=device)
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self.h = ks.ks_model_create(self.cfg, self.kw, self.workspace.data_ptr(), self.ws_bytes, self.stream)

    # a1 .. a3
    def prefill(self, tokens) -> int:
        return ks.ks_prefill(self.h, tokens)

    def rewind(self) -> int:
        return ks.ks_rewind(self.h)

    def draft(self, mask, gamma: int):
        return ks.ks_draft(self.h, mask, gamma)

    def draft_sample(self, mask, gamma: int, samp, step: int):
        """Sampled drafts (Sec. 2.1, sampling); the draft distributions stay on the device."""
        return ks.ks_draft_sample(self.h, mask, gamma, samp, step)

    def verify_sample(self, gamma: int, samp, step: int):
        return ks.ks_verify_sample(self.h, gamma, samp, step)

    def draft_dynamic(self, mask, gamma: int, tau_conf: float):
        """Drafts with the dynamic exit (Sec. 3.5): (n_drafted, confidences, tokens)."""
        return ks.ks_draft_dynamic(self.h, mask, gamma, tau_conf)

    def verify(self, drafts, gamma: int):
        return ks.ks_verify(self.h, drafts, gamma)

    def decode_greedy(self, n_tokens: int):
        return ks.ks_decode_greedy(self.h, n_tokens)

    def position(self):
        return ks.ks_model_position(self.h)

    def generate(self, n_tokens: int, gamma: int, mask=None, latency=None, budget_frac: float = 0.5,
                 resolve_every: int = 64, max_steps: int = 0, tpt=None, tau_conf: float = 0.0, sampling=None,
                 dp=None):
        """Speculative decoding: a fixed mask (policy 0), the knapsack policy
        (policy 1, latency given) or the TPT stage (policy 2, latency and
        tpt = (n_candidates, max_gamma) given); tau_conf > 0 adds the dynamic
        drafting exit; sampling (a KsSampling) selects sampling mode; dp = (max_gamma, tau,
        max_states, max_rows) with a latency selects the hidden-state DP policy."""
        n = self.shape.n_sublayers
        keep = []
        if latency is None:
            m = np.ascontiguousarray(mask if mask is not None else np.ones(n), dtype=np.uint8)
            keep.append(m)
            lat, _ = ks.latency(0, 1.0, 0.0, 1.0)
            p = ks.KsSpecParams(gamma, 0, m.ctypes.data_as(ks.C.POINTER(ks.C.c_uint8)), lat, 0.0, 1, max_steps,
                                0, 0, float(tau_conf))
        else:
            lat, u = latency
            keep.append(u)
            if tpt is None:
                p = ks.KsSpecParams(gamma, 1, None, lat, float(budget_frac), int(resolve_every), max_steps,
                                    0, 0, float(tau_conf))
            else:
                p = ks.KsSpecParams(gamma, 2, None, lat, 0.0, int(resolve_every), max_steps,
                                    int(tpt[0]), int(tpt[1]), float(tau_conf))
        if sampling is not None:
            p.sampling = sampling
        scratch = None
        if dp is not None:
            # policy 3: the hidden-state DP every resolve_every steps; dp = (max_gamma, tau, max_states, max_rows)
            import torch
            D, tau, max_states, max_rows = dp
            nb = ks.load().ks_dp_scratch_bytes(self.h, max_states, max_rows)
            scratch = torch.empty(nb + 256, dtype=torch.uint8, device=self.workspace.device)
            p.policy = 3
            p.tpt_max_gamma = int(D)
            p.dp_scratch = (scratch.data_ptr() + 255) // 256 * 256
            p.dp_scratch_bytes = nb
            p.dp_tau = float(tau)
            p.dp_max_states = int(max_states)
            p.dp_max_rows = int(max_rows)
        out = ks.ks_generate_speculative(self.h, p, n_tokens)
        del scratch
        return out

    def select_dp(self, latency, max_gamma: int, tau: float = 0.5, max_states: int = 128, max_rows: int = 32):
        """Alg. 1 on the current history and the TPT grid over its candidates:
        (mask, gamma, tpt, js, alphas, candidate masks)."""
        import torch
        lat, _u = latency
        nb = ks.load().ks_dp_scratch_bytes(self.h, max_states, max_rows)
        if nb == 0:
            raise ValueError("bad max_states / max_rows")
        scratch = torch.empty(nb + 256, dtype=torch.uint8, device=self.workspace.device)
        ptr = (scratch.data_ptr() + 255) // 256 * 256
        return ks.ks_select_dp(self.h, lat, self.shape.n_sublayers, tau, max_gamma, max_states, max_rows, ptr, nb)

    def select_tpt(self, latency, n_candidates: int, max_gamma: int):
        """The TPT stage on the current history: (mask, gamma, tpt, alphas, candidates)."""
        lat, _u = latency
        return ks.ks_select_tpt(self.h, lat, self.shape.n_sublayers, n_candidates, max_gamma)

    def history_similarities(self):
        import torch
        sims = torch.empty(self.shape.n_sublayers, dtype=torch.float32, device=self.workspace.device)
        r = ks.ks_history_similarities(self.h, sims)
        self.stream.synchronize()
        return sims.cpu().numpy(), r

    # diagnostics
    def logits(self, rows: int):
        return ks.ks_debug_read(self.h, 0, 0, 0, rows, np.zeros((rows, self.shape.vocab), np.float32))

    def residual(self, rows: int):
        return ks.ks_debug_read(self.h, 1, 0, 0, rows, np.zeros((rows, self.shape.d_model), np.float32))

    def kv(self, layer: int, start: int, count: int, which: str = "k"):
        sh = self.shape
        dt = np.float32 if sh.dtype == "f32" else np.uint16
        out = np.zeros((sh.n_kv_heads, count, sh.head_dim), dt)
        ks.ks_debug_read(self.h, 2 if which == "k" else 3, layer, start, count, out)
        if sh.dtype == "bf16":
            out = (out.astype(np.uint32) << 16).view(np.float32)
        return out

    def history(self):
        """X^(0..2L) of the rows in the history ring: [2L+1, r, d] fp32."""
        sh = self.shape
        r = np.zeros(1, np.int32)
        ks.ks_debug_read(self.h, 4, 0, 0, 0, r)
        buf = np.zeros((sh.n_sublayers + 1, int(r[0]), sh.d_model), np.float32)
        return ks.ks_debug_read(self.h, 4, 0, 0, int(r[0]), buf)

    def launches(self) -> int:
        return ks.ks_launch_count(self.h)

    def close(self):
        if getattr(self, "h", None):
            ks.ks_model_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
