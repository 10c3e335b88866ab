"""Small, self-contained decode case for profilers (ncu) and kernel timing.

Runs a workload's model shape truncated to a few layers (full width, full
vocabulary) with a short prompt, then a few speculative steps, and prints the
average CUDA-event time of each kernel class.  Sized to keep a profiler's
capture short: a few GB of device memory, a few hundred kernel launches.

  python -m paper_2602_20217_gb300.profile --workload llama8b-4k --layers 2 --prompt 512 --steps 3

The speculative steps run inside an NVTX range named "decode", so a profiler
can skip the prefill (ncu --nvtx --nvtx-include "decode/").
"""
from __future__ import annotations

import argparse
import json

import numpy as np


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="llama8b-4k")
    ap.add_argument("--layers", type=int, default=2)
    ap.add_argument("--prompt", type=int, default=512)
    ap.add_argument("--steps", type=int, default=3)
    ap.add_argument("--gamma", type=int, default=4)
    ap.add_argument("--vocab", type=int, default=0, help="override the vocabulary (0: keep)")
    ap.add_argument("--timing", action="store_true", help="bracket every launch with CUDA events")
    args = ap.parse_args()

    import torch

    from . import build, knapspec as ks, synth
    from .configs import WORKLOADS, truncated
    from .model import Model
    build.build()
    wl = WORKLOADS[args.workload]
    sh = truncated(wl.shape, args.layers)
    if args.vocab:
        from dataclasses import replace
        sh = replace(sh, vocab=args.vocab)
    prompt = synth.prompt_tokens(sh, args.prompt, seed=wl.prompt_seed)
    m = Model(sh, max_seq=args.prompt + (args.steps + 2) * (args.gamma + 1) + 16, seed=wl.weight_seed)
    m.prefill(prompt)
    if args.timing:
        for k in ks.KLASS.values():   # every class: the projections then run one per launch
            ks.ks_kernel_timing(m.h, k, True)
    mask = np.array([0, 1] * sh.n_layers, np.uint8)   # draft: MLP sublayers only
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_push("decode")              # profilers can filter on this range
    out, st, acc = m.generate(1 << 20, args.gamma, mask=mask, max_steps=args.steps)
    torch.cuda.synchronize()
    torch.cuda.nvtx.range_pop()
    res = {"workload": wl.name, "layers": sh.n_layers, "prompt": args.prompt, "steps": int(st.steps),
           "accepted": int(st.accepted)}
    if args.timing:
        res["avg_us"] = {name: round(1e3 * ms / max(1, n), 2)
                         for name, (n, ms) in ((nm, ks.ks_kernel_time(m.h, k)) for nm, k in ks.KLASS.items())}
    print(json.dumps(res))
    m.close()


if __name__ == "__main__":
    main()
