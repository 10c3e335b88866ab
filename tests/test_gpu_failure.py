"""The error path, exercised without a GPU fault: the device status word is
set from the host (ks_debug_set_status writes the code a kernel whose bounded
wait gave up would write), and

* every later synchronising call reports it (KS_ERR_TIMEOUT), so a job
  enqueued after it cannot pass for a good one;
* the chained projection kernels of those jobs do no work: the LM head's
  logits of the last good pass are still in place, bit for bit;
* once the word is cleared, the rewound model decodes as before."""
import numpy as np
import pytest

from helpers import need_gpu

pytestmark = pytest.mark.gpu


def test_status_word_voids_later_jobs():
    need_gpu()
    from paper_2602_20217_gb300 import knapspec as ks, synth
    from paper_2602_20217_gb300.configs import ModelShape
    from paper_2602_20217_gb300.model import Model
    shape = ModelShape("status-bf16", 2, 512, 8, 2, 128, 1368, 2000, qk_norm=True, dtype="bf16",
                       rope_theta=500000.0)
    m = Model(shape, max_seq=512, seed=0)
    m.prefill(synth.prompt_tokens(shape, 100, seed=1))
    ref = list(m.decode_greedy(8))
    m.rewind()
    last = m.logits(1)          # the LM head's output of the last greedy pass

    ks.ks_debug_set_status(m.h, 1)
    with pytest.raises(ks.KsError) as e:
        m.decode_greedy(32)
    assert e.value.status == ks.KS_ERR_TIMEOUT
    with pytest.raises(ks.KsError) as e:     # the word stays set
        m.draft(np.ones(shape.n_sublayers, np.uint8), 2)
    assert e.value.status == ks.KS_ERR_TIMEOUT

    ks.ks_debug_set_status(m.h, 0)
    assert np.array_equal(m.logits(1), last)  # no LM-head phase ran meanwhile
    m.rewind()
    assert list(m.decode_greedy(8)) == ref
    m.close()
