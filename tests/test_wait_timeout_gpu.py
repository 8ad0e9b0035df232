"""Bounded device waits of the persistent chain kernel, made to run out.

The test hook wq4_test_chain_waits shortens every wait of the chain kernel
and makes one stage poll for an epoch that no CTA writes.  The call must
return, wq4_device_status must report the flag-wait bit (bit 1), and the next
normal call must be clean and give the same logits as before, bit for bit.
"""
import time

import numpy as np
import pytest
import torch

from paper_2412_15803_gb300 import synth, wq4
from paper_2412_15803_gb300.model import DecodeModel, ModelShape

pytestmark = pytest.mark.gpu

TINY = ModelShape("tiny", 3, 256, 512, 2, 1, 128, 1001)
FLAG_TIMEOUT = 2


def _decode(model, xd):
    logits = torch.empty((model.batch, model.shape.vocab), dtype=torch.int16, device="cuda")
    rc = model.decode(xd, logits, check=False)
    torch.cuda.synchronize()
    return rc, logits.cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("batch", [1, 2])
@pytest.mark.parametrize("stall", ["o", "down", "lm_head"])
def test_stalled_stage_times_out_and_next_call_is_clean(batch, stall):
    model = DecodeModel(TINY, batch=batch, seed=70 + batch)
    L = TINY.num_layers
    stage = {"o": 4 * 1 + 1, "down": 4 * 2 + 3, "lm_head": 4 * L}[stall]
    x = synth.activations(71, batch, TINY.hidden)
    xd = torch.from_numpy(x.view(np.int16)).cuda()

    assert wq4.wq4_device_status() == 0
    rc, ref = _decode(model, xd)
    assert rc == 0 and wq4.wq4_device_status() == 0

    try:
        wq4.wq4_test_chain_waits(20_000, stage)          # 20 us per wait
        t0 = time.perf_counter()
        rc, _ = _decode(model, xd)
        took = time.perf_counter() - t0
        flags = wq4.wq4_device_status()
    finally:
        wq4.wq4_test_chain_waits(500_000_000, -1)
    assert rc == 0                      # the launch itself is fine
    assert flags & FLAG_TIMEOUT, f"status {flags:#x}"
    assert took < 5.0                    # returned, bounded

    rc, again = _decode(model, xd)
    assert rc == 0 and wq4.wq4_device_status() == 0
    assert np.array_equal(again, ref)

