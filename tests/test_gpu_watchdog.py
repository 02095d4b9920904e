"""Failure detection without a GPU fault: a bounded tensor-core wait runs
out on purpose (an mbarrier that nothing arrives on, a short test limit),
the kernel raises the watchdog flag and returns, featfix_get_log reports
FEATFIX_ERR_CUDA, and the context keeps producing the same results."""

import pytest
import torch

from paper_2607_27842_gb300 import featfix as ff, synthetic as syn

from .gpu_helpers import Case

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_is_reported(cuda):
    c = Case(syn.workload("tiny"))
    try:
        c.schedule("featfix")
        before = c.sample(seed=3).clone()
        ff.featfix_get_log(c.ctx)                      # clean: no watchdog
        ff.featfix_debug_watchdog_probe(c.ctx, 2_000_000)   # 2 ms
        with pytest.raises(ff.FeatFixError) as e:
            ff.featfix_get_log(c.ctx)
        assert e.value.status == ff.ERR_CUDA
        assert "watchdog" in str(e.value)
        # the flag is cleared once reported and the context is still usable
        after = c.sample(seed=3)
        logs, counters = ff.featfix_get_log(c.ctx)
        assert torch.equal(before, after)
        assert counters["steps_done"] == c.wl.steps
        with pytest.raises(ff.FeatFixError) as e:
            ff.featfix_debug_watchdog_probe(c.ctx, 10)      # below 1 us: rejected, nothing launched
        assert e.value.status == ff.ERR_INVALID_ARG
        ff.featfix_get_log(c.ctx)
    finally:
        c.close()
