"""Failure detection on the GPU without a fault: every wait inside a kernel is bounded, and a wait
that runs out records code 2 (with the wait's site) in the device error word and lets the kernel
return, so the context stays usable. The self-test entry point waits with the kernels' own bounded
wait on an mbarrier that nothing arrives at (no copy or MMA in flight), a few milliseconds long."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_2608_06146_gb300 import build as pbuild
from paper_2608_06146_gb300 import inputs
from paper_2608_06146_gb300 import padoc_attn as pa
from paper_2608_06146_gb300.engine import DecodePlan

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _build():
    pbuild.build()
    pa.load_library()


def test_bounded_wait_runs_out_reports_code_2_and_site_then_decode_is_exact():
    pa.padoc_check_device_errors()                # start from a clear error word
    gave_up = torch.zeros(1, dtype=torch.int32, device=DEV)
    pa.padoc_selftest_wait_timeout(3000, 91, gave_up)
    with pytest.raises(pa.PadocError) as e:
        pa.padoc_check_device_errors()
    assert e.value.status == 5 and e.value.device_code == 2 and e.value.device_detail == 91
    assert int(gave_up.item()) == 64              # every thread of the CTA gave up and returned
    pa.padoc_check_device_errors()                # the word was cleared

    # the context is still usable: a normal decode step afterwards matches the oracle
    wl = inputs.decode_page()
    di = inputs.decode_inputs(wl, 41)
    plan = DecodePlan(wl.pages, 16, 2, 128, DEV)
    S = plan.num_streams
    out = torch.full((S, 16, 128), float("nan"), dtype=torch.bfloat16, device=DEV)
    lse = torch.full((S, 16), float("nan"), dtype=torch.float32, device=DEV)
    scale = 1.0 / math.sqrt(128)
    plan.run(di.k_pool.to(DEV), di.v_pool.to(DEV), torch.from_numpy(di.page_table).to(DEV),
             torch.from_numpy(di.stream_table).to(DEV), di.q.to(DEV), scale, out, lse)
    pa.padoc_check_device_errors()
    ref_o, ref_l = oracle.decode_pages(wl.pages, di, scale)
    assert np.abs(out.float().cpu().numpy() - ref_o).max() <= 1.5e-2
    assert np.abs(lse.cpu().numpy() - ref_l).max() <= 1e-3


def test_two_timeouts_in_a_row_keep_the_first_site():
    # the first error recorded wins: two timeouts in a row report the first one's site
    pa.padoc_check_device_errors()
    gave_up = torch.zeros(1, dtype=torch.int32, device=DEV)
    pa.padoc_selftest_wait_timeout(1000, 7, gave_up)
    pa.padoc_selftest_wait_timeout(1000, 8, gave_up)
    with pytest.raises(pa.PadocError) as e:
        pa.padoc_check_device_errors()
    assert e.value.device_code == 2 and e.value.device_detail == 7
    assert int(gave_up.item()) == 128
