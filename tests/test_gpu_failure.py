"""Bounded device waits: a wait whose condition never comes true gives up,
reports through the workspace status word, and leaves the context usable.

The failure is made without any fault: the waited-on word is a flag that
nothing sets, or an mbarrier phase that nothing completes.
"""

import time

import pytest
import torch

import oracle
from parity import assert_verify_exact, host_f64, host_int
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def test_met_conditions_return_at_once(rt):
    ws = rt.Workspace(1, 4, 16, 256, torch.bfloat16)
    flag = torch.full((1,), 5, dtype=torch.int32, device="cuda")
    t0 = time.perf_counter()
    rt.retrace_wait_selftest(0, flag, 5, ws)
    rt.retrace_wait_selftest(1, None, 0, ws)
    assert ws.check() == 0
    assert time.perf_counter() - t0 < 0.5


@pytest.mark.parametrize("kind", [0, 1])
def test_expired_wait_reports_and_the_context_stays_usable(rt, kind):
    ws = rt.Workspace(2, 4, 1024, 256, torch.float32)
    flag = torch.zeros((1,), dtype=torch.int32, device="cuda")  # nothing ever raises it
    t0 = time.perf_counter()
    rt.retrace_wait_selftest(kind, flag if kind == 0 else None, 1, ws)
    flags = ws.check()
    elapsed = time.perf_counter() - t0
    assert flags == 1  # bit 0: a bounded wait expired
    assert 0.5 < elapsed < 30.0  # the bound is about one second
    # same context, same workspace after re-initialisation: a correct verification
    rt.retrace_workspace_init(ws)
    cfg = CONFIGS[2].__class__("after-timeout", 2, 4, 1024, 256, "f32", 1.0, "uniform", seed_offset=31)
    x = make_round_inputs(cfg, device="cuda")
    acc = torch.empty(2, dtype=torch.int32, device="cuda")
    com = torch.empty(2, 5, dtype=torch.int32, device="cuda")
    bon = torch.empty(2, dtype=torch.int32, device="cuda")
    tgt = torch.empty(2, 5, dtype=torch.int32, device="cuda")
    rt.retrace_verify(x["logits"], x["draft"], acc, com, bon, ws, target_argmax=tgt)
    torch.cuda.synchronize()
    assert ws.check() == 0
    want = oracle.verify(host_f64(x["logits"]), host_int(x["draft"]))
    assert_verify_exact(want, acc, com, bon, tgt)
