"""Failure detection without a GPU fault: every wait inside the tensor-core
kernels is bounded.  With a wait budget of 0 the first wait that is not
already satisfied gives up; the CTA drains its own copies and MMAs, frees its
tensor memory and returns, and the host reads EC2MOE_ERR_TIMEOUT.  The same
process then runs the layer normally and gets the same output as before."""
import pytest
import torch

from paper_2508_06024_gb300 import build as B
from paper_2508_06024_gb300 import ec2moe as C
from paper_2508_06024_gb300 import synth as S
from paper_2508_06024_gb300.runner import LayerRun

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    B.build()
    C.load()


@pytest.mark.parametrize("cfg", [S.preset("switch_bf16", T=512, seed=31),
                                 S.preset("finegrained_bf16", T=300, seed=32)],
                         ids=["switch", "finegrained"])
def test_zero_wait_budget_times_out_and_recovers(cfg):
    inp = S.make_inputs(cfg, device="cuda")
    run = LayerRun(cfg, inp)
    y_ref = run.forward().clone()
    assert C.ec2moe_last_device_error() == C.OK
    old = C.ec2moe_get_wait_budget()
    try:
        C.ec2moe_set_wait_budget(0)
        run.forward()
        status = C.ec2moe_last_device_error()
    finally:
        C.ec2moe_set_wait_budget(old)
    assert status == C.ERR_TIMEOUT
    assert C.ec2moe_last_device_error() == C.OK  # the error word was read and cleared
    y = run.forward().clone()
    assert C.ec2moe_last_device_error() == C.OK
    assert torch.equal(y, y_ref)


def test_wait_budget_rejects_negative():
    with pytest.raises(C.Ec2moeError) as e:
        C.ec2moe_set_wait_budget(-1)
    assert e.value.status == C.ERR_INVALID_ARG
