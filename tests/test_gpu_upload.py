"""The end-to-end upload copies q only in the rows the verification reads (dcd.upload_inputs:
rows of sampled sequences whose node has a child).  With every other row NaN on the device,
every output equals that of a call on fully copied inputs, bit for bit."""

import numpy as np
import pytest
import torch

from paper_2608_12913_gb300 import dcd, workloads

pytestmark = pytest.mark.gpu

KEYS = ("z_exp", "z_ama", "q", "tokens", "parents", "alpha", "beta", "temperature")


@pytest.mark.parametrize("distinct", [False, True])
def test_upload_copies_only_read_rows_of_q(distinct):
    w = workloads.make_config(3, B=6, V=5003, seed=41)  # sequences alternate greedy / sampled
    host = {k: getattr(w, k).pin_memory() for k in KEYS}
    full = {k: v.to("cuda") for k, v in host.items()}
    part = {k: torch.empty_like(v, device="cuda") for k, v in host.items()}
    part["q"].fill_(float("nan"))
    nbytes = dcd.upload_inputs(host, part, w.N)
    expect = sum(v.numel() * v.element_size() for k, v in host.items() if k != "q")
    read_rows = w.sampled_rows_with_children()  # the rows whose q the rules read
    assert nbytes == expect + read_rows * w.V * 4

    def run(d):
        o = dcd.dcd_verify_sample(d["z_exp"], d["z_ama"], d["q"], d["tokens"], d["parents"], d["alpha"],
                                  d["temperature"], w.seed, 7, d["beta"], residual=True, distinct=distinct)
        torch.cuda.synchronize()
        return {k: v.cpu().numpy() for k, v in o.items() if k != "workspace"}

    a, b = run(full), run(part)
    for k in a:
        assert np.array_equal(a[k], b[k], equal_nan=True), k
    assert np.isfinite(b["cd_lse"]).all()

