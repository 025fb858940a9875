"""The fused AdamW step on the GPU against the fp64 reference (oracle/adamw.py)
over several steps: tensors of ragged lengths (scalar and float4 paths),
with and without weight decay, NOBLE's per-group learning rates, and bf16
copies of the updated values."""
import numpy as np
import pytest

from oracle import adamw
from paper_2603_06492_gb300 import binding

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2603_06492_gb300.build import build
    build()
    binding.load()


def test_adamw_matches_reference_over_steps():
    import torch
    rng = np.random.default_rng(9)
    sizes = [1, 3, 64, 1000, 4098, 65536, 7, 12, 20, 5, 17, 8, 9, 33, 4, 6, 11, 200]  # 18 tensors: two launches
    mults = [1.0, 5.278, 3.482, 3.0, 5.0] * 4
    lr, wd = 2e-3, 0.01
    host, dev = [], []
    for i, n in enumerate(sizes):
        p = rng.standard_normal(n)
        host.append({"p": p, "m": np.zeros(n), "v": np.zeros(n), "mult": mults[i], "decay": i % 3 != 1})
        d = {k: torch.tensor(p if k == "param" else np.zeros(n), dtype=torch.float32, device="cuda")
             for k in ("param", "exp_avg", "exp_avg_sq")}
        d["grad"] = torch.empty(n, dtype=torch.float32, device="cuda")
        d["param_bf16"] = torch.empty(n, dtype=torch.bfloat16, device="cuda") if i % 2 == 0 else None
        d["lr_mult"], d["decay"] = mults[i], i % 3 != 1
        dev.append(d)
    # the reference starts from the fp32 values the GPU holds
    for h, d in zip(host, dev):
        h["p"] = d["param"].cpu().numpy().astype(np.float64)
    for step in range(1, 5):
        for h, d in zip(host, dev):
            g = rng.standard_normal(h["p"].shape)
            d["grad"].copy_(torch.tensor(g, dtype=torch.float32))
            g32 = d["grad"].cpu().numpy().astype(np.float64)
            h["p"], h["m"], h["v"] = adamw.adamw_step(h["p"], g32, h["m"], h["v"], step, lr * h["mult"],
                                                      weight_decay=wd, decay=h["decay"])
        binding.noble_adamw_step(dev, lr=lr, weight_decay=wd, step=step)
        torch.cuda.synchronize()
        for h, d in zip(host, dev):
            p = d["param"].cpu().numpy().astype(np.float64)
            assert np.max(np.abs(p - h["p"])) <= 1e-6 * max(1.0, np.max(np.abs(h["p"]))), step
            np.testing.assert_allclose(d["exp_avg"].cpu().numpy(), h["m"], rtol=2e-6, atol=1e-7)
            np.testing.assert_allclose(d["exp_avg_sq"].cpu().numpy(), h["v"], rtol=2e-6, atol=1e-8)
            if d["param_bf16"] is not None:
                assert torch.equal(d["param_bf16"], d["param"].to(torch.bfloat16))
    binding.noble_get_device_status(None)


def test_noble_layer_parameter_groups():
    """One optimizer step over a layer's parameters with the multipliers the
    library derives for its shape: every tensor moves by its own group's rate."""
    import torch
    d_in, d_out, r = 256, 512, 32
    k = binding.noble_linear_lr_multipliers(binding.make_desc(64, d_in, d_out, r, "bf16"))
    ref = adamw.lr_multipliers(d_in, d_out, r)
    groups = {"W": (d_out * d_in, k[0], True), "bias": (d_out, k[0], False), "W_down": (r * d_in, k[0], True),
              "W_up": (d_out * r, k[1], True), "M": (r * r, k[2], True), "omega1": (r, k[3], False),
              "phi1": (r, k[4], False)}
    lr = 1e-3
    ts = []
    for name, (n, mult, decay) in groups.items():
        ts.append({"param": torch.zeros(n, device="cuda"), "grad": torch.ones(n, device="cuda"),
                   "exp_avg": torch.zeros(n, device="cuda"), "exp_avg_sq": torch.zeros(n, device="cuda"),
                   "lr_mult": mult, "decay": decay, "name": name})
    binding.noble_adamw_step(ts, lr=lr, step=1)
    torch.cuda.synchronize()
    # first step from zero with g = 1: p = -a / (1 + eps), a = lr * group multiplier
    want = {"W": 1.0, "bias": 1.0, "W_down": 1.0, "W_up": ref["W_up"], "M": ref["M"], "omega1": 3.0, "phi1": 5.0}
    for t in ts:
        got = t["param"].cpu().numpy()
        np.testing.assert_allclose(got, -lr * want[t["name"]] / (1 + 1e-8), rtol=1e-5)
