"""The training driver: prox then debias steps with per-step JSON records,
and a checkpoint that restores the CSR arrays exactly."""

import io
import json
import os

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def R():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import run
    return run


@pytest.mark.parametrize("config", ["mlp", "lenet"])
def test_prox_then_debias_records(R, config, tmp_path):
    buf = io.StringIO()
    ckpt = str(tmp_path / "w.npz")
    recs = R.run(config, prox_steps=3, debias_steps=3, batches=2, out=buf, save_path=ckpt)
    lines = [json.loads(l) for l in buf.getvalue().splitlines()]
    assert lines == recs and len(recs) == 6
    assert [r["phase"] for r in recs] == ["prox"] * 3 + ["debias"] * 3
    for r in recs:
        assert np.isfinite(r["loss"]) and r["ms"] > 0 and r["samples_per_s"] > 0 and "status" not in r
        for l in r["layers"]:
            assert 0 <= l["nnz"] <= l["rows"] * l["cols"]
            assert l["compression"] == pytest.approx(l["nnz"] / (l["rows"] * l["cols"]), abs=1e-6)
    # the debias phase keeps every pattern (Section 2.4)
    debias = [[l["nnz"] for l in r["layers"]] for r in recs[3:]]
    assert all(d == debias[0] for d in debias)
    assert debias[0] == [l["nnz"] for l in recs[2]["layers"]]

    # the checkpoint restores the arrays exactly
    net, _ = R.build(config, seed=5, precision=1)
    R.load(net, ckpt)
    data = np.load(ckpt)
    for i, W in enumerate(R.weights(net)):
        (rp, ci, v), t = W.to_host()
        np.testing.assert_array_equal(rp, data[f"row_ptr{i}"])
        np.testing.assert_array_equal(ci, data[f"col_idx{i}"])
        np.testing.assert_array_equal(v.view(np.uint32), data[f"val{i}"].view(np.uint32))
        if t is not None:
            from paper_1905_07931_gb300 import csrtrain as C
            assert C.validate_csr(W, net.ws) is None
    assert os.path.getsize(ckpt) > 0


def test_single_fc_prox_steps(R):
    recs = R.run("single_fc", prox_steps=2, debias_steps=5)
    assert [r["phase"] for r in recs] == ["prox", "prox"]
    assert recs[0]["loss"] is None and recs[0]["layers"][0]["rows"] == 300


def test_load_rejects_a_broken_checkpoint(R, tmp_path):
    ckpt = str(tmp_path / "w.npz")
    R.run("mlp", prox_steps=1, debias_steps=0, batches=1, save_path=ckpt)
    data = dict(np.load(ckpt))
    ci = data["col_idx0"].copy()
    ci[0], ci[1] = ci[1], ci[0]          # unsorted columns in row 0
    data["col_idx0"] = ci
    bad = str(tmp_path / "bad.npz")
    np.savez(bad, **data)
    net, _ = R.build("mlp", seed=0, precision=1)
    with pytest.raises(ValueError, match="not valid"):
        R.load(net, bad)


def test_prefetched_batches_match_direct_copies(R):
    """The input pipeline (copy of batch i+1 on a copy stream while step i
    runs) feeds every step the same batch as a plain copy before the step,
    whether the slot is copied into the network's input (load) or the
    network reads the slot itself (set_input + acquire / release)."""
    from paper_1905_07931_gb300.train import BatchPrefetcher
    cfg_pool = None
    losses, finals = [], []
    for mode in ("direct", "load", "bound"):
        net, cfg = R.build("mlp", seed=3, precision=1)
        if cfg_pool is None:
            cfg_pool = R._pool("mlp", cfg, 3, seed=3)
        pf = BatchPrefetcher(net) if mode != "direct" else None
        out = []
        for i in range(5):
            x, y = cfg_pool[i % 3]
            slot = None
            if pf is None:
                net.x_in.copy_(x.view(net.x_in.shape), non_blocking=True)
                net.labels.copy_(y, non_blocking=True)
            else:
                if i == 0:
                    pf.issue(x, y)
                if mode == "load":
                    pf.load()
                else:
                    slot = pf.acquire()
                    net.set_input(pf.x[slot], pf.y[slot])
                if i + 1 < 5:
                    pf.issue(*cfg_pool[(i + 1) % 3])
            lt = net.step("prox", 0.01, 1e-4)
            if slot is not None:
                pf.release(slot)
            out.append(float(lt[0].item()))
        torch.cuda.synchronize()
        losses.append(out)
        finals.append([W.to_host()[0] for W in R.weights(net)])
    assert losses[0] == losses[1] == losses[2]
    for other in finals[1:]:
        for a, b in zip(finals[0], other):
            for u, v in zip(a, b):
                np.testing.assert_array_equal(u, v)
    with pytest.raises(RuntimeError, match="no batch"):
        BatchPrefetcher(net).load()
    with pytest.raises(ValueError):
        net.set_input(torch.zeros(3, device="cuda"), net.labels)
