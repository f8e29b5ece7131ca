"""LeNet-5 inference, compressed and dense, against the oracle's forward.

The three inference paths of the compressed-vs-dense comparison (CSR weights
with convolutions that read the input in place; the dense im2col + SGEMM
lowering; dense cuDNN) compute the same function; each one's logits on a
batch are checked against the CPU oracle's forward of the same network.
"""

import numpy as np
import pytest

import oracle as O
from tests import chain_bound

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def infer():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_1905_07931_gb300 import infer as I
    return I


def _oracle_logits(ws, bs, images):
    """The oracle's float64 logits (batch x 10) and the element-wise bound on
    a float32 evaluation carried through the network (tests/chain_bound.py)."""
    from paper_1905_07931_gb300.train import lenet_layers
    layers = lenet_layers()
    net = O.Net([dict(l) for l in layers], [])
    pi = 0
    for L in layers:
        if L["kind"] in ("fc", "conv"):
            net.params.append({"W": O.csr_from_dense(ws[pi]), "b": bs[pi]})
            pi += 1
        else:
            net.params.append(None)
    b = images.shape[0]
    z, F, _ = chain_bound.forward_bounds(net, images.reshape(1, b, 28, 28).astype(np.float32), b)
    return z.T, F.T


def test_weights_have_the_paper_counts(infer):
    ws, bs = infer.lenet_weights(0)
    assert [int((w != 0).sum()) for w in ws] == list(infer.SPC_NNZ)
    assert [w.shape for w in ws] == list(infer.SHAPES)


@pytest.mark.parametrize("batch", [32, 7])
def test_inference_paths_against_oracle(infer, batch):
    torch.backends.cuda.matmul.allow_tf32 = False
    torch.backends.cudnn.allow_tf32 = False
    ws, bs = infer.lenet_weights(0)
    rng = np.random.default_rng(batch)
    images = rng.random((batch, 28, 28), dtype=np.float32)
    ref, bound = _oracle_logits(ws, bs, images)
    for cls in (infer.Compressed, infer.DenseGemm, infer.DenseCudnn):
        got = infer.logits_of(cls(ws, bs, batch), images)
        assert got.shape == (batch, 10)
        # element by element: rtol 1e-4 / atol 1e-6, else the carried summation bound
        chain_bound.assert_within(got, ref, bound, what=cls.__name__)


def test_timing_runs_on_a_small_set(infer):
    ws, bs = infer.lenet_weights(0)
    imgs = torch.rand(64, 28, 28, device="cuda")
    paths = {"compressed": infer.Compressed(ws, bs, 32), "dense_gemm": infer.DenseGemm(ws, bs, 32)}
    ms = infer.time_paths(paths, imgs, 32, reps=1, warmup=1)
    assert set(ms) == {"compressed", "dense_gemm"} and all(v > 0 for v in ms.values())
