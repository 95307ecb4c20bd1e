"""quan_qconv2d_bwd_data_static, the input gradient for callers that cannot allocate
device memory (its scratch is a fixed 2 MiB buffer in the library's static device memory),
against quan_qconv2d_bwd_data with a caller workspace: two calls in a row on one stream,
each with its own layer, through the C ABI.  Collected last, so that a run stopping at the
first failure has run every other test before it."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import assert_bf16_close, out_f64, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    yield quan.load()


def _layer(name, N, H, W, Cin, Cout, k, s, p, seed):
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(seed, 0))
    d = inputs.layer_inputs(spec)
    dy = to_dev(inputs.grad_output(spec), "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    return spec, dy, w


def _with_workspace(spec, dy, w):
    return quan.qconv2d_backward_data(dy, *w, H=spec.H, W=spec.W, stride=spec.stride,
                                      pad=spec.pad)


def _static(spec, dy, w):
    dx = torch.full((spec.N, spec.H, spec.W, spec.Cin), float("nan"), dtype=torch.bfloat16,
                    device="cuda")
    quan.quan_qconv2d_bwd_data_static(dy, *w, spec.N, spec.H, spec.W, spec.Cin, spec.Cout,
                                      spec.kh, spec.kw, spec.stride, spec.pad, dx)
    return dx


@pytest.mark.parametrize("layers", [
    # two tensor-core layers with different letters: the second call rewrites the scratch
    [("a", 2, 12, 10, 64, 128, 3, 1, 1, 700), ("b", 1, 9, 11, 64, 64, 3, 1, 1, 701)],
    # the CUDA-core route (stride 2), then the tensor-core route
    [("c", 2, 15, 13, 64, 128, 3, 2, 1, 702), ("d", 2, 8, 8, 128, 64, 1, 1, 0, 703)],
], ids=["tc_tc", "simt_tc"])
def test_static_scratch_matches_workspace_entry(layers):
    made = [_layer(*L) for L in layers]
    got = [_static(*m) for m in made]            # two calls in a row
    ref = [_with_workspace(*m) for m in made]
    torch.cuda.synchronize()
    for (spec, _, _), g, r in zip(made, got, ref):
        assert not torch.isnan(g.float()).any(), spec.name
        assert_bf16_close(out_f64(g), out_f64(r), spec.name)


def test_static_scratch_rejects_oversize():
    # 1024 -> 1024 real channels, 3x3: 4.7 MB of transformed letters > 2 MiB
    assert quan.quan_qconv2d_bwd_data_workspace_size(1024, 1024, 3, 3) > 2 << 20
    f = quan.load().quan_qconv2d_bwd_data_static
    st = f(0x10000, 0x20000, 0x30000, 0x40000, 0x50000, 1, 8, 8, 1024, 1024, 3, 3, 1, 1,
           0x9000000, None)
    assert st == quan.QUAN_ERR_UNSUPPORTED
