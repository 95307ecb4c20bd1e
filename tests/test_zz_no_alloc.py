"""quan_qconv2d_bwd_data_static, the input gradient for callers that cannot allocate
device memory (its scratch is a fixed 2 MiB buffer in the library's static device memory),
against quan_qconv2d_bwd_data given a caller workspace of the same 2 MiB: two calls in a
row on one stream, each with its own layer, through the C ABI.  The two entry points run
the same kernels on the same inputs, so their outputs must be equal bit for bit; both are
also held to the bf16 tolerance of the fp64 oracle's input gradient.  Collected last, so
that a run stopping at the first failure has run every other test before it."""
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import assert_bf16_close, host_f64, out_f64, to_dev

pytestmark = pytest.mark.gpu

SCRATCH = 2 << 20  # bytes of the library's static scratch


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    quan.load()
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    yield


def _layer(name, N, H, W, Cin, Cout, k, s, p, seed):
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(seed, 0))
    d = inputs.layer_inputs(spec)
    dy_bits = inputs.grad_output(spec)
    dy = to_dev(dy_bits, "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    return spec, d, dy_bits, dy, w


def _nan_dx(spec):
    return torch.full((spec.N, spec.H, spec.W, spec.Cin), float("nan"), dtype=torch.bfloat16,
                      device="cuda")


def _static(spec, dy, w):
    dx = _nan_dx(spec)
    quan.quan_qconv2d_bwd_data_static(dy, *w, spec.N, spec.H, spec.W, spec.Cin, spec.Cout,
                                      spec.kh, spec.kw, spec.stride, spec.pad, dx)
    return dx, quan.quan_last_path()


def _with_workspace(spec, dy, w):
    # the workspace entry point with the static buffer's capacity: same route, same kernels
    ws = torch.empty(SCRATCH, dtype=torch.uint8, device="cuda")
    dx = _nan_dx(spec)
    quan.quan_qconv2d_bwd_data(dy, *w, spec.N, spec.H, spec.W, spec.Cin, spec.Cout, spec.kh,
                               spec.kw, spec.stride, spec.pad, ws, SCRATCH, dx)
    return dx, quan.quan_last_path()


TC, SIMT = quan.QUAN_PATH_TC, quan.QUAN_PATH_SIMT


@pytest.mark.parametrize("layers", [
    # two stride-1 tensor-core layers with different letters: the second call rewrites the
    # scratch the first one left
    [("a", 2, 12, 10, 64, 128, 3, 1, 1, 700, TC), ("b", 1, 9, 11, 64, 64, 3, 1, 1, 701, TC)],
    # a strided layer whose letters fit but whose spread-out dy (8 x 56 x 56 x 128 bf16,
    # 6.4 MB) does not: the CUDA-core route; then a 1x1 tensor-core layer
    [("c", 8, 56, 56, 64, 128, 3, 2, 1, 702, SIMT), ("d", 2, 8, 8, 128, 64, 1, 1, 0, 703, TC)],
    # a strided layer whose letters and spread-out dy both fit: the tensor-core route of a
    # strided forward, then the CUDA-core route again
    [("e", 2, 15, 13, 64, 128, 3, 2, 1, 704, TC), ("f", 6, 40, 40, 64, 128, 3, 2, 1, 705, SIMT)],
], ids=["tc_tc", "simt_tc", "stridedtc_simt"])
def test_static_scratch_matches_workspace_entry_and_oracle(layers):
    made = [(_layer(*L[:10]), L[10]) for L in layers]
    got = []
    for (spec, _, _, dy, w), want_path in made:  # two static calls in a row
        dx, path = _static(spec, dy, w)
        assert path == want_path, (spec.name, path)
        got.append(dx)
    ref = []
    for (spec, _, _, dy, w), want_path in made:
        dx, path = _with_workspace(spec, dy, w)
        assert path == want_path, (spec.name, path)
        ref.append(dx)
    torch.cuda.synchronize()
    assert quan.quan_device_status()[0] == quan.QUAN_OK
    for ((spec, d, dy_bits, _, _), _), g, r in zip(made, got, ref):
        assert not torch.isnan(g.float()).any(), spec.name
        assert torch.equal(g, r), spec.name
        f = lambda k: host_f64(d[k], "bf16")
        want = oracle.qconv2d_bwd_data(host_f64(dy_bits, "bf16"), f("wr"), f("wi"), f("wj"),
                                       f("wk"), H=spec.H, W=spec.W, stride=spec.stride,
                                       pad=spec.pad)
        assert_bf16_close(out_f64(g), want, spec.name)


def test_static_scratch_rejects_oversize():
    # 1024 -> 1024 real channels, 3x3: 4.7 MB of transformed letters > 2 MiB; the call is
    # rejected on the host, before any launch (real device tensors all the same)
    assert quan.quan_qconv2d_bwd_data_workspace_size(1024, 1024, 3, 3) > SCRATCH
    dy = torch.zeros((1, 8, 8, 1024), dtype=torch.bfloat16, device="cuda")
    w = [torch.zeros((256, 3, 3, 256), dtype=torch.bfloat16, device="cuda") for _ in range(4)]
    dx = torch.zeros((1, 8, 8, 1024), dtype=torch.bfloat16, device="cuda")
    st = quan.load().quan_qconv2d_bwd_data_static(dy.data_ptr(), *(t.data_ptr() for t in w), 1,
                                                  8, 8, 1024, 1024, 3, 3, 1, 1, dx.data_ptr(),
                                                  None)
    assert st == quan.QUAN_ERR_UNSUPPORTED
    assert int(dx.float().abs().sum()) == 0  # nothing was written
