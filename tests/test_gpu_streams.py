"""Concurrent streams: one training step of a LLaMA-shaped MLP (gate and up
2048 -> 5632 scaled down to 1024 -> 2816, down back, 2048 tokens) enqueued on
four streams with cross-stream waits, as the benchmark schedules it, must give
exactly the bytes of the same launches on one stream.  Every kernel is
deterministic (the token-sliced weight gradient sums its slices in a fixed
order, the changed-code counters are integer sums), so any difference means a
race: shared state between concurrent calls, or a workspace or output read
before the launch that writes it has finished.  Each stream that runs a
weight-gradient call gets its own workspace, as the C ABI requires."""
import pytest
import torch

from paper_2412_04787_gb300 import dqt, inputs

pytestmark = pytest.mark.gpu

T, H, I = 2048, 1024, 2816
PROJ = [("gate", H, I), ("up", H, I), ("down", I, H)]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2412_04787_gb300 import build
    build.build()
    dqt.lib()
    yield
    torch.cuda.synchronize()


def _state():
    dev = torch.device("cuda")
    grid = (-1, 1)
    st = {"X": inputs.normal((T, H), 1.0, seed=1, dtype=torch.bfloat16).to(dev),
          "H": inputs.normal((T, I), 1.0, seed=2, dtype=torch.bfloat16).to(dev)}
    for i, (name, K, N) in enumerate(PROJ):
        W, s_w = dqt.dqt_absmean_init(inputs.normal((N, K), 0.02, seed=10 + i).to(dev), grid)
        st[name] = {"W": W, "s_w": s_w,
                    "m": torch.zeros((N, K), dtype=torch.float32, device=dev),
                    "v": torch.zeros((N, K), dtype=torch.float32, device=dev),
                    "dY": inputs.normal((T, N), 1e-2, seed=20 + i, dtype=torch.bfloat16).to(dev),
                    "img": torch.empty((N, K), dtype=torch.bfloat16, device=dev),
                    "Y": torch.empty((T, N), dtype=torch.bfloat16, device=dev),
                    "dX": torch.empty((T, K), dtype=torch.bfloat16, device=dev),
                    "changed": torch.zeros(1, dtype=torch.int64, device=dev)}
    for src, K in (("X", H), ("H", I)):
        st["aq_" + src] = (torch.empty(T, dtype=torch.float32, device=dev),
                           torch.empty((T, K), dtype=torch.bfloat16, device=dev),
                           torch.empty((T, K), dtype=torch.bfloat16, device=dev))
    nbw = max(dqt.dqt_bwd_dw_img_workspace_size(T, N, K) for _, K, N in PROJ)
    st["ws"] = [torch.empty(max(nbw, 16), dtype=torch.uint8, device=dev) for _ in range(4)]
    return st


def _step(st, streams, step_no=1):
    grid = (-1, 1)
    hp = dqt.adamw(lr=1e-3, step=step_no)
    main = torch.cuda.current_stream()
    s = streams

    def after(stream, *others):
        for o in others:
            if o is not stream:
                e = torch.cuda.Event()
                e.record(o)
                stream.wait_event(e)

    def on(stream, fn):
        with torch.cuda.stream(stream):
            fn()

    def aq(src, stream):
        s_x, img, xdq = st["aq_" + src]
        on(stream, lambda: dqt.dqt_act_quant_images(st[src], None, s_x, img, xdq, want=()))

    def codes(name, stream):
        p = st[name]
        on(stream, lambda: dqt.dqt_codes_to_bf16(p["W"], p["img"]))

    def fwd(name, stream):
        p = st[name]
        s_x, img, _ = st["aq_H" if name == "down" else "aq_X"]
        on(stream, lambda: dqt.dqt_bitlinear_fwd_img(img, s_x, p["img"], p["s_w"], grid, Y=p["Y"]))

    def dx(name, stream):
        p = st[name]
        on(stream, lambda: dqt.dqt_bitlinear_bwd_dx_img(p["dY"], p["img"], p["s_w"], dX=p["dX"]))

    def dw(i, name, stream):
        p = st[name]
        xdq = st["aq_H" if name == "down" else "aq_X"][2]
        ws = st["ws"][s.index(stream)]
        on(stream, lambda: dqt.dqt_bitlinear_bwd_dw_update_img(
            p["dY"], xdq, p["W"], p["s_w"], p["m"], p["v"], hp, dqt.sr_stream(seed=7, tensor_id=i),
            grid, changed_out=p["changed"], ws=ws))

    for x in s:
        after(x, main)
    aq("X", s[0])
    codes("gate", s[1])
    codes("up", s[2])
    codes("down", s[3])
    after(s[1], s[0])
    after(s[2], s[0])
    fwd("gate", s[1])
    fwd("up", s[2])
    after(s[2], s[0], s[1], s[3])
    aq("H", s[2])
    fwd("down", s[2])
    # the weight images are rewritten only in the next step; each dX reads
    # its image while the weight-gradient call beside it updates the codes
    after(s[3], s[2])
    dx("down", s[2])
    dw(2, "down", s[3])
    for x in (s[0], s[1], s[3]):
        after(x, s[2])
    dw(0, "gate", s[1])
    dx("gate", s[0])
    dw(1, "up", s[3])
    dx("up", s[2])
    for x in s:
        after(main, x)


def _snapshot(st):
    out = {}
    for name, _, _ in PROJ:
        for key in ("W", "m", "v", "Y", "dX", "changed"):
            out[name + "." + key] = st[name][key].clone()
    return out


def test_four_streams_equal_one_stream():
    one = torch.cuda.current_stream()
    serial, concurrent = _state(), _state()
    streams = [torch.cuda.Stream() for _ in range(4)]
    for step_no in (1, 2, 3):
        _step(serial, [one] * 4, step_no)
        _step(concurrent, streams, step_no)
    torch.cuda.synchronize()
    dqt.dqt_check_device_status()
    a, b = _snapshot(serial), _snapshot(concurrent)
    for key in a:
        assert torch.equal(a[key], b[key]), key
    # the steps did change codes (the comparison is not of untouched state)
    assert all(int(serial[name]["changed"].item()) > 0 for name, _, _ in PROJ)
