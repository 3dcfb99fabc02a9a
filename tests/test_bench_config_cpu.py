"""The benchmark's workloads are the configurations they are named for: the
LLaMA-MLP GEMM set (8192 tokens, 2048 -> 5632 -> 2048) and the two decoders,
whose BitLinear weight counts and forward + dX + dW FLOPs per step follow from
their shapes (about 84.9 M weights and 8.35 TFLOP for the 12-layer d-768
decoder at 16 x 1024 tokens, about 1.13 B weights and 111 TFLOP for the
22-layer d-2048 one at 8 x 2048).  No GPU needed."""
import bench


def _bitlinear_weights(sz):
    h, f = sz["hidden"], sz["ffn"]
    return sz["layers"] * (4 * h * h + 3 * h * f)  # q, k, v, o; gate, up, down


def test_mlp_workload_shapes():
    assert (bench.T_TOK, bench.HID, bench.INTER) == (8192, 2048, 5632)
    assert bench.PROJ == [("gate", 2048, 5632), ("up", 2048, 5632), ("down", 5632, 2048)]


def test_decoder_sizes():
    small, large = bench.DECODER_SIZES["130m"], bench.DECODER_SIZES["1b"]
    assert small == dict(layers=12, hidden=768, heads=12, ffn=2048, batch=16, seq=1024)
    assert large == dict(layers=22, hidden=2048, heads=32, ffn=5632, batch=8, seq=2048)
    assert round(_bitlinear_weights(small) / 1e6, 1) == 84.9
    assert round(_bitlinear_weights(large) / 1e9, 2) == 1.13
    for sz, tflop in ((small, 8.35), (large, 111.0)):
        tokens = sz["batch"] * sz["seq"]
        assert abs(6.0 * tokens * _bitlinear_weights(sz) / 1e12 - tflop) / tflop < 0.01


def test_changed_counts_are_labelled_by_call():
    """The bench line's changed-code counts name the weight-gradient call they
    come from: one count for gate and up when they are stacked."""
    import bench
    assert bench.changed_by_projection([5, 0, 7], True) == {"gate+up": 5, "down": 7}
    assert bench.changed_by_projection([5, 6, 7], False) == {"gate": 5, "up": 6, "down": 7}
