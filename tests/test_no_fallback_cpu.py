"""The product path has no CPU fallback: every entry point of the binding
refuses CPU tensors before anything runs, a BitLinear layer cannot be built on
the CPU, and a missing library raises instead of degrading.  No GPU needed."""
import pytest
import torch

from paper_2412_04787_gb300 import build, dqt


@pytest.fixture(scope="module")
def built():
    build.build()
    return dqt.lib()


def test_entry_points_refuse_cpu_tensors(built):
    x = torch.zeros(8, 64, dtype=torch.bfloat16)
    w = torch.zeros(64, 64, dtype=torch.int8)
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_act_quant_images(x)
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_codes_to_bf16(w)
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_absmean_init(torch.zeros(64, 64), 1.58)
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_sr_update(torch.zeros(64), torch.zeros(64, dtype=torch.int8), 1.0,
                          torch.zeros(64), torch.zeros(64), dqt.adamw(), dqt.sr_stream(), 1.58)
    # decoder support
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_rope_bf16(torch.zeros(1, 4, 2, 64, dtype=torch.bfloat16), torch.zeros(4, 32, 2))
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_swiglu_bf16(x, x)
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_rmsnorm_bf16(x, torch.ones(64, dtype=torch.bfloat16), 1e-6)
    with pytest.raises(ValueError, match="CUDA"):
        dqt.dqt_cross_entropy_fwd_bf16(x, torch.zeros(8, dtype=torch.int64))


def test_bitlinear_cannot_be_built_on_cpu(built):
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    with pytest.raises(ValueError, match="CUDA"):
        DQTBitLinear(64, 64, bits=1.58, device="cpu")


def test_missing_library_raises(monkeypatch):
    monkeypatch.setattr(dqt, "_LIB_PATH", "/nonexistent/libdqt.so")
    monkeypatch.setattr(dqt, "_lib", None)
    with pytest.raises(RuntimeError, match="no CPU fallback"):
        dqt.lib()


def test_decoder_attention_is_pinned_off_cudnn():
    """The decoder's attention is pinned to FlashAttention / memory-efficient
    attention: cuDNN's fused attention is never selected, whatever PyTorch's
    default priority."""
    from torch.nn.attention import SDPBackend

    from paper_2412_04787_gb300 import decoder
    assert SDPBackend.CUDNN_ATTENTION not in decoder._SDPA_BACKENDS
    assert decoder._SDPA_BACKENDS[0] == SDPBackend.FLASH_ATTENTION
