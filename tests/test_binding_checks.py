"""The Python binding hands the library only pointers its kernels can use: every
tensor argument is checked (CUDA, current device, contiguous, dtype, length)
before any call, so a host tensor, int32 offsets where int64 are read, or a
short output buffer raises in Python instead of reaching a kernel."""
import pytest
import torch

from paper_2609_36830_gb300 import pace


def test_host_tensors_and_non_tensors_are_refused_before_any_call():
    with pytest.raises(ValueError, match="CUDA"):
        pace._arg(torch.zeros(3, dtype=torch.int64), torch.int64, 3, "offsets")
    with pytest.raises(TypeError):
        pace._arg([0, 1, 2], torch.int64, 3, "offsets")
    assert pace._arg(None, torch.int64, 3, "offsets") is None
    with pytest.raises(ValueError, match="CUDA"):
        pace.make_batch(torch.tensor([0, 4], dtype=torch.int64), 4)


@pytest.mark.gpu
def test_device_tensors_wrong_dtype_length_layout():
    dev = "cuda"
    off32 = torch.tensor([0, 4], dtype=torch.int32, device=dev)
    with pytest.raises(ValueError, match="int64"):
        pace.make_batch(off32, 4)
    off = torch.tensor([0, 4], dtype=torch.int64, device=dev)
    with pytest.raises(ValueError, match="at least 4"):
        pace.make_batch(off, 4, mask=torch.ones(3, dtype=torch.uint8, device=dev))
    b = pace.make_batch(off, 4)
    hidden = torch.zeros(4, 64, dtype=torch.bfloat16, device=dev)
    w = torch.zeros(256, 64, dtype=torch.bfloat16, device=dev)
    y = torch.zeros(4, dtype=torch.int32, device=dev)
    with pytest.raises(ValueError, match="int32"):
        pace.token_logprob(b, hidden, w, y.to(torch.int64))
    with pytest.raises(ValueError, match="contiguous"):
        pace.token_logprob(b, hidden, torch.zeros(64, 256, dtype=torch.bfloat16, device=dev).t(), y)
    with pytest.raises(ValueError, match="bfloat16"):
        pace.token_logprob(b, hidden.float(), w, y)
    with pytest.raises(ValueError, match="rows"):
        pace.token_logprob(b, hidden[:3], w, y)
    with pytest.raises(ValueError, match="at least 4"):
        pace.token_logprob(b, hidden, w, y, logprob=torch.zeros(3, device=dev))
    lp = pace.token_logprob(b, hidden, w, y)  # the same call with valid arguments runs
    torch.cuda.synchronize()
    assert torch.allclose(lp, torch.full_like(lp, -5.545177), atol=1e-4)  # uniform: -ln 256
