"""The binding's stream argument: with no stream given, a call goes to the
caller's current stream (the raw handle it reads must be the one
torch.cuda.current_stream() reports, on the default stream and inside a
stream context)."""
import pytest
import torch

from _util import lib

pytestmark = pytest.mark.gpu


def test_default_stream_argument_is_the_current_stream():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    N = lib()
    # The default stream's handle is 0, which ctypes reports as None.
    assert (N._stream(None).value or 0) == torch.cuda.current_stream().cuda_stream
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        assert N._stream(None).value == s.cuda_stream == torch.cuda.current_stream().cuda_stream
    assert N._stream(s).value == s.cuda_stream
