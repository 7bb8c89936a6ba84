"""The end-to-end measurement's host-to-device upload (SM loads of pinned host
memory, synth_upload_2d) delivers strided rows byte for byte and leaves the
bytes between destination rows alone."""
import pytest
import torch

from synth.device import upload_2d

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("rows,width,dgap,ctas", [(32, 4096, 512, 32), (3, 16, 48, 1), (7, 65536, 0, 100)])
def test_strided_upload_is_exact(gpu_lib, rows, width, dgap, ctas):
    g = torch.Generator().manual_seed(rows * width + dgap)
    src = torch.randint(0, 256, (rows, width), dtype=torch.uint8, generator=g).pin_memory()
    dpitch = width + dgap
    dst = torch.full((rows * dpitch,), 0x5A, dtype=torch.uint8, device="cuda")
    upload_2d(dst.data_ptr(), dpitch, src.data_ptr(), width, width, rows, ctas)
    torch.cuda.synchronize()
    got = dst.view(rows, dpitch).cpu()
    assert torch.equal(got[:, :width], src)
    assert bool((got[:, width:] == 0x5A).all())
