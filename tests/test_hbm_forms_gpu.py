"""resbm_measure_hbm_form (the HBM access-form probe) through the C ABI: every form runs as one
launch, reports no wait timeout, and moves the bytes it claims to. Write forms cover every byte
of b with 0xA5; the copy makes b equal to a; read forms leave b alone. Sizes give CTAs
unequal runs (more boxes than SMs but not a multiple), and fewer stages than CTAs."""
import pytest
import torch

from paper_2604_11947_gb300 import resbm

pytestmark = pytest.mark.gpu

MIB = 1 << 20


@pytest.mark.parametrize("mib", [1, 3, 17])
@pytest.mark.parametrize("form", sorted(resbm.HBM_FORMS))
def test_form_moves_its_bytes(form, mib):
    n = mib * MIB
    g = torch.Generator(device="cuda").manual_seed(mib)
    a = torch.randint(0, 256, (n,), dtype=torch.uint8, device="cuda", generator=g)
    a[a == 0xA5] = 0x11   # no byte of a equals the write pattern
    b = torch.zeros(n, dtype=torch.uint8, device="cuda")
    a0 = a.clone()
    before = resbm.resbm_kernel_launches()
    resbm.resbm_measure_hbm_form(form, a, b)
    torch.cuda.synchronize()
    assert resbm.resbm_kernel_launches() - before == 1
    assert resbm.resbm_device_error() == 0
    assert torch.equal(a, a0)   # a is never written
    if form.startswith("write"):
        assert bool((b == 0xA5).all())
    elif form.startswith("copy"):
        assert torch.equal(b, a)
    elif form == "read_v4":
        assert int(b[4:].count_nonzero()) == 0   # at most the 4-byte sink
    else:
        assert int(b.count_nonzero()) == 0


def test_form_rejects_unequal_buffers():
    a = torch.zeros(MIB, dtype=torch.uint8, device="cuda")
    b = torch.zeros(2 * MIB, dtype=torch.uint8, device="cuda")
    with pytest.raises(ValueError):
        resbm.resbm_measure_hbm_form("copy_v4", a, b)
