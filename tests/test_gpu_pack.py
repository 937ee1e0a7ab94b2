"""Anchor-row pack / unpack kernels (Sec. 3.2, batch-sliced anchor forward)
against the oracle's definition: bit-exact for every dtype, for row sizes
that allow 16-byte, 4-byte and only 1-byte copies."""
import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def gc():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_13255_gb300 import build as gbuild
    gbuild.build()
    from paper_2608_13255_gb300 import geocache
    geocache.load()
    return geocache


CASES = [
    (torch.bfloat16, (3, 6, 4, 64, 64), [0, 3]),    # latents, 16-byte rows
    (torch.float32, (2, 12, 16, 32, 32), [1, 4, 7, 10]),
    (torch.int32, (4, 6, 3), [2, 5]),               # structural indices, 12-byte rows
    (torch.uint8, (3, 6, 7, 5, 3), [0, 1, 4]),      # 105-byte rows
    (torch.float32, (1, 64, 2, 8, 8), list(range(0, 64, 5))),
]


@pytest.mark.parametrize("dtype,shape,anchors", CASES, ids=[str(i) for i in range(len(CASES))])
def test_pack_unpack_bit_exact(gc, dtype, shape, anchors):
    g = torch.Generator().manual_seed(3)
    if dtype.is_floating_point:
        src = torch.randn(shape, generator=g).to(dtype)
    else:
        src = torch.randint(0, 100, shape, generator=g).to(dtype)
    raw = lambda t: t.contiguous().view(torch.uint8).numpy() if t.dtype != torch.uint8 else t.numpy()
    d_src = src.cuda()
    packed = torch.empty((shape[0], len(anchors)) + shape[2:], dtype=dtype, device="cuda")
    gc.pack_anchors(d_src, packed, anchors)
    torch.cuda.synchronize()
    ref = oracle.pack_anchors(raw(src).reshape(shape[0], shape[1], -1), anchors)
    np.testing.assert_array_equal(raw(packed.cpu()).reshape(ref.shape), ref)
    # unpack fresh rows into a copy of src: anchor rows replaced, others kept
    new = torch.randint(0, 100, packed.shape, generator=g).to(dtype).cuda()
    out = d_src.clone()
    gc.unpack_anchors(new, out, anchors)
    torch.cuda.synchronize()
    ref2 = oracle.unpack_anchors(raw(new.cpu()).reshape(ref.shape), raw(src).reshape(shape[0], shape[1], -1), anchors)
    np.testing.assert_array_equal(raw(out.cpu()).reshape(ref2.shape), ref2)
