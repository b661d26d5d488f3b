"""bom_get_stats_async / bom_stats_decode: the step's statistics block read
into pinned host memory without a synchronisation gives what bom_get_stats
gives, the latched error code included."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


@pytest.mark.parametrize("name", ["lm_head_small", "tiny_mlp_f32"])
def test_async_stats_match_the_synchronising_read(name):
    wl = I.WORKLOADS[name]
    gpu = G.GpuBom(wl, I.init_params(wl, 1))
    buf = torch.empty(B.bom_stats_transfer_bytes(), dtype=torch.uint8).pin_memory()
    ev = torch.cuda.Event()
    for t in range(1, 3):
        x, y = I.make_batch(wl, seed=1, step=t)
        ref = gpu.step(x, y, t)["stats"]   # the synchronising read
        B.bom_get_stats_async(gpu.model.h, buf)
        ev.record()
        ev.synchronize()
        got = B.bom_stats_decode(buf)
        assert got == ref
        assert got["n_t"] > 0 and np.isfinite(got["loss"])


def test_async_stats_carry_the_latched_error():
    wl = I.LM_HEAD_SMALL
    gpu = G.GpuBom(wl, I.init_params(wl, 2))
    buf = torch.empty(B.bom_stats_transfer_bytes(), dtype=torch.uint8).pin_memory()
    x, y = I.make_batch(wl, seed=2, step=1)
    y = y.copy()
    y[5] = wl.vocab   # out of range
    gpu.step(x, y, 1, check=False)
    B.bom_get_stats_async(gpu.model.h, buf)
    torch.cuda.synchronize()
    got = B.bom_stats_decode(buf, check=False)
    assert got["code"] == B.BOM_ELABEL
    with pytest.raises(B.BomError):
        B.bom_stats_decode(buf)


def test_async_stats_argument_checks():
    wl = I.TINY_MLP_F32
    gpu = G.GpuBom(wl, I.init_params(wl, 0))
    assert B.lib().bom_get_stats_async(None, None, None) == B.BOM_EINVAL
    assert B.lib().bom_get_stats_async(gpu.model.h, None, None) == B.BOM_EINVAL
    assert B.lib().bom_stats_decode(None, None) == B.BOM_EINVAL
