"""The five workloads at full size, in the benchmark's launch configuration
(messages pushed by reference), against the oracle following a sample of rows
and dense parameters through the same stream (needs a GPU; config 5 holds
~110 GB of device memory)."""
import pytest
import torch

from paper_2205_11048_gb300 import workload as W
from tests import _harness as H

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("n", [2, 3, 4, 5])
def test_full_size_sampled(n):
    cfg = W.config(n)
    free, total = torch.cuda.mem_get_info()
    need = sum(t.rows * t.dim * 4 * (2 if t.opt.kind == 0 else 3) for t in cfg.tables)
    if need > 0.8 * free:
        pytest.skip(f"needs {need / 1e9:.0f} GB of free device memory")
    worst = H.run_fullsize(cfg, steps=3, tol=H.TOL_ONE_STEP)
    print(cfg.name, {k: f"{v:.2e}" for k, v in worst.items()})
