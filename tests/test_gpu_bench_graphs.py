"""The bench's trajectory graphs compute what its eager trajectory computes:
one trajectory replayed from the CUDA graphs `bench.Trajectory.capture`
records (the correspondence build on a side stream beside the opening full
steps, which read no correspondence, joined before the first cached step;
then one graph per run of full or cached steps) against the same trajectory
launched eagerly, the final latents compared bitwise.  The correspondence
buffers are cleared before the replay, so a cached step that ran before the
build finished would read empty tiles and change the result."""
import pytest
import torch

import bench
from paper_2608_13255_gb300 import synth

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


@pytest.mark.parametrize("name,B", [("batch128", 4), ("ring12_128", 1)])
def test_trajectory_graphs_equal_eager(gc, name, B):
    w = synth.make_workload(name, B=B)
    traj = bench.Trajectory(w, "cuda")
    x_T = traj.x.clone()
    traj.run()
    torch.cuda.synchronize()
    eager = traj.x.clone()
    assert traj.capture(), "graph capture failed"
    assert traj.build_in_head, "the trajectory opens with a full step: the build belongs in its graph"
    keep = traj.corr._keep
    for key in ("keep", "tile_ptr", "records"):
        keep[key].zero_()
    traj.x.copy_(x_T)
    traj.replay(None)
    torch.cuda.synchronize()
    gc.device_status()
    assert torch.equal(traj.x.view(torch.int16) if traj.x.dtype == torch.bfloat16 else traj.x.view(torch.int32),
                       eager.view(torch.int16) if eager.dtype == torch.bfloat16 else eager.view(torch.int32))
    assert not torch.equal(eager, x_T)
