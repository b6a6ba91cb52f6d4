"""bench.py's N > 1 path on the CPU: two gloo ranks, one replica each (no data-path collective; only the timing and
token counts are combined): the whole-job figures are the slowest rank's time and the sum of every rank's work."""
import json
import os
import socket
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, sys
sys.path.insert(0, {root!r})
import torch.distributed as dist
import bench
dist.init_process_group("gloo")
rank, world, _ = bench.dist_env()
maxes, sums = bench.aggregate_over_ranks([10.0 + 3 * rank, 2.0 - rank], [100.0 * (rank + 1), 0.5], world, "cpu")
print("RESULT", json.dumps([rank, world, maxes, sums]))
dist.destroy_process_group()
"""


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_combine_max_time_and_summed_work():
    port = str(_free_port())
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2", MASTER_ADDR="127.0.0.1",
                   MASTER_PORT=port)
        procs.append(subprocess.Popen([sys.executable, "-c", CHILD.format(root=ROOT)], cwd=ROOT, env=env,
                                      stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = [p.communicate(timeout=300) for p in procs]
    for p, (out, err) in zip(procs, outs):
        assert p.returncode == 0, err[-2000:]
    res = sorted(json.loads([l for l in out.splitlines() if l.startswith("RESULT")][-1].split(" ", 1)[1])
                 for out, _ in outs)
    for rank, world, maxes, sums in res:
        assert world == 2
        assert maxes == [13.0, 2.0]          # max over ranks, element by element
        assert sums == [300.0, 1.0]          # 100 + 200 tokens, 0.5 + 0.5


def test_single_process_is_unchanged():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.aggregate_over_ranks([4.0], [7, 8], 1) == ([4.0], [7.0, 8.0])
