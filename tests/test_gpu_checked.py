"""The checked build on the GPU: the same seeded cases through the checked
library (every data-dependent index tested against its buffer, run in a child
process with DOPR_CHECKED=1) and through the plain library give the same
scores bit for bit, and no index test fails.  The cases cover short and long
attention tiles (prefixes of 0 to 256 rows, queries up to 300 tokens), the
last layer's score rows, and the offline selection -> build -> score path."""
import os
import subprocess
import sys

import numpy as np
import pytest

from paper_2609_03311_gb300 import build as libbuild
from paper_2609_03311_gb300 import dopr, synth

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SHAPE = synth.ModelShape("checked-g4", n_layers=3, hidden=512, n_q_heads=8, n_kv_heads=2, head_dim=128, ffn=640,
                         vocab=777)


def run_cases() -> dict:
    """Scores of the seeded cases through whichever library this process loads."""
    out = {}
    w = synth.make_weights(SHAPE, seed=7, norms="random")
    cfg = dopr.make_config(SHAPE, max_position=2048)
    model = dopr.Model(cfg, w)
    doc_m = {0: 0, 1: 1, 2: 37, 3: 64, 4: 130, 5: 256}
    store = dopr.Store(cfg, 9, sum(dopr.prefix_bytes(cfg, m) for m in doc_m.values()) + (1 << 16))
    for d, m in doc_m.items():
        store.put(d, *synth.make_prefix(SHAPE, m, d, seed=7))
    rng = np.random.default_rng(7)
    lens = np.concatenate([rng.integers(0, 40, size=40), [300, 200, 129, 1, 0]])
    qo = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    qt = rng.integers(0, SHAPE.vocab, size=int(qo[-1])).astype(np.int32)
    di = rng.integers(0, len(doc_m), size=len(lens)).astype(np.int64)
    out["ragged"] = dopr.score(model, store, qo, qt, di).numpy()
    # offline selection -> prefix build -> online scoring
    dl = [120, 3, 260]
    doff = np.concatenate([[0], np.cumsum(dl)]).astype(np.int32)
    dtok = rng.integers(0, SHAPE.vocab, size=int(doff[-1])).astype(np.int32)
    K = 16
    pos, x, u = dopr.select_prefix_inputs(model, doff, dtok, K, 8)
    out["positions"], out["salience"] = pos, u
    bstore = dopr.Store(cfg, len(dl) - 1, len(dl) * dopr.prefix_bytes(cfg, K))
    dopr.build_prefixes(model, bstore, np.arange(len(dl)), np.arange(0, K * len(dl) + 1, K, dtype=np.int32),
                        x.reshape(-1, SHAPE.hidden))
    bdi = rng.integers(0, len(dl), size=12).astype(np.int64)
    bl = rng.integers(0, 30, size=12)
    bqo = np.concatenate([[0], np.cumsum(bl)]).astype(np.int32)
    bqt = rng.integers(0, SHAPE.vocab, size=int(bqo[-1])).astype(np.int32)
    out["built"] = dopr.score(model, bstore, bqo, bqt, bdi).numpy()
    model.close()
    store.close()
    bstore.close()
    return out


_CHILD = """
import os, sys
sys.path.insert(0, {root!r}); sys.path.insert(0, os.path.join({root!r}, "tests"))
import numpy as np
import test_gpu_checked as t
from paper_2609_03311_gb300 import dopr
assert dopr.lib_path().endswith(os.path.join("_build_checked", "libdopr.so"))
np.savez({out!r}, **t.run_cases())
"""


def test_checked_build_matches_plain_build_bit_for_bit(tmp_path):
    libbuild.build(checked=True)
    out = str(tmp_path / "checked.npz")
    env = dict(os.environ, DOPR_CHECKED="1")
    r = subprocess.run([sys.executable, "-c", _CHILD.format(root=ROOT, out=out)], env=env, cwd=ROOT,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]  # a failed index test raises DOPR_ERR_INTERNAL
    got = np.load(out)
    want = run_cases()
    assert set(got.files) == set(want)
    for k, v in want.items():
        np.testing.assert_array_equal(got[k], v, err_msg=k)
