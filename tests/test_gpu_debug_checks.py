"""The index-checking build (CS_DEBUG_CHECKS; cs_build_flags() bit 0), a stand-in for a
device memory checker: on the tiny search it gives the normal build's results bit for
bit, and an out-of-range compaction index is reported as CS_ERR_BOUNDS with the access
skipped (GPU; each library runs in its own process)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import hashlib, json, sys
import torch
sys.path.insert(0, sys.argv[1])
from paper_2607_23159_gb300 import binding as B, search as S, synth
cfg = synth.CONFIGS["tiny"]
m = cfg.model
flat, _ = synth.make_params(m)
model = B.Model(m, cfg.N)
model.load_weights(flat)
model.set_text_context(torch.from_numpy(synth.text_context(m)).cuda())
st = B.new_state(cfg.N, m.D)
st["x"].copy_(torch.from_numpy(synth.initial_noise(m, range(cfg.N)).reshape(cfg.N, -1)))
skip = torch.zeros(cfg.N, dtype=torch.uint8, device="cuda")
t = S.time_grid(cfg.T)
masks = []
for k in range(1, cfg.T + 1):
    model.search_step(st, k, cfg.T, float(t[k - 1]), float(t[k]), cfg.tau, cfg.K_w, cfg.K_c, skip)
    masks.append(skip.cpu().tolist())
torch.cuda.synchronize()
out = {"checks": B.index_checks(), "x": hashlib.sha1(st["x"].cpu().numpy().tobytes()).hexdigest(),
       "masks": masks, "err": model.device_error()}
if B.index_checks():     # only the index-checking library is given a bad index: it skips the access
    v = torch.zeros(cfg.N, m.D, device="cuda")
    idx = torch.tensor([1, -1], dtype=torch.int32, device="cuda")
    model.dit_forward(st["x"], idx, 2, 0.5, v)
    torch.cuda.synchronize()
    out["bad_err"] = model.device_error()
    out["row1_written"] = bool(v[1].abs().sum() > 0)
    out["other_rows_untouched"] = bool(v[0].abs().sum() == 0 and v[2:].abs().sum() == 0)
print(json.dumps(out))
"""


def _run(variant):
    env = dict(os.environ, CS_LIBRARY_VARIANT=variant)
    r = subprocess.run([sys.executable, "-c", SCRIPT, ROOT], env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return json.loads(r.stdout.strip().splitlines()[-1])


def test_index_checking_build_matches_and_reports_bad_indices():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_23159_gb300 import build as b
    b.build(debug=True)
    rel, dbg = _run("release"), _run("debug")
    assert rel["checks"] is False and dbg["checks"] is True
    assert rel["err"] == 0 and dbg["err"] == 0
    assert dbg["x"] == rel["x"] and dbg["masks"] == rel["masks"]
    assert any(any(s) for s in rel["masks"])            # the rule skipped somewhere
    assert dbg["bad_err"] == 7                          # CS_ERR_BOUNDS
    assert dbg["row1_written"] and dbg["other_rows_untouched"]
