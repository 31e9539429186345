"""Host threads calling the library at once.

Each kernel's shared-memory limit and occupancy answers are set up per device
on first use, behind one lock.  In a fresh process, four threads make their
first calls at the same time (reducer widths that share one kernel
instantiation with different shared-memory sizes, and a draft step), each on
its own stream; their results must equal the same calls made serially
afterwards, bit for bit."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys, threading
import torch
sys.path.insert(0, ROOT)
from paper_2606_26744_gb300 import hdf
from paper_2606_26744_gb300 import workloads as W

torch.cuda.set_device(0)
widths = [(7168, 300), (4096, 500), (2048, 700), (16384, 64)]
red = {d: W.make_reduce_inputs(n, 4, d, "bf16", 0.1, seed=d, device="cuda") for d, n in widths}
cfg = W.scaled(W.CONFIGS["decode"], d=512, n_heads=4, ffn=1024, vocab=4096, batch=3, ctx_len=300)
inp = W.make_draft_inputs(cfg, seed=5)
w = inp["weights"]
wc = {k: v.cuda() for k, v in w.items() if k != "layers"}
wc["layers"] = [{k: v.cuda() for k, v in lw.items()} for lw in w["layers"]]
lens = inp["ctx_lens"]
dH, dWf, db = inp["H"].cuda(), inp["Wf"].cuda(), inp["b"].cuda()
cu, anchor = inp["cu_ctx"].cuda(), inp["anchor"].cuda()
drafter = hdf.Drafter(wc, n_heads=cfg.n_heads, head_dim=cfg.head_dim, rope_max_pos=max(lens) + cfg.block)
torch.cuda.synchronize()

def draft(stream):
    y = hdf.hdf_gated_reduce(dH, dWf, db, stream=stream)
    h = drafter.hdf_draft_block(y, cu, anchor, block=cfg.block, max_ctx=max(lens), stream=stream)
    tok, _, _ = hdf.hdf_lm_head_argmax(h, wc["lm_head"], stream=stream)
    return h, tok

jobs = [("reduce", d) for d, _ in widths] + [("draft", 0)]
results, errors = {}, []
start = threading.Barrier(4)

def worker(k):
    try:
        s = torch.cuda.Stream()
        start.wait()
        with torch.cuda.stream(s):
            for it in range(6):
                kind, d = jobs[(k + it) % len(jobs)]
                if kind == "reduce":
                    i = red[d]
                    out = (hdf.hdf_gated_reduce(i["H"], i["Wf"], i["b"], stream=s),)
                else:
                    out = draft(s)
                s.synchronize()
                results.setdefault((kind, d), []).append(tuple(o.clone() for o in out))
    except Exception as e:  # reported below
        errors.append(repr(e))

ts = [threading.Thread(target=worker, args=(k,)) for k in range(4)]
for t in ts:
    t.start()
for t in ts:
    t.join()
torch.cuda.synchronize()
assert not errors, errors
assert hdf.device_status() == 0
n = 0
for (kind, d), outs in results.items():
    if kind == "reduce":
        i = red[d]
        ref = (hdf.hdf_gated_reduce(i["H"], i["Wf"], i["b"]),)
    else:
        ref = draft(torch.cuda.current_stream())
    torch.cuda.synchronize()
    for out in outs:
        for a, b in zip(out, ref):
            assert torch.equal(a.view(torch.uint8), b.view(torch.uint8)), (kind, d)
            n += 1
print("threads ok", n)
"""


def test_first_calls_from_concurrent_threads_match_serial_calls():
    r = subprocess.run([sys.executable, "-c", f"ROOT = {ROOT!r}\n" + SCRIPT], capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert "threads ok" in r.stdout
