"""Runs a few decode steps with whichever libpced the environment selects
(PCED_LIB=checked: the bounds-checked build) and prints, per case, the device
status word, the chosen tokens and a hash of the final hidden states as one
JSON line.  Used by test_gpu_checked.py in a child process."""
import hashlib
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

CASES = [("tiny", {}, 4, {}), ("llama8", {"L": 4}, 2, {}), ("tiny", {}, 3, {"aggregation": 1}),
         ("tiny", {}, 3, {"dynamic_beta": True}), ("llama8", {"L": 2}, 2, {"paged": 64})]


def run_cases():
    import torch
    import paper_2601_08670_gb300 as pced
    import synth
    out = []
    for name, over, steps, kw in CASES:
        kw = dict(kw)
        paged = kw.pop("paged", 0)
        w = synth.get(name, **over)
        t = synth.device_inputs(w, "cuda", paged=paged)
        dm = pced.dims(w.B, w.N, w.L, w.Hq, w.Hkv, w.D, w.V)
        dec = pced.decoder_from_inputs(dm, t, gamma=w.gamma, max_steps=w.steps, bos=w.bos, keep_hidden=True, **kw)
        for _ in range(steps):
            dec.step()
        torch.cuda.synchronize()
        h = dec.hidden.cpu().view(torch.int16).numpy().tobytes()
        out.append({"case": f"{name}{over}{kw}{'paged' if paged else ''}", "status": dec.status(),
                    "tokens": dec.history[:, :steps].cpu().numpy().tolist(),
                    "hidden": hashlib.sha256(h).hexdigest()[:16]})
        del dec, t
        torch.cuda.empty_cache()
    return out


if __name__ == "__main__":
    print(json.dumps(run_cases()))
