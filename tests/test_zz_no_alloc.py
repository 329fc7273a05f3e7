"""adept_skip_kv_fill_noalloc, the fill entry point for callers that cannot allocate
device memory (e.g. code recording a CUDA graph, or serving loops on a fixed memory
budget): through the C ABI its cache writes equal those of adept_skip_kv_fill on two
calls in a row, and a call above its fixed scratch size is refused with a clear error.

This file is collected last so that a run stopping at the first failure has already run
every other test; it also passes when run alone in a fresh process."""
import numpy as np
import pytest
import torch

import synth
from parity_utils import TOL, assert_rows_close

pytestmark = pytest.mark.gpu


def _cfg():
    return synth.ModelConfig(family=synth.LLAMA, n_layers=8, d_model=256, n_heads=2, head_dim=128, d_ffn=512,
                             vocab=1000, dtype="bf16", max_batch=4, max_seq=160, hsm_m1=512, hsm_m2=1024,
                             block_shuffle_seed=3)


def _inputs(seed, cfg, n):
    h = synth.make_mapped_states(seed, n, cfg.d_model, dtype=torch.bfloat16)
    el = synth.forced_exits_uniform(seed + 1, n, 1, cfg.n_layers, name="el")
    seq = synth.randint(seed + 2, "seq", n, 0, cfg.max_batch - 1).numpy()
    pos = np.zeros(n, dtype=np.int64)
    for b in range(cfg.max_batch):
        idx = np.nonzero(seq == b)[0]
        pos[idx] = np.arange(len(idx)) + (seed % 7)
    dev = lambda x: torch.as_tensor(np.asarray(x), dtype=torch.int32).cuda().contiguous()  # noqa: E731
    return h.cuda().contiguous(), dev(el.numpy()), dev(seq), dev(pos), el.numpy(), seq, pos


def test_noalloc_fill_matches_allocating_fill_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2601_03700_gb300 as adept
    cfg = _cfg()
    W = synth.make_weights(cfg, seed=30)
    ref = adept.Model(cfg, W)      # adept_skip_kv_fill
    new = adept.Model(cfg, W)      # adept_skip_kv_fill_noalloc
    for m in (ref, new):
        adept.adept_seq_reserve(m.h, [cfg.max_seq] * cfg.max_batch)
    for call, (seed, n) in enumerate(((40, 150), (50, 97))):
        h, el, seq, pos, el_h, seq_h, pos_h = _inputs(seed, cfg, n)
        adept.adept_skip_kv_fill(ref.h, n, h, el, seq, pos)
        adept.adept_skip_kv_fill_noalloc(new.h, n, h, el, seq, pos)
        ref.check()
        new.check()
        compared = 0
        for r in range(2, cfg.n_layers + 1):
            for b in range(cfg.max_batch):
                rows = np.nonzero((seq_h == b) & (el_h < r))[0]
                if len(rows) == 0:
                    continue
                kr, vr = ref.read_kv(r, b, 0, cfg.max_seq)
                kn, vn = new.read_kv(r, b, 0, cfg.max_seq)
                p = pos_h[rows]
                assert_rows_close(kn.float().cpu().numpy()[p], kr.float().cpu().numpy()[p], TOL["bf16"],
                                  f"call {call} K layer {r}")
                assert_rows_close(vn.float().cpu().numpy()[p], vr.float().cpu().numpy()[p], TOL["bf16"],
                                  f"call {call} V layer {r}")
                compared += len(rows)
        assert compared > n
    # above the fixed scratch: refused, nothing enqueued
    too_many = int(adept.__dict__.get("NOALLOC_SCRATCH_BYTES", 16 << 20) // (cfg.d_model * 2 + 4)) + 64
    hb = torch.zeros(too_many, cfg.d_model, dtype=torch.bfloat16, device="cuda")
    z = torch.zeros(too_many, dtype=torch.int32, device="cuda")
    with pytest.raises(adept.AdeptError) as ei:
        adept.adept_skip_kv_fill_noalloc(new.h, too_many, hb, z + 1, z, z)
    assert ei.value.status == 3 and "scratch" in str(ei.value)
    ref.close()
    new.close()
