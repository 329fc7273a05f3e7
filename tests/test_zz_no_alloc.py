"""adept_skip_kv_fill_noalloc, the fill entry point for callers that cannot allocate device
memory (code recording a CUDA graph, where cudaMalloc and the synchronisation of cudaFree
cannot be captured; serving loops that run on a fixed memory budget or their own allocator).

Through the C ABI, on two calls in a row per size:
  * its cache writes equal those of adept_skip_kv_fill bit for bit where both take the
    tensor-core path (more than 8 tokens), and equal the oracle's K/V projection of s~
    within the bf16 tolerance at every size, including the small-row paths (1, 5, 24, 40
    tokens: 2-D A boxes of 8 to 64 rows, which the allocating fill does not use there);
  * a call above its fixed scratch size is refused with a clear error;
  * it adds its launches to adept_launch_count.

This file is collected last so that a run stopping at the first failure has already run
every other test; it also passes when run alone in a fresh process."""
import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
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
    return h, dev(el.numpy()), dev(seq), dev(pos), el.numpy(), seq, pos


@pytest.mark.parametrize("sizes", [(150, 97), (40, 24), (5, 1)])
def test_noalloc_fill_matches_allocating_fill_and_oracle_on_two_calls(sizes):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2601_03700_gb300 as adept
    cfg = _cfg()
    W = synth.make_weights(cfg, seed=30)
    om = O.OracleModel(cfg, W)
    ref = adept.Model(cfg, W)      # adept_skip_kv_fill
    new = adept.Model(cfg, W)      # adept_skip_kv_fill_noalloc
    for m in (ref, new):
        adept.adept_seq_reserve(m.h, [cfg.max_seq] * cfg.max_batch)
    for call, n in enumerate(sizes):
        seed = 40 + 10 * call + n
        h, el, seq, pos, el_h, seq_h, pos_h = _inputs(seed, cfg, n)
        hd = h.cuda().contiguous()
        adept.adept_skip_kv_fill(ref.h, n, hd, el, seq, pos)
        adept.adept_launch_count(new.h)
        adept.adept_skip_kv_fill_noalloc(new.h, n, hd, el, seq, pos)
        assert adept.adept_launch_count(new.h) >= 2     # the bucket sort (1 or 2) and at least one GEMM
        ref.check()
        new.check()
        want = O.skip_kv_fill(om, h.double().numpy(), el_h, pos_h)
        compared = 0
        for r in range(2, cfg.n_layers + 1):
            for b in range(cfg.max_batch):
                rows = np.nonzero((seq_h == b) & (el_h < r))[0]
                if len(rows) == 0:
                    continue
                kr, vr = ref.read_kv(r, b, 0, cfg.max_seq)
                kn, vn = new.read_kv(r, b, 0, cfg.max_seq)
                p = pos_h[rows]
                k_new, v_new = kn.float().cpu().numpy()[p], vn.float().cpu().numpy()[p]
                if n > 8:   # both on the grouped tensor-core GEMM: the same sums in the same order
                    assert np.array_equal(k_new, kr.float().cpu().numpy()[p]), f"call {call} K layer {r} differs"
                    assert np.array_equal(v_new, vr.float().cpu().numpy()[p]), f"call {call} V layer {r} differs"
                ko, vo, sel = want[r]
                at = np.searchsorted(sel, rows)
                assert_rows_close(k_new, ko[at], TOL["bf16"], f"call {call} K layer {r} vs oracle")
                assert_rows_close(v_new, vo[at], TOL["bf16"], f"call {call} V layer {r} vs oracle")
                compared += len(rows)
        assert compared >= n - int(np.sum(el_h == cfg.n_layers))
    ref.close()
    new.close()


def test_noalloc_fill_refuses_sizes_above_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2601_03700_gb300 as adept
    cfg = _cfg()
    m = adept.Model(cfg, synth.make_weights(cfg, seed=30))
    adept.adept_seq_reserve(m.h, [cfg.max_seq] * cfg.max_batch)
    too_many = int((16 << 20) // (cfg.d_model * 2 + 4)) + 64
    hb = torch.zeros(too_many, cfg.d_model, dtype=torch.bfloat16, device="cuda")
    z = torch.zeros(too_many, dtype=torch.int32, device="cuda")
    adept.adept_launch_count(m.h)
    with pytest.raises(adept.AdeptError) as ei:
        adept.adept_skip_kv_fill_noalloc(m.h, too_many, hb, z + 1, z, z)
    assert ei.value.status == 3 and "scratch" in str(ei.value)
    assert adept.adept_launch_count(m.h) == 0    # nothing enqueued
    m.check()
    m.close()
