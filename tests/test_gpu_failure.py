"""Failure detection without a GPU fault.

* Bounded device waits: adept_set_wait_limit shortens the kernels' waits on pipeline progress
  to a few cycles, so the waits of a bf16 prompt pass (tensor-core GEMMs) and of generation
  steps at a shape that takes the stream-K weight-streaming GEMM run out.  The call must then
  report ADEPT_ERR_TIMEOUT through adept_check_device_status, the context must stay usable,
  and with the limit restored the same model and a fresh one must match the oracle.
* Device allocation failure: adept_set_alloc_fail_after makes the library's device
  allocations fail from a chosen point on; model loading and the fill workspace's growth must
  return ADEPT_ERR_OOM, release what they allocated, and leave the library usable."""
import numpy as np
import pytest
import torch

import synth
from parity_utils import Pair, compare_decode, compare_prefill

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu

TIMEOUT, OOM = 5, 2


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()
    yield
    adept.adept_set_wait_limit(0)
    adept.adept_set_alloc_fail_after(-1)


def _small():
    return synth.ModelConfig(family=synth.LLAMA, n_layers=4, d_model=256, n_heads=2, head_dim=128, d_ffn=512,
                             vocab=1000, dtype="bf16", max_batch=2, max_seq=64, hsm_m1=512, hsm_m2=1024,
                             block_shuffle_seed=4)


def _expect_timeout(m):
    with pytest.raises(adept.AdeptError) as ei:
        m.check()
    assert ei.value.status == TIMEOUT, str(ei.value)


def test_short_wait_limit_times_out_prompt_pass_and_recovers():
    cfg = _small()
    pair = Pair(cfg, seed=50)
    tokens = synth.make_tokens(50, 2, 40, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(50, 80, 2, cfg.n_layers).numpy().reshape(2, 40)
    adept.adept_set_wait_limit(32)
    try:
        pair.gm.prefill(torch.as_tensor(tokens).cuda(), 0.9, torch.as_tensor(forced).cuda())
        _expect_timeout(pair.gm)
    finally:
        adept.adept_set_wait_limit(0)
    pair.gm.check()   # the error word was cleared; nothing else pending
    ores, cache, _ = compare_prefill(pair, tokens, 0.9, forced)
    compare_decode(pair, cache, ores.next_token, 2, 0.9, np.full((2, 2), 3))
    fresh = Pair(cfg, weights=pair.W)
    compare_prefill(fresh, tokens, 0.9, forced)
    fresh.close()
    pair.close()


def test_short_wait_limit_times_out_stream_k_generation_step_and_recovers():
    # the wide GEMMs of a generation step (QKV, gate/up, mapper FC2, head, fills) take the
    # stream-K kernel here
    cfg = synth.ModelConfig(family=synth.LLAMA, n_layers=4, d_model=2048, n_heads=24, head_dim=128, d_ffn=5504,
                            vocab=9000, dtype="bf16", hsm_m1=4096, hsm_m2=16384, max_batch=1, max_seq=32,
                            max_pass_tokens=32)
    W = synth.make_weights(cfg, seed=51, device="cuda")
    pair = Pair(cfg, weights=W)
    tokens = synth.make_tokens(51, 1, 24, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(51, 24, 2, cfg.n_layers).numpy().reshape(1, 24)
    ores, cache, _ = compare_prefill(pair, tokens, 0.9, forced)
    step_tok = torch.as_tensor(ores.next_token, dtype=torch.int32).cuda()
    adept.adept_set_wait_limit(32)
    try:
        for _ in range(2):
            pair.gm.decode_step(step_tok, 0.9, torch.full((1,), 3, dtype=torch.int32, device="cuda"))
            _expect_timeout(pair.gm)
    finally:
        adept.adept_set_wait_limit(0)
    # the stream-K arrival counters were reset with the error word: fresh prompt pass and
    # generation steps on the same model match the oracle again
    ores, cache, _ = compare_prefill(pair, tokens, 0.9, forced)
    compare_decode(pair, cache, ores.next_token, 3, 0.9, np.array([[3], [2], [4]]))
    pair.close()


def test_wait_limit_rejects_negative_values():
    with pytest.raises(adept.AdeptError) as ei:
        adept.adept_set_wait_limit(-1)
    assert ei.value.status == 1


def test_allocation_failure_returns_oom_and_releases_memory():
    cfg = _small()
    W = synth.make_weights(cfg, seed=52)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    try:
        for n in (0, 1, 7, 30):   # the n+1-th device allocation of the load fails
            adept.adept_set_alloc_fail_after(n)
            with pytest.raises(adept.AdeptError) as ei:
                adept.Model(cfg, W)
            assert ei.value.status == OOM and "allocation-failure hook" in str(ei.value)
        adept.adept_set_alloc_fail_after(-1)
        m = adept.Model(cfg, W)
        adept.adept_seq_reserve(m.h, [cfg.max_seq] * cfg.max_batch)
        n = 40
        h = synth.make_mapped_states(53, n, cfg.d_model).cuda()
        z = torch.zeros(n, dtype=torch.int32, device="cuda")
        pos = torch.arange(n, dtype=torch.int32, device="cuda") // 2
        seq = torch.arange(n, dtype=torch.int32, device="cuda") % 2
        adept.adept_set_alloc_fail_after(0)    # the fill workspace cannot grow
        with pytest.raises(adept.AdeptError) as ei:
            adept.adept_skip_kv_fill(m.h, n, h, z + 1, seq, pos)
        assert ei.value.status == OOM
        adept.adept_set_alloc_fail_after(-1)
        adept.adept_skip_kv_fill(m.h, n, h, z + 1, seq, pos)   # grows now, and runs
        m.check()
        m.close()
    finally:
        adept.adept_set_alloc_fail_after(-1)
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info()[0]
    assert abs(free1 - free0) < (64 << 20), f"device memory not released: {(free0 - free1) / 2**20:.1f} MiB"
