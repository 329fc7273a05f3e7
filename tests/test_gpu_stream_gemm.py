"""The stream-K weight-streaming GEMM (generation steps and small fills) against the oracle.

The model is sized so that the wide GEMMs of a generation step (at least 8 MB of weights and
8192 outputs) take the stream-K kernel: a Llama-family decoder with D = 2048, 24 heads x 128
(QKV 9216 outputs), SwiGLU 5504 (gate/up 11008 outputs; K = 5504 of the down projection ends in
a half k-block), the 36 D^2 mapper (FC2 has 16384 outputs), a 9000-token vocabulary (the head's
last 32-feature tile is ragged) and the grouped fills (6144 outputs per layer); the narrower
products take the cluster K-split kernel.  Batches of 1, 5 and 12 sequences cover one and two 8-token
blocks of the A operand.  Generation steps (forced exits through every layer, the mapper,
the grouped skipped-layer fill and the head) are compared with the oracle, with the cluster
K-split kernel, and with themselves run again (the split tiles are summed in a fixed order, so
the results are bit-identical); skipped-layer fills of 1 to 16 tokens through
adept_skip_kv_fill are compared entry by entry with the oracle."""
import numpy as np
import pytest
import torch

import synth
from oracle import adept_oracle as O
from parity_utils import TOL, Pair, assert_rows_close, compare_decode, compare_prefill, row_rel_err

import paper_2601_03700_gb300 as adept

pytestmark = pytest.mark.gpu


def _cfg(B):
    return synth.ModelConfig(family=synth.LLAMA, n_layers=4, d_model=2048, n_heads=24, head_dim=128, d_ffn=5504,
                             vocab=9000, dtype="bf16", hsm_m1=4096, hsm_m2=16384, max_batch=B, max_seq=48,
                             max_pass_tokens=B * 40, block_shuffle_seed=9)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    adept.load_library()


@pytest.mark.parametrize("B", [1, 5, 12])
def test_stream_gemm_generation_steps_match_oracle(B):
    cfg = _cfg(B)
    W = synth.make_weights(cfg, seed=40, device="cuda")
    pair = Pair(cfg, weights=W)
    P = 40
    tokens = synth.make_tokens(40, B, P, cfg.vocab).numpy()
    forced = synth.forced_exits_uniform(40, B * P, 2, cfg.n_layers).numpy().reshape(B, P)
    ores, cache, _ = compare_prefill(pair, tokens, 0.9, forced)
    fd = synth.forced_exits_uniform(41, 4 * B, 2, cfg.n_layers, name="forced_decode").numpy().reshape(4, B)
    compare_decode(pair, cache, ores.next_token, 4, 0.9, fd)
    pair.compare_cache(cache, B, P + 4)
    pair.close()


def _steps(cfg, W, stream, repeat=1, tiled=1):
    B, P = cfg.max_batch, 40
    out = []
    for _ in range(repeat):
        m = adept.Model(cfg, W)
        adept.adept_set_option(m.h, adept.OPT_DECODE_STREAM, stream)
        adept.adept_set_option(m.h, adept.OPT_DECODE_TILED, tiled)
        tokens = synth.make_tokens(42, B, P, cfg.vocab).cuda()
        forced = synth.forced_exits_uniform(42, B * P, 2, cfg.n_layers).view(B, P).cuda()
        m.prefill(tokens, 0.9, forced)
        fs = synth.forced_exits_uniform(43, 4 * B, 2, cfg.n_layers).view(4, B).cuda()
        ts = synth.make_tokens(44, 4, B, cfg.vocab).cuda()
        steps = []
        for s in range(4):
            ex, lg, nx, _ = m.decode_step(ts[s].contiguous(), 0.9, fs[s])
            steps.append((ex.cpu().numpy(), lg.cpu().numpy(), m.final_states(B).cpu().numpy()))
        m.check()
        kv = [m.read_kv(r, B - 1, 0, P + 4)[0].float().cpu().numpy() for r in range(1, cfg.n_layers + 1)]
        out.append((steps, kv))
        m.close()
    return out


@pytest.mark.parametrize("B", [1, 12])
def test_stream_gemm_matches_cluster_kernel_and_repeats_bit_for_bit(B):
    cfg = _cfg(B)
    W = synth.make_weights(cfg, seed=45, device="cuda")
    new = _steps(cfg, W, 1, repeat=2)
    old = _steps(cfg, W, 0)[0]
    for a, b in zip(new[0][0], new[1][0]):        # the same sums in the same order
        for x, y in zip(a, b):
            assert np.array_equal(x, y)
    for x, y in zip(new[0][1], new[1][1]):
        assert np.array_equal(x, y)
    for a, b in zip(new[0][0], old[0]):
        np.testing.assert_array_equal(a[0], b[0])
        assert row_rel_err(a[1], b[1]).max() < 2e-2
        assert row_rel_err(a[2], b[2]).max() < 2e-2
    for x, y in zip(new[0][1], old[1]):
        assert row_rel_err(x.reshape(len(x), -1), y.reshape(len(y), -1)).max() < 2e-2


@pytest.mark.parametrize("B", [1, 5])
def test_tile_contiguous_weights_give_identical_results(B):
    """The weight-streaming kernels reading the tile-contiguous weight copies by bulk copy equal
    the same kernels reading the row-major weights through tensor maps bit for bit (the same
    bytes reach the same shared-memory layout), for both the stream-K and the cluster kernel."""
    cfg = _cfg(B)
    W = synth.make_weights(cfg, seed=49, device="cuda")
    for stream in (1, 0):
        a = _steps(cfg, W, stream, tiled=1)[0]
        b = _steps(cfg, W, stream, tiled=0)[0]
        for x, y in zip(a[0], b[0]):
            for u, v in zip(x, y):
                assert np.array_equal(u, v), f"stream={stream}"
        for u, v in zip(a[1], b[1]):
            assert np.array_equal(u, v), f"stream={stream}"


def test_stream_gemm_small_fills_match_oracle():
    """adept_skip_kv_fill of 1, 3, 8, 9 and 16 tokens (the grouped stream-K launch over the
    layers that have rows; 9-16 tokens use two 8-token blocks) against the oracle."""
    cfg = _cfg(4)
    W = synth.make_weights(cfg, seed=46, device="cuda")
    pair = Pair(cfg, weights=W)
    adept.adept_seq_reserve(pair.gm.h, [cfg.max_seq] * cfg.max_batch)
    for n in (1, 3, 8, 9, 16):
        h = synth.make_mapped_states(47 + n, n, cfg.d_model)
        el = synth.forced_exits_uniform(48 + n, n, 1, cfg.n_layers, name="el").numpy()
        seq = np.arange(n) % cfg.max_batch
        pos = np.arange(n) // cfg.max_batch + n
        dev = lambda x: torch.as_tensor(x, dtype=torch.int32).cuda().contiguous()  # noqa: E731
        adept.adept_skip_kv_fill(pair.gm.h, n, h.cuda(), dev(el), dev(seq), dev(pos))
        pair.gm.check()
        checked = 0
        for r, (k, v, sel) in O.skip_kv_fill(pair.om, h.double().numpy(), el, pos).items():
            for b in range(cfg.max_batch):
                rows = sel[seq[sel] == b]
                if len(rows) == 0:
                    continue
                gk, gv = pair.gpu_kv(r, b, cfg.max_seq)
                at = np.searchsorted(sel, rows)
                assert_rows_close(gk[pos[rows]], k[at], TOL["bf16"], f"n={n} K r={r}")
                assert_rows_close(gv[pos[rows]], v[at], TOL["bf16"], f"n={n} V r={r}")
                checked += len(rows)
        assert checked >= n - int(np.sum(el == cfg.n_layers))
    pair.close()


def test_span_timer_sums_within_the_step_and_changes_nothing():
    """With the span timer on, the weight-streaming launches of generation steps record their
    in-situ spans: every step records the same launches, the summed spans stay within the steps'
    elapsed time, and the results equal those of the same steps without the timer bit for bit."""
    cfg = _cfg(2)
    W = synth.make_weights(cfg, seed=50, device="cuda")
    B, P = cfg.max_batch, 40
    res = []
    for timer in (0, 1):
        m = adept.Model(cfg, W)
        adept.adept_set_option(m.h, adept.OPT_SPAN_TIMER, timer)
        tokens = synth.make_tokens(50, B, P, cfg.vocab).cuda()
        forced = synth.forced_exits_uniform(50, B * P, 2, cfg.n_layers).view(B, P).cuda()
        m.prefill(tokens, 0.9, forced)
        adept.adept_span_read(m.h, adept.PROF_GEMM_DECODE)
        adept.adept_span_read(m.h, adept.PROF_KV_FILL)
        ts = synth.make_tokens(51, 5, B, cfg.vocab).cuda()
        fs = torch.full((B,), 3, dtype=torch.int32, device="cuda")
        out, counts = [], []
        for s in range(5):   # direct launches first, then graph replays
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            ex, lg, nx, _ = m.decode_step(ts[s].contiguous(), 0.9, fs)
            e1.record()
            torch.cuda.synchronize()
            n_g, ms_g = adept.adept_span_read(m.h, adept.PROF_GEMM_DECODE)
            n_f, ms_f = adept.adept_span_read(m.h, adept.PROF_KV_FILL)
            counts.append((n_g, n_f))
            if timer:
                assert n_g > 0 and n_f == 1
                assert 0 < ms_g + ms_f <= e0.elapsed_time(e1), (ms_g, ms_f, e0.elapsed_time(e1))
            else:
                assert n_g == 0 and n_f == 0
            out.append((ex.cpu().numpy(), lg.cpu().numpy(), m.final_states(B).cpu().numpy()))
        m.check()
        assert len(set(counts)) == 1, counts
        res.append(out)
        m.close()
    for a, b in zip(res[0], res[1]):
        for x, y in zip(a, b):
            assert np.array_equal(x, y)
