"""The allocation-free QKV entry point, for callers that cannot give the library
device memory (a plugin whose host process owns the memory pool, a loop that must
not enter an allocator).  Its scratch is a fixed array inside the library; these
checks compare it with the workspace-based entry point on the same inputs, over
two calls in a row (the second reuses what the first left in the array), and check
that sizes beyond the array are refused.  Both entry points launch the same kernels on
the same inputs, so their outputs - including the cache rows no call writes - must agree
bit for bit.  Collected last on purpose."""
import pytest
import torch

from paper_2609_09768_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def kvb():
    from paper_2609_09768_gb300 import kvblend
    kvblend.lib()
    return kvblend


def _run_pair(kvb, shape, m, n_src, seed):
    cfg = kvb.config(shape)
    lw = {k: v.cuda() for k, v in synth.make_layer_weights(shape, 1, seed=seed).items()}
    lws = kvb.layer_struct(lw)
    g = torch.Generator().manual_seed(seed)
    x = (torch.randn(n_src, shape.hidden, generator=g) * 2.0).cuda()
    row_idx = torch.sort(torch.randperm(n_src, generator=g)[:m]).values.to(torch.int32).cuda()
    rope_pos = torch.randint(0, n_src + 7, (m,), generator=g, dtype=torch.int32).cuda()
    kv_dst = torch.randperm(n_src + 3, generator=g)[:m].to(torch.int32).cuda()
    rope = kvb.RopeTable(cfg, n_src + 7)
    outs = []
    for noalloc in (False, True):
        q = torch.zeros(m, shape.q_dim, dtype=torch.bfloat16, device="cuda")
        kc = torch.zeros(n_src + 3, shape.kv_dim, dtype=torch.bfloat16, device="cuda")
        vc = torch.zeros(n_src + 3, shape.kv_dim, dtype=torch.float16, device="cuda")
        if noalloc:
            status = torch.zeros(4, dtype=torch.int32, device="cuda")
            kvb.gather_rmsnorm_qkv_noalloc(cfg, lws, rope, x, row_idx, rope_pos, m, q, kc, vc, kv_dst, status)
            torch.cuda.synchronize()
            assert int(status[0]) == 0
        else:
            ws = kvb.workspace(cfg, m)
            kvb.gather_rmsnorm_qkv(cfg, lws, rope, x, row_idx, rope_pos, m, q, kc, vc, kv_dst, ws)
            torch.cuda.synchronize()
        outs.append((q, kc, vc))
    return outs


@pytest.mark.parametrize("shape,m,n_src", [(synth.LLAMA8B.with_layers(2), 1024, 3904), (synth.TINY, 300, 544),
                                           (synth.YARN_GQA7, 700, 3904)])
def test_noalloc_matches_workspace_entry_point_on_two_calls(kvb, shape, m, n_src):
    for seed, mm in ((21, m), (22, m // 3 + 1)):       # two calls in a row, the second smaller
        (q, kc, vc), (q2, kc2, vc2) = _run_pair(kvb, shape, mm, n_src, seed)
        assert torch.equal(q2, q), "q (no-alloc vs workspace)"
        assert torch.equal(kc2, kc), "k cache rows (no-alloc vs workspace)"
        assert torch.equal(vc2, vc), "v cache rows (no-alloc vs workspace)"


def test_noalloc_rejects_sizes_beyond_its_scratch(kvb):
    shape = synth.LLAMA8B.with_layers(2)
    cfg = kvb.config(shape)
    lws = kvb.layer_struct({k: v.cuda() for k, v in synth.make_layer_weights(shape, 1, seed=1).items()})
    m = kvb.NOALLOC_MAX_ELEMS // shape.hidden + 1
    x = torch.zeros(m, shape.hidden, device="cuda")
    pos = torch.zeros(m, dtype=torch.int32, device="cuda")
    q = torch.zeros(m, shape.q_dim, dtype=torch.bfloat16, device="cuda")
    kc = torch.zeros(m, shape.kv_dim, dtype=torch.bfloat16, device="cuda")
    vc = torch.zeros(m, shape.kv_dim, dtype=torch.float16, device="cuda")
    rope = kvb.RopeTable(cfg, 8)
    with pytest.raises(kvb.KvbError, match="exceeds the fixed scratch"):
        kvb.gather_rmsnorm_qkv_noalloc(cfg, lws, rope, x, None, pos, m, q, kc, vc, None)
