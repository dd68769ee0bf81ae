"""GPU: a chain of calls enqueued back to back on one stream, each reading what
the kernels of the call before it wrote, with no host wait anywhere in the
chain.

The library launches its kernels so that one may be scheduled while the
kernel ahead of it on the stream drains, and lets a kernel read its own
host-written descriptors before it waits for that kernel.  Every read of
data a kernel wrote must still come after that kernel: the checkpoint of
buffers a restore has just written, the fork of records a checkpoint has just
finalised, a prune whose queries a restore has just written, and the pack of
bank rows gathered by the indices the top-k has just chosen.  The results are
compared with the sources and with the oracle once the chain has finished."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_21686_gb300 import pcs
from helpers import np_view

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("it", range(3))
def test_dependent_calls_on_one_stream(ctx, dev, it):
    S, D = 8, 128  # 8 observations of 196,608 B: the TMA kernels
    n = [300, 1, 77, 512, 130]
    g = torch.Generator(device=dev).manual_seed(1000 + it)
    obs = torch.randint(0, 256, (S, 3, 256, 256), generator=g, device=dev, dtype=torch.uint8)
    rng = torch.randint(-2**62, 2**62, (S, 2), generator=g, device=dev, dtype=torch.int64)
    keys = [torch.randn(x, D, generator=g, device=dev).half() for x in n]
    vals = [torch.randint(0, 256, (x, 2048), generator=g, device=dev, dtype=torch.uint8) for x in n]
    q_true = torch.randn(len(n), D, generator=g, device=dev).half()
    q_buf = torch.zeros_like(q_true)
    # The queries' record, written before the chain starts.
    qsec = lambda t: [pcs.contig_section(pcs.PCS_SEC_OBS, t.view(torch.uint8).reshape(-1))]
    qsnap = ctx.checkpoint([pcs.Session(90, pcs.PCS_KIND_BANK, qsec(q_true), keep=[q_true])])[0]
    ctx.sync()
    torch.cuda.synchronize()

    obs_b, rng_b = torch.zeros_like(obs), torch.zeros_like(rng)
    obs_c, rng_c = torch.zeros_like(obs), torch.zeros_like(rng)
    A = [pcs.markov_session(s, obs[s], rng[s]) for s in range(S)]
    B = [pcs.markov_session(s, obs_b[s], rng_b[s]) for s in range(S)]
    C = [pcs.markov_session(s, obs_c[s], rng_c[s]) for s in range(S)]
    banks = ctx.banks_array(keys, [q_buf[i] for i in range(len(n))], 2 * D + 2048)
    params = ctx.params(pcs.PCS_K_FIXED, k_max=64)
    ks = ctx.prune_counts(banks, len(n), params)  # host arithmetic only
    koff = np.concatenate([[0], np.cumsum(ks)]).astype(np.int64)
    kept = torch.full((int(koff[-1]),), -1, dtype=torch.int32, device=dev)
    scores = torch.zeros(sum(n), dtype=torch.float32, device=dev)
    bank_sess = [pcs.bank_session(i, keys[i], vals[i], kept[koff[i]:koff[i + 1]])
                 for i in range(len(n))]

    # --- the chain: nothing below waits on the host until ctx.sync() ---
    snaps_a = ctx.checkpoint(A)
    ctx.restore(snaps_a, B, verify=2)                 # writes obs_b, rng_b
    snaps_b = ctx.checkpoint(B)                       # reads them
    kids = [ctx.fork(x) for x in snaps_b]             # copies the records just finalised
    ctx.restore(kids, C, verify=2)                    # writes obs_c, rng_c
    ctx.restore([qsnap], [pcs.Session(90, pcs.PCS_KIND_BANK, qsec(q_buf), keep=[q_buf])],
                verify=2)                             # writes the queries
    ctx.prune(banks, len(n), params, kept, None, scores)  # reads them; writes kept
    snaps_k = ctx.checkpoint(bank_sess)               # gathers rows by kept
    ctx.sync()
    torch.cuda.synchronize()

    assert torch.equal(obs_c, obs) and torch.equal(rng_c, rng)
    for s in range(S):
        ra = ctx.record(snaps_a[s]).numpy()
        assert np.array_equal(ctx.record(snaps_b[s]).numpy(), ra), s
        assert np.array_equal(ctx.record(kids[s]).numpy(), ra), s
    sc_h, kept_h = scores.cpu().numpy(), kept.cpu().numpy()
    eo = 0
    for i, x in enumerate(n):
        s32 = oracle.scores(np_view(q_true[i].cpu()), np_view(keys[i].cpu()))
        assert np.array_equal(sc_h[eo:eo + x].view(np.uint32), s32.view(np.uint32)), i
        want = oracle.topk(s32, ks[i])
        assert kept_h[koff[i]:koff[i + 1]].tolist() == want.tolist(), i
        ref = oracle.pack(oracle.bank_session(i, np_view(keys[i].cpu()), np_view(vals[i].cpu()),
                                              want, oracle.DT_F16, oracle.DT_U8))
        assert np.array_equal(ctx.record(snaps_k[i]).numpy(), ref), i
        eo += x
    for x in snaps_a + snaps_b + kids + snaps_k + [qsnap]:
        ctx.delete(x)
