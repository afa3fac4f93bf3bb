"""The whole stage through the public API: merged queries get exactly their
representative's results (the kept node's output flows to every merged node,
Section 3.3 (I)), and those results match the oracle."""
import numpy as np
import pytest

import oracle
import paper_2607_22578_gb300 as hs
from hs_testutil import check_rows, to_dev
from synth import configs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("cfg", [configs.TINY, configs.RAG_MIX])
def test_stage_matches_oracle(cfg):
    w = configs.build_retrieval_mix(cfg)
    stage = hs.EmbedRetrieveStage(to_dev(w["corpus"]), w["k"], max_queries=len(w["queries"]),
                                  max_chunk_rows=w["tokens"].shape[0])
    nu, uidx, inv, fp = stage.dedup_chunks(to_dev(w["tokens"]))
    hs.hs_get_device_error()
    ou, oi = oracle.unique_inverse(w["tokens"])
    n = int(nu.item())
    assert n == len(ou)
    assert (uidx[:n].cpu().numpy() == ou).all() and (inv.cpu().numpy() == oi).all()
    assert (fp.cpu().numpy().view(np.uint64) == oracle.fingerprint(w["tokens"])).all()

    Q = w["queries"]
    scores, ids, nu_dev = stage.retrieve(to_dev(Q))
    hs.hs_get_device_error()
    n_unique = int(nu_dev.item())
    quidx, qinv = oracle.unique_inverse(Q.view(np.int32))
    assert n_unique == len(quidx)
    s, i = scores.cpu().numpy(), ids.cpu().numpy()
    # Every query equals its representative's row of the result.
    rep = quidx[qinv]
    assert (s == s[rep]).all() and (i == i[rep]).all()
    # every merged query against the oracle (at the RAG mix: all 1434)
    check_rows(Q, w["corpus"], w["k"], s, i, quidx, tag="%s_corpus_seed0" % cfg["name"])


def test_step_runs_both_paths_and_matches_separate_calls():
    w = configs.build_retrieval_mix(configs.TINY)
    stage = hs.EmbedRetrieveStage(to_dev(w["corpus"]), w["k"], max_queries=len(w["queries"]),
                                  max_chunk_rows=w["tokens"].shape[0])
    t, q = to_dev(w["tokens"]), to_dev(w["queries"])
    (cnu, cuidx, cinv, cfp), (s, i, qnu) = stage.step(t, q)
    hs.hs_get_device_error()
    ou, oi = oracle.unique_inverse(w["tokens"])
    n = int(cnu.item())
    assert n == len(ou) and (cuidx[:n].cpu().numpy() == ou).all()
    assert (cinv.cpu().numpy() == oi).all()
    s2, i2, _ = stage.retrieve(q)
    hs.hs_get_device_error()
    assert (s.cpu() == s2.cpu()).all() and (i.cpu() == i2.cpu()).all()


def test_host_feed_matches_device_step():
    import torch
    w = configs.build_retrieval_mix(configs.TINY)
    stage = hs.EmbedRetrieveStage(to_dev(w["corpus"]), w["k"], max_queries=len(w["queries"]),
                                  max_chunk_rows=w["tokens"].shape[0])
    s_ref, i_ref, nu_ref = stage.retrieve(to_dev(w["queries"]))
    hs.hs_get_device_error()
    s_ref, i_ref, nu_ref = s_ref.cpu(), i_ref.cpu(), int(nu_ref.item())
    h_tok = torch.from_numpy(w["tokens"]).pin_memory()
    h_q = torch.from_numpy(w["queries"].view(np.int16)).pin_memory()
    feed = hs.HostFeed(stage, w["tokens"].shape[0], w["tokens"].shape[1], len(w["queries"]))
    prev = None
    for _ in range(5):                       # alternate both buffers twice over
        slot = feed.submit(h_tok, h_q)
        if prev is not None:
            s, i, nu = feed.fetch(prev)
            assert nu == nu_ref and torch.equal(s, s_ref) and torch.equal(i, i_ref)
        prev = slot
    s, i, nu = feed.fetch(prev)
    hs.hs_get_device_error()
    assert nu == nu_ref and torch.equal(s, s_ref) and torch.equal(i, i_ref)


def test_step_graph_replays_match_eager_step():
    import torch
    w = configs.build_retrieval_mix(configs.TINY)
    stage = hs.EmbedRetrieveStage(to_dev(w["corpus"]), w["k"], max_queries=len(w["queries"]),
                                  max_chunk_rows=w["tokens"].shape[0])
    t, q = to_dev(w["tokens"]), to_dev(w["queries"])
    (cnu, cu, ci, _), (s, i, nu) = stage.step(t, q)
    hs.hs_get_device_error()
    ref = [x.cpu().clone() for x in (cnu, cu, ci, s, i, nu)]
    g = hs.StepGraph(stage, t, q)
    assert g.launches > 0
    for _ in range(3):
        (cnu, cu, ci, _), (s, i, nu) = g.replay()
        hs.hs_get_device_error()
        n = int(cnu.item())
        got = [x.cpu() for x in (cnu, cu, ci, s, i, nu)]
        assert torch.equal(got[0], ref[0]) and torch.equal(got[1][:n], ref[1][:n])
        assert all(torch.equal(a, b) for a, b in zip(got[2:], ref[2:]))
    # new contents in the captured buffers are picked up by the next replay
    q2 = to_dev(w["queries"][::-1].copy())
    q.copy_(q2)
    _, (s2, i2, _) = g.replay()
    s2, i2 = s2.cpu(), i2.cpu()          # host copies: retrieve() reuses the buffers
    s3, i3, _ = stage.retrieve(q2)
    hs.hs_get_device_error()
    assert torch.equal(s2, s3.cpu()) and torch.equal(i2, i3.cpu())
    assert not torch.equal(s2, ref[3])   # the reversed batch has different results


def test_retrieve_graph_matches_eager_retrieve():
    import torch
    w = configs.build_retrieval_mix(configs.TINY)
    stage = hs.EmbedRetrieveStage(to_dev(w["corpus"]), w["k"], max_queries=len(w["queries"]))
    g = hs.RetrieveGraph(stage, len(w["queries"]))
    for qs in (w["queries"], w["queries"][::-1].copy()):
        qd = to_dev(qs)
        s, i, nu = g.run(qd)
        s, i, nu = s.cpu(), i.cpu(), int(nu.item())
        s2, i2, nu2 = stage.retrieve(qd)
        hs.hs_get_device_error()
        assert nu == int(nu2.item()) and torch.equal(s, s2.cpu()) and torch.equal(i, i2.cpu())
