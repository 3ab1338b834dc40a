"""End-to-end parity of apack_prune_step on the five audio-video workloads
(full sizes, the launch configuration the benchmark times), step by step
through progressive schedules.

Each step is checked against the oracle on the GPU's own previous-step
result, so that a legitimate near-tie reordering in one step does not
cascade: every score of S within 2e-3|ref| (the strict relative rule, which
at 10^5 tokens is the only one with content) and within 1e-5 + 2e-3|ref|;
kept indices identical up to tokens within 2e|I_k| of the k-th score, e the
largest relative score error measured at that step; compacted K/V/hidden rows
bit-exact given the GPU's indices (sampled layers), modality and offsets
exact, planted tokens kept.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import check_scores, check_keep, tie_bands

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ap():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_08794_gb300 as ap
    return ap


def host_u16(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def oracle_counts(wl):
    """The oracle's keep counts per step and the joint flag."""
    from synth.inputs import base_counts
    if wl.joint_step_keep is None:
        return [oracle.step_keep_counts(r, base_counts(wl)) for r in wl.ratios], False
    n = [a + v for a, v in base_counts(wl)]
    out = []
    for _ in wl.prune_layers:
        k = [oracle.keep_count(wl.joint_step_keep, x) for x in n]
        out.append([(x, 0) for x in k])
        n = k
    return out, True


@pytest.mark.parametrize("name,domain", [(n, 0) for n in ["tiny", "3b_60s", "7b_2min", "7b_10min", "7b_ragged16",
                                                          "7b_10min_paper"]] +
                         [(n, 1) for n in ["tiny", "3b_60s", "7b_2min", "7b_10min_paper"]])
def test_workload_parity(ap, name, domain):
    """domain 1: the causal-row softmax domain (the text-query rows are the last n_q
    tokens of every synthetic sequence)."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs
    from synth.inputs import key_slab, planted_tokens

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod0 = wl.modality()
    mod_d = torch.from_numpy(mod0).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    ref_counts, joint = oracle_counts(wl)
    assert [c.tolist() for c in counts] == [[list(x) for x in r] for r in ref_counts]
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode, softmax_domain=domain)
    qs = fill_progressive_inputs(pp, wl)

    composite = np.arange(wl.total_tokens)
    mod_cur, cu_cur = mod0, cu0
    l0 = wl.prune_layers[0]
    exempt_total = band_graded = band_strict = 0
    worst_rel = 0.0
    for i, layer in enumerate(wl.prune_layers):
        seqs, k_in, v_in, in_stride, h_in = pp.step_args(i)
        new_cu = pp.run_step(i)
        torch.cuda.synchronize()
        assert ap.apack_device_error(pp.ws) == ap.APACK_OK
        T_in, t_out = int(cu_cur[-1]), pp.t_out[i]
        # scores
        k_host = key_slab(wl, layer, qs[i])[composite]
        ref_scores = oracle.relevance_scores(qs[i], k_host, cu_cur, cuq, mod_cur, wl.num_q_heads, wl.num_kv_heads,
                                             softmax_domain=domain)
        got = pp.scores[:T_in].cpu().numpy()
        max_rel = check_scores(got, ref_scores)
        # selection: a token may be kept by one side only if the measured score error explains it
        ref_keep = oracle.select_keep(ref_scores, mod_cur, cu_cur, [tuple(c) for c in counts[i]], joint=joint)
        keep = pp.keep_idx[i][:t_out].cpu().numpy().astype(np.int64)
        exempt_total += check_keep(keep, ref_keep, ref_scores, mod_cur, cu_cur, joint=joint,
                                   rel_band=2.01 * max_rel + 1e-12)
        g_band, s_band = tie_bands(ref_scores, ref_keep, mod_cur, cu_cur, joint=joint)
        band_graded += g_band
        band_strict += s_band
        worst_rel = max(worst_rel, max_rel)
        # the GPU's own selection is exact on its own fp32 scores
        np.testing.assert_array_equal(keep, oracle.select_keep(got, mod_cur, cu_cur, [tuple(c) for c in counts[i]],
                                                               joint=joint))
        np.testing.assert_array_equal(new_cu, oracle.new_cu_seqlens(keep, cu_cur))
        np.testing.assert_array_equal(pp.mod_out[i % 2][:t_out].cpu().numpy(), mod_cur[keep])
        # compaction, bit-exact given the GPU's indices, on sampled layers
        k_out, v_out = pp.output_kv(i)
        n_l = wl.num_layers - layer
        row_elems = wl.num_kv_heads * wl.head_dim
        keep_t = torch.from_numpy(keep).cuda()
        for j in sorted({0, n_l // 2, n_l - 1}):
            src_k = k_in[j * T_in * row_elems:(j + 1) * T_in * row_elems].view(T_in, row_elems)
            src_v = v_in[j * T_in * row_elems:(j + 1) * T_in * row_elems].view(T_in, row_elems)
            assert torch.equal(k_out[j].reshape(t_out, row_elems).view(torch.int16),
                               src_k.index_select(0, keep_t).view(torch.int16))
            assert torch.equal(v_out[j].reshape(t_out, row_elems).view(torch.int16),
                               src_v.index_select(0, keep_t).view(torch.int16))
        if i == 0:
            # slab 0 of the first input is the planted key cache the host generator defines
            np.testing.assert_array_equal(host_u16(k_out[0]).reshape(t_out, -1), k_host.reshape(T_in, -1)[keep])
        h_out = pp.output_hidden(i)
        assert torch.equal(h_out.view(torch.int16), h_in[:T_in].index_select(0, keep_t).view(torch.int16))
        composite = composite[keep]
        mod_cur = mod_cur[keep]
        cu_cur = new_cu
    tok, _ = planted_tokens(wl)
    assert np.isin(tok, composite).all(), "a planted token was dropped"
    # the graded rule would exempt band_graded tokens, the strict one band_strict; kept by one side: exempt_total
    print(f"{name} (softmax domain {domain}): max rel score error {worst_rel:.2e}; tokens kept by one side only "
          f"{exempt_total}; tie bands graded {band_graded}, strict {band_strict}")


def snapshot(pp):
    """Every output the schedule leaves behind: per-step indices and offsets, the
    last two steps' K/V (both ping-pong buffers), hidden states and modality."""
    n = len(pp.layers)
    out = {"keep": [pp.keep_idx[i][:pp.t_out[i]].clone() for i in range(n)],
           "cu": [np.asarray(c).copy() for c in pp.new_cu]}
    for i in range(max(0, n - 2), n):
        k, v = pp.output_kv(i)
        out[f"k{i}"], out[f"v{i}"] = k.clone(), v.clone()
        out[f"h{i}"] = pp.output_hidden(i).clone()
        out[f"m{i}"] = pp.mod_out[i % 2][:pp.t_out[i]].clone()
    return out


def same(a, b):
    assert a.keys() == b.keys()
    for key in a:
        if key == "cu":
            for x, y in zip(a[key], b[key]):
                np.testing.assert_array_equal(x, y)
        elif key == "keep":
            for x, y in zip(a[key], b[key]):
                assert torch.equal(x, y)
        else:
            assert torch.equal(a[key].view(torch.int8) if a[key].dtype != torch.uint8 else a[key],
                               b[key].view(torch.int8) if b[key].dtype != torch.uint8 else b[key]), key


@pytest.mark.parametrize("name", ["3b_60s", "7b_2min", "7b_10min", "7b_ragged16", "7b_10min_paper"])
def test_schedule_runner_is_bit_identical_to_single_steps(ap, name):
    """apack_prune_schedule leaves exactly the outputs of one apack_prune_step per step."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    pp.run_steps()
    torch.cuda.synchronize()
    ref = snapshot(pp)
    pp.run()
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    same(ref, snapshot(pp))


@pytest.mark.parametrize("name", ["7b_2min", "7b_ragged16", "7b_10min_paper"])
def test_schedule_graph_replay_is_bit_identical(ap, name):
    """apack_prune_schedule_graph captures the schedule once; every replay leaves
    exactly the outputs of apack_prune_schedule (also after the outputs were
    wiped), and counts the captured kernels as launched per replay only."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    c0 = ap.apack_launch_count()
    pp.run()
    torch.cuda.synchronize()
    per_run = ap.apack_launch_count() - c0
    ref = snapshot(pp)
    c1 = ap.apack_launch_count()
    graph = pp.capture()
    assert ap.apack_launch_count() == c1          # capturing runs nothing
    for buf in pp.k_out + pp.v_out + pp.h_out + pp.mod_out + pp.keep_idx:
        if buf is not None:
            buf.zero_()
    for _ in range(2):
        graph.launch()
    torch.cuda.synchronize()
    assert ap.apack_launch_count() - c1 == 2 * per_run
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    same(ref, snapshot(pp))
    graph.close()


@pytest.mark.parametrize("name", ["7b_2min", "7b_ragged16", "7b_10min_paper"])
def test_in_place_schedule_equals_ping_pong(ap, name):
    """ProgressivePrune(in_place=True): every step compacts within k_in / v_in / hidden_in
    (apack_compact in place); the last step's caches, hidden states, modality, offsets and
    every step's kept indices equal those of the ping-pong schedule, through the schedule
    call, per-step calls and a captured graph."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)

    def make(in_place):
        pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                              wl.prune_layers, counts, select_mode=mode, in_place=in_place)
        fill_progressive_inputs(pp, wl)
        return pp

    def result(pp):
        n = len(pp.layers)
        k, v = pp.output_kv(n - 1)
        return ([pp.keep_idx[i][:pp.t_out[i]].clone() for i in range(n)], [np.asarray(c).copy() for c in pp.new_cu],
                k.contiguous().view(torch.int16).clone(), v.contiguous().view(torch.int16).clone(),
                pp.output_hidden(n - 1).view(torch.int16).clone(), pp.mod_out[(n - 1) % 2][:pp.t_out[-1]].clone())

    def check(a, b):
        for x, y in zip(a[0], b[0]):
            assert torch.equal(x, y)
        for x, y in zip(a[1], b[1]):
            np.testing.assert_array_equal(x, y)
        for x, y in zip(a[2:], b[2:]):
            assert torch.equal(x, y)

    ref_pp = make(False)
    ref_pp.run()
    torch.cuda.synchronize()
    ref = result(ref_pp)
    del ref_pp
    pp = make(True)
    pp.run()
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    check(ref, result(pp))
    pp = make(True)
    pp.run_steps()
    torch.cuda.synchronize()
    check(ref, result(pp))
    pp = make(True)
    graph = pp.capture()
    graph.launch()
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    check(ref, result(pp))
    graph.close()


@pytest.mark.parametrize("name", ["7b_2min", "7b_ragged16"])
def test_first_step_from_host_caches_is_bit_identical(ap, name):
    """Step 0 with the K/V caches and hidden states in pinned host memory (only the scored
    layer's keys on the device; the compaction reads the kept rows over the host link),
    then the remaining steps on the device: the same outputs as the all-device schedule."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    pp.run()
    torch.cuda.synchronize()
    ref = snapshot(pp)
    h_k = pp.k_in.cpu().pin_memory()
    h_v = pp.v_in.cpu().pin_memory()
    h_h = pp.hidden_in.cpu().pin_memory()
    for buf in pp.k_out + pp.v_out + pp.h_out + pp.mod_out + pp.keep_idx:
        buf.zero_()
    pp.k_in[1:].zero_()                          # only the scored layer's keys stay on the device
    pp.v_in.zero_()
    pp.hidden_in.zero_()
    pp.run_first_step_from_host(h_k, h_v, h_h)
    for i in range(1, len(pp.layers)):
        pp.run_step(i)
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    same(ref, snapshot(pp))


@pytest.mark.parametrize("name,streams", [("3b_60s", 1), ("7b_2min", 2), ("7b_ragged16", 2),
                                          ("7b_10min_paper", 2)])
def test_schedule_from_host_caches_gathers_each_layer_at_its_final_level(ap, name, streams):
    """run_from_host: caches in pinned host memory, every layer's rows gathered over the host
    link once, at the level that layer ends at.  Each step's indices, offsets, modality and the
    final hidden states equal the per-step device schedule's bit for bit, and every layer's final
    cache equals its own step's device output and the original rows at the composed indices
    (oracle compact_rows)."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    n = len(pp.layers)
    ends = list(pp.layers[1:]) + [pp.L]
    ref_kv, ref_m = [], []
    for i in range(n):                           # the device schedule, one step at a time
        pp.run_step(i)
        k, v = pp.output_kv(i)
        c = ends[i] - pp.layers[i]
        ref_kv.append((k[:c].clone(), v[:c].clone()))
        ref_m.append(pp.mod_out[i % 2][:pp.t_out[i]].clone())
    torch.cuda.synchronize()
    ref_keep = [pp.keep_idx[i][:pp.t_out[i]].clone() for i in range(n)]
    ref_cu = [np.asarray(c).copy() for c in pp.new_cu]
    ref_h = pp.output_hidden(n - 1).clone()
    h_k = pp.k_in.cpu().pin_memory()
    h_v = pp.v_in.cpu().pin_memory()
    h_h = pp.hidden_in.cpu().pin_memory()
    for buf in pp.k_out + pp.v_out + pp.h_out + pp.mod_out + pp.keep_idx:
        buf.zero_()
    pp.k_in[1:].zero_()                          # only the scored layer's keys stay on the device
    pp.v_in.zero_()
    pp.hidden_in.zero_()
    side = torch.cuda.Stream() if streams == 2 else None
    pp.run_from_host(h_k, h_v, h_h, gather_stream=side)
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    for i in range(n):
        assert torch.equal(pp.keep_idx[i][:pp.t_out[i]], ref_keep[i]), i
        np.testing.assert_array_equal(pp.new_cu[i], ref_cu[i])
    assert torch.equal(pp.mod_out[(n - 1) % 2][:pp.t_out[n - 1]], ref_m[n - 1])
    assert torch.equal(pp.output_hidden(n - 1).view(torch.int16), ref_h.view(torch.int16))
    k_np, v_np = h_k.view(torch.int16).numpy(), h_v.view(torch.int16).numpy()
    comp = np.arange(pp.T0)
    for i in range(n):
        comp = comp[pp.keep_idx[i][:pp.t_out[i]].cpu().numpy()]
        k, v = pp.final_kv(i)
        assert torch.equal(k.view(torch.int16), ref_kv[i][0].view(torch.int16)), i
        assert torch.equal(v.view(torch.int16), ref_kv[i][1].view(torch.int16)), i
        l0 = pp.layers[i] - pp.layers[0]
        for j in (0, k.shape[0] - 1):            # first and last layer of the step's range
            np.testing.assert_array_equal(k[j].view(torch.int16).cpu().numpy(),
                                          oracle.compact_rows(k_np[l0 + j], comp))
            np.testing.assert_array_equal(v[j].view(torch.int16).cpu().numpy(),
                                          oracle.compact_rows(v_np[l0 + j], comp))


@pytest.mark.parametrize("name", ["7b_2min", "7b_ragged16"])
def test_final_level_schedule_from_device_inputs(ap, name):
    """run_from_host with the device inputs as its source (every layer written once, at its final
    level, by device gathers): the same indices as the per-step schedule, and every layer's final
    cache equal to its own step's output, bit for bit."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode)
    fill_progressive_inputs(pp, wl)
    n = len(pp.layers)
    ends = list(pp.layers[1:]) + [pp.L]
    ref = []
    for i in range(n):
        pp.run_step(i)
        k, v = pp.output_kv(i)
        c = ends[i] - pp.layers[i]
        ref.append((pp.keep_idx[i][:pp.t_out[i]].clone(), k[:c].clone(), v[:c].clone()))
    ref_h = pp.output_hidden(n - 1).clone()
    for buf in pp.keep_idx + pp.h_out:
        buf.zero_()
    pp.run_from_host(pp.k_in, pp.v_in, pp.hidden_in)
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    for i in range(n):
        k, v = pp.final_kv(i)
        assert torch.equal(pp.keep_idx[i][:pp.t_out[i]], ref[i][0]), i
        assert torch.equal(k.view(torch.int16), ref[i][1].view(torch.int16)), i
        assert torch.equal(v.view(torch.int16), ref[i][2].view(torch.int16)), i
    assert torch.equal(pp.output_hidden(n - 1).view(torch.int16), ref_h.view(torch.int16))


@pytest.mark.parametrize("name", ["7b_2min", "7b_10min_paper"])
def test_slicing_below_the_pruning_layers_keeps_every_layer_consistent(ap, name):
    """With slice_below, every step also compacts the caches of the layers below its
    pruning layer; afterwards layer j's cache holds the original rows of layer j at
    the tokens kept by all steps, for every layer (checked bit for bit)."""
    from paper_2608_08794_gb300.schedule import ProgressivePrune, schedule_keep_counts
    from synth import workload
    from synth.device import fill_progressive_inputs

    wl = workload(name)
    cu0, cuq = wl.cu_seqlens(), wl.cu_qlens()
    na = np.array([s.n_audio for s in wl.seqs], np.int32)
    nv = np.array([s.n_visual for s in wl.seqs], np.int32)
    mod_d = torch.from_numpy(wl.modality()).cuda()
    counts, mode = schedule_keep_counts(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, mod_d,
                                        len(wl.prune_layers), wl.ratios, wl.joint_step_keep)
    pp = ProgressivePrune(cu0, cuq, na, nv, wl.num_q_heads, wl.num_kv_heads, wl.num_layers, wl.hidden,
                          wl.prune_layers, counts, select_mode=mode, slice_below=True)
    fill_progressive_inputs(pp, wl)
    pp.run()
    torch.cuda.synchronize()
    assert ap.apack_device_error(pp.ws) == ap.APACK_OK
    composite = torch.arange(wl.total_tokens, device="cuda")
    for i in range(len(wl.prune_layers)):
        composite = composite.index_select(0, pp.keep_idx[i][:pp.t_out[i]].long())
    last = len(wl.prune_layers) - 1
    l0, l_last = wl.prune_layers[0], wl.prune_layers[last]
    low_k, low_v = pp.output_low_kv(last)
    top_k, top_v = pp.output_kv(last)
    for j in range(wl.num_layers):
        src_k = pp.k_low_in[j] if j < l0 else pp.k_in[j - l0]
        src_v = pp.v_low_in[j] if j < l0 else pp.v_in[j - l0]
        got_k = low_k[j] if j < l_last else top_k[j - l_last]
        got_v = low_v[j] if j < l_last else top_v[j - l_last]
        assert torch.equal(got_k.view(torch.int16), src_k.index_select(0, composite).view(torch.int16)), j
        assert torch.equal(got_v.view(torch.int16), src_v.index_select(0, composite).view(torch.int16)), j
