"""bsr_plan_*: a product sequence captured once into a CUDA graph.

Section 2.2's task buffer reuses identical tasks and schedules similar ones
next to each other. A plan over independent products groups those that share
X, puts kernels of one template (and handles of one schedule) next to each
other and fuses them as bsr_spmm_batch does; a plan over dependent products
(a chain of layers) keeps their order. Every replay must give, bit for bit,
what the same bsr_spmm calls give on the buffers' current contents, and the
products must stay within the oracle's tolerance."""
import numpy as np
import pytest
import torch

import oracle
import synth
from tests.gpu_util import build_on_gpu, check_product, to_dev, to_host

pytestmark = pytest.mark.gpu


def _bsr():
    import paper_2106_08846_gb300 as bsr
    return bsr


def _weight(seed, M, K, R, C, dtype, density, long_rows=()):
    MB, KB = M // R, K // C
    if long_rows:
        cnt = np.full(MB, max(1, int(KB * density)), dtype=np.int64)
        cnt[list(long_rows)] = KB
        mask = synth.mask_from_row_counts(seed, cnt, KB)
    else:
        mask = synth.uniform_block_mask(seed, MB, KB, max(1, int(round(MB * KB * density))))
    return synth.make_weight("p", seed, M, K, R, C, dtype, 0, mask=mask)


def _handle(w):
    bsr = _bsr()
    return bsr.bsr_create(*build_on_gpu(w.W, w.R, w.C), w.R, w.C, w.M, w.K)


def _singles(hs, Xs, bs, Ms, Ns):
    """The same products as separate bsr_spmm calls (fresh outputs)."""
    bsr = _bsr()
    out = []
    for h, X, b, M, N in zip(hs, Xs, bs, Ms, Ns):
        Y = torch.empty((N, M), device="cuda", dtype=X.dtype)
        bsr.bsr_spmm(h, X, b, Y, N)
        out.append(Y)
    torch.cuda.synchronize()
    return [to_host(y) for y in out]


def test_plan_of_independent_products_groups_fuses_and_matches_single_calls():
    """Two attention layers' Q/K/V (sharing the layer's X) and O (its own X),
    plus, on layer 0's X, a tensor-core weight, a generic-kernel weight, a
    weight with split rows and a second handle on Q0's structure: one plan,
    replayed twice with new X contents."""
    bsr = _bsr()
    N, H = 200, 256
    ws = []
    for layer in range(2):
        for j, d in enumerate((0.3, 0.2, 0.1, 0.25)):                 # Q, K, V, O
            ws.append(_weight(2000 + 10 * layer + j, H, H, 32, 1, "f32", d))
    ws.append(_weight(2100, H, H, 32, 32, "f32", 0.3))               # 8: tensor cores
    ws.append(_weight(2101, 255, H, 3, 2, "f32", 0.2))                # 9: generic kernel
    ws.append(_weight(2102, H, H, 16, 1, "f32", 0.05, long_rows=(1, 6)))   # 10: split rows
    ws.append(ws[0])                                                  # 11: Q0's structure, second handle
    hs = [_handle(w) for w in ws]
    assert hs[11].schedule()["cache_hit"] == 1 and hs[10].schedule()["split_rows"] >= 1
    assert [hs[i].schedule()["variant"] for i in (0, 8, 9)] == ["xstage", "tcgen05", "generic"]
    X_np = [synth.activations(2200 + i, N, H, "f32") for i in range(4)]   # layer0 in, layer0 attn, layer1 in, layer1 attn
    Xd = [to_dev(x) for x in X_np]
    x_of = [0, 0, 0, 1, 2, 2, 2, 3, 0, 0, 0, 0]
    Xs = [Xd[k] for k in x_of]
    bs = [to_dev(w.bias) for w in ws]
    bs[9] = None
    Ys = [torch.empty((N, w.M), device="cuda") for w in ws]
    plan = bsr.bsr_plan_create(hs, Xs, bs, Ys, independent=True)
    order, call, n_kernels = plan.order()
    assert sorted(order) == list(range(len(ws)))
    # the products on layer 0's input come first and share calls: Q0, K0, V0 and
    # the second Q0 handle (same template) are fused; the split-row weight runs
    # on the SIMT kernel with a different block shape, the generic one last
    pos = {p: k for k, p in enumerate(order)}
    first = [p for p in order if x_of[p] == 0]
    assert order[:len(first)] == first and first[-1] == 9
    assert call[pos[0]] == call[pos[1]] == call[pos[2]] == call[pos[11]]
    assert abs(pos[0] - pos[11]) == 1                                 # one schedule, adjacent
    assert len(set(call)) < len(ws) and n_kernels < sum(h.schedule()["launches_per_call"] for h in hs)
    for rep in range(2):
        if rep:
            for k in range(4):
                X_np[k] = synth.activations(2300 + k, N, H, "f32")
                Xd[k].copy_(to_dev(X_np[k]))
        plan.launch()
        torch.cuda.synchronize()
        got = [to_host(y) for y in Ys]
        want = _singles(hs, Xs, bs, [w.M for w in ws], [N] * len(ws))
        for i, (g, w) in enumerate(zip(got, want)):
            assert np.array_equal(g, w), i
        for i in (0, 3, 8, 9, 10):
            check_product(got[i], oracle.bsr_from_dense(ws[i].W, ws[i].R, ws[i].C), X_np[x_of[i]],
                          None if bs[i] is None else ws[i].bias, ws[i].M)
    for h in hs:
        assert h.check_device_status() == 0
    plan.destroy()


def test_plan_of_a_chain_keeps_order_and_replays_on_new_input():
    """X -> 32x1 -> 32x32 (tensor cores) -> 16x1 with split rows -> 1x1, each
    product's X the previous product's Y (not independent): the plan keeps the
    order, one call per product; a replay after X changes gives the new chain."""
    bsr = _bsr()
    N = 130
    ws = [_weight(2401, 256, 512, 32, 1, "f32", 0.2), _weight(2402, 512, 256, 32, 32, "f32", 0.3),
          _weight(2403, 256, 512, 16, 1, "f32", 0.05, long_rows=(2,)), _weight(2404, 512, 256, 1, 1, "f32", 0.2)]
    hs = [_handle(w) for w in ws]
    X0 = to_dev(synth.activations(2405, N, 512, "f32"))
    Ys = [torch.empty((N, w.M), device="cuda") for w in ws]
    Xs = [X0] + Ys[:-1]
    bs = [to_dev(w.bias) for w in ws]
    plan = bsr.bsr_plan_create(hs, Xs, bs, Ys, independent=False)
    order, call, _ = plan.order()
    assert order == [0, 1, 2, 3] and call == [0, 1, 2, 3]
    for seed in (2406, 2407):
        X_np = synth.activations(seed, N, 512, "f32")
        X0.copy_(to_dev(X_np))
        plan.launch()
        torch.cuda.synchronize()
        got = [to_host(y) for y in Ys]
        ins = [X_np] + got[:-1]
        for i, w in enumerate(ws):   # each product against the oracle on its actual input
            check_product(got[i], oracle.bsr_from_dense(w.W, w.R, w.C), ins[i], w.bias, w.M)
        # and bit for bit against the same chain of single calls
        xs = [X0]
        for i, (h, w) in enumerate(zip(hs, ws)):
            Y = torch.empty((N, w.M), device="cuda")
            bsr.bsr_spmm(h, xs[-1], bs[i], Y, N)
            xs.append(Y)
        torch.cuda.synchronize()
        for i in range(4):
            assert np.array_equal(got[i], to_host(xs[i + 1])), i


def test_plan_owns_its_workspace_and_splits_a_repeated_handle():
    """One split-row handle used twice on the same X (two biases): the plan
    puts the two uses in different calls; a later bsr_spmm with a larger N
    regrows the handle's own workspace, and the plan still replays correctly."""
    bsr = _bsr()
    N = 100
    w = _weight(2501, 256, 512, 16, 1, "f32", 0.05, long_rows=(0, 3))
    h = _handle(w)
    X_np = synth.activations(2502, N, 512, "f32")
    X = to_dev(X_np)
    b1 = to_dev(w.bias)
    b2 = to_dev(np.ascontiguousarray(w.bias[::-1]))
    Y1, Y2 = torch.empty((N, 256), device="cuda"), torch.empty((N, 256), device="cuda")
    plan = bsr.bsr_plan_create([h, h], [X, X], [b1, b2], [Y1, Y2], independent=True)
    order, call, _ = plan.order()
    assert order == [0, 1] and call == [0, 1]
    big = 4 * N
    Xb = to_dev(synth.activations(2503, big, 512, "f32"))
    Yb = torch.empty((big, 256), device="cuda")
    bsr.bsr_spmm(h, Xb, b1, Yb, big)   # grows the handle's workspace
    plan.launch()
    torch.cuda.synchronize()
    want = _singles([h, h], [X, X], [b1, b2], [256, 256], [N, N])
    assert np.array_equal(to_host(Y1), want[0]) and np.array_equal(to_host(Y2), want[1])
    check_product(to_host(Y2), oracle.bsr_from_dense(w.W, 16, 1), X_np, np.ascontiguousarray(w.bias[::-1]), 256)
    assert h.check_device_status() == 0


def test_plan_bf16_tensor_core_group():
    """bf16 Q/K/V on one X (16x16 tensor cores and re-blocked 1x1) fused in one
    plan call; bit-identical to single calls."""
    bsr = _bsr()
    N = 300
    ws = [_weight(2601, 256, 256, 16, 16, "bf16", 0.3), _weight(2602, 256, 256, 16, 16, "bf16", 0.2),
          _weight(2603, 256, 256, 1, 1, "bf16", 0.3)]
    hs = [_handle(w) for w in ws]
    X_np = synth.activations(2604, N, 256, "bf16")
    X = to_dev(X_np)
    bs = [to_dev(w.bias) for w in ws]
    Ys = [torch.empty((N, 256), device="cuda", dtype=X.dtype) for _ in ws]
    plan = bsr.bsr_plan_create(hs, [X] * 3, bs, Ys, independent=True)
    order, call, _ = plan.order()
    assert call[order.index(0)] == call[order.index(1)]
    plan.launch()
    torch.cuda.synchronize()
    want = _singles(hs, [X] * 3, bs, [256] * 3, [N] * 3)
    for i in range(3):
        got = to_host(Ys[i])
        assert np.array_equal(got.view(np.uint16), want[i].view(np.uint16)), i
        check_product(got, oracle.bsr_from_dense(ws[i].W, ws[i].R, ws[i].C), X_np, ws[i].bias, 256)


def test_plan_argument_errors():
    bsr = _bsr()
    N = 64
    w = _weight(2701, 128, 128, 8, 1, "f32", 0.2)
    h1, h2 = _handle(w), _handle(_weight(2702, 128, 128, 8, 1, "f32", 0.3))
    X = to_dev(synth.activations(2703, N, 128, "f32"))
    Y1, Y2 = torch.empty((N, 128), device="cuda"), torch.empty((N, 128), device="cuda")
    with pytest.raises(bsr.BsrError):   # independent, but product 1 reads product 0's output
        bsr.bsr_plan_create([h1, h2], [X, Y1], None, [Y1, Y2], independent=True)
    bsr.bsr_plan_create([h1, h2], [X, Y1], None, [Y1, Y2], independent=False).destroy()   # a chain is fine
    with pytest.raises(bsr.BsrError):   # two outputs on one buffer
        bsr.bsr_plan_create([h1, h2], [X, X], None, [Y1, Y1], independent=True)
    with pytest.raises(bsr.BsrError):   # output overlapping its own input
        bsr.bsr_plan_create([h1], [X], None, [X], independent=False)
    with pytest.raises(bsr.BsrError):   # host buffers are not accepted
        bsr.bsr_plan_create([h1], [torch.zeros((N, 128))], None, [Y1], independent=False)
    empty = bsr.bsr_plan_create([], [], None, [], independent=True)   # nothing to run
    empty.launch()
    assert empty.order() == ([], [], 0)
    zero = bsr.bsr_plan_create([h1], [X], None, [Y1], Ns=[0])        # N = 0: a no-op product
    assert zero.order()[0] == []
    zero.launch()
    torch.cuda.synchronize()
