"""Pins for the fp64 CPU oracle (oracle/): it is checked against things other
than itself -- a hand-worked example, hand-written scan orders, brute-force
quadratic forms, closed forms and invariants of the recurrence in Sec. 3.1 --
so that a dropped term, a wrong sign or index, a transposed operand or a wrong
scan order fails at least one test.  Everything here runs on the CPU."""
import json
import os

import numpy as np
import pytest

import oracle
from paper_2609_26590_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
ORDERS = (oracle.ROW_FWD, oracle.ROW_REV, oracle.COL_FWD, oracle.COL_REV)


def _scan_by_hand(order, gh, gw):
    """Scan order written out as nested loops over rows / columns (independent
    of the oracle's index formula)."""
    row_major = [y * gw + x for y in range(gh) for x in range(gw)]
    col_major = [y * gw + x for x in range(gw) for y in range(gh)]
    return {oracle.ROW_FWD: row_major, oracle.ROW_REV: row_major[::-1],
            oracle.COL_FWD: col_major, oracle.COL_REV: col_major[::-1]}[order]


def _rand(rng, B, T, H, Dk, Dv, gate_scale=1.0):
    q = rng.standard_normal((B, T, H, Dk))
    k = rng.standard_normal((B, T, H, Dk))
    v = rng.standard_normal((B, T, H, Dv))
    g = -gate_scale * rng.random((B, T, H, Dk))          # log-decay <= 0
    return q, k, v, g


def _brute_force(q, k, v, g, gh, gw, order):
    """o_t = sum_{s<=t} (q_t . (prod_{r=s+1..t} gamma_r * k_s)) v_s along the scan,
    and final = sum_s Diag(prod_{r>s} gamma_r) k_s^T v_s (quadratic form)."""
    B, T, H, Dk = q.shape
    Dv = v.shape[3]
    seq = _scan_by_hand(order, gh, gw)
    out = np.zeros((B, T, H, Dv))
    fs = np.zeros((B, H, Dk, Dv))
    gam = np.exp(g)
    for b in range(B):
        for h in range(H):
            for pt, t in enumerate(seq):
                acc = np.zeros(Dv)
                for ps in range(pt + 1):
                    s = seq[ps]
                    decay = np.ones(Dk)
                    for pr in range(ps + 1, pt + 1):
                        decay = decay * gam[b, seq[pr], h]
                    acc += np.dot(q[b, t, h], decay * k[b, s, h]) * v[b, s, h]
                out[b, t, h] = acc
            for ps in range(T):
                s = seq[ps]
                decay = np.ones(Dk)
                for pr in range(ps + 1, T):
                    decay = decay * gam[b, seq[pr], h]
                fs[b, h] += np.outer(decay * k[b, s, h], v[b, s, h])
    return out, fs


def _rel(a, b):
    return np.linalg.norm((a - b).ravel()) / max(np.linalg.norm(b.ravel()), 1e-300)


# --------------------------------------------------------------------------------------
# hand-worked fixtures
# --------------------------------------------------------------------------------------

def test_scan_orders_match_hand_lists():
    with open(os.path.join(GOLDEN, "scan_orders_2x3.json")) as f:
        gold = json.load(f)
    for order, name in oracle.ORDER_NAMES.items():
        got = oracle.scan_tokens(order, gold["grid_h"], gold["grid_w"])
        assert got.tolist() == gold[name], name
        assert _scan_by_hand(order, gold["grid_h"], gold["grid_w"]) == gold[name], name


def _golden_case():
    with open(os.path.join(GOLDEN, "hand_worked_1x3.json")) as f:
        gold = json.load(f)
    q = np.array(gold["q"], float).reshape(1, 3, 1, 2)
    k = np.array(gold["k"], float).reshape(1, 3, 1, 2)
    v = np.array(gold["v"], float).reshape(1, 3, 1, 3)
    g = np.log(np.array(gold["gamma"], float)).reshape(1, 3, 1, 2)
    return gold, q, k, v, g


@pytest.mark.parametrize("name,order", [("row_fwd", oracle.ROW_FWD), ("row_rev", oracle.ROW_REV)])
def test_hand_worked_recurrence(name, order):
    gold, q, k, v, g = _golden_case()
    out, fs = oracle.recurrence(q, k, v, g, 1, 3, order)
    np.testing.assert_allclose(out.reshape(3, 3), gold[name]["out"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(fs.reshape(2, 3), gold[name]["final_state"], rtol=0, atol=1e-14)


@pytest.mark.parametrize("chunk", [1, 2, 3, 64])
@pytest.mark.parametrize("name,order", [("row_fwd", oracle.ROW_FWD), ("row_rev", oracle.ROW_REV)])
def test_hand_worked_chunkwise(name, order, chunk):
    gold, q, k, v, g = _golden_case()
    out, fs = oracle.chunkwise(q, k, v, g, 1, 3, order, chunk=chunk)
    np.testing.assert_allclose(out.reshape(3, 3), gold[name]["out"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(fs.reshape(2, 3), gold[name]["final_state"], rtol=0, atol=1e-14)


# --------------------------------------------------------------------------------------
# brute force on tiny inputs
# --------------------------------------------------------------------------------------

@pytest.mark.parametrize("order", ORDERS)
@pytest.mark.parametrize("gh,gw", [(3, 5), (4, 2), (1, 7), (6, 1)])
def test_brute_force_quadratic_form(order, gh, gw):
    rng = np.random.default_rng(100 + order * 10 + gh)
    q, k, v, g = _rand(rng, 2, gh * gw, 2, 3, 4, gate_scale=0.7)
    ref_o, ref_s = _brute_force(q, k, v, g, gh, gw, order)
    o, s = oracle.recurrence(q, k, v, g, gh, gw, order)
    assert _rel(o, ref_o) < 1e-12
    assert _rel(s, ref_s) < 1e-12
    oc, sc = oracle.chunkwise(q, k, v, g, gh, gw, order, chunk=4)
    assert _rel(oc, ref_o) < 1e-12
    assert _rel(sc, ref_s) < 1e-12


def test_pairs_subset_matches_full():
    rng = np.random.default_rng(7)
    q, k, v, g = _rand(rng, 3, 12, 4, 5, 3)
    full_o, full_s = oracle.recurrence(q, k, v, g, 3, 4, oracle.COL_REV)
    pairs = [(2, 1), (0, 3)]
    o, s = oracle.recurrence(q, k, v, g, 3, 4, oracle.COL_REV, pairs=pairs)
    for b, h in pairs:
        np.testing.assert_array_equal(o[b, :, h], full_o[b, :, h])
        np.testing.assert_array_equal(s[b, h], full_s[b, h])
    assert np.isnan(o[1, :, 0]).all()


# --------------------------------------------------------------------------------------
# closed forms
# --------------------------------------------------------------------------------------

@pytest.mark.parametrize("order", ORDERS)
def test_gate_one_is_causal_linear_attention(order):
    gh, gw = 5, 7
    rng = np.random.default_rng(11)
    q, k, v, _ = _rand(rng, 2, gh * gw, 3, 6, 5)
    g = np.zeros_like(q)
    o, s = oracle.recurrence(q, k, v, g, gh, gw, order)
    seq = np.array(_scan_by_hand(order, gh, gw))
    for b in range(2):
        for h in range(3):
            Q, K, V = q[b, seq, h], k[b, seq, h], v[b, seq, h]
            ref = np.tril(Q @ K.T) @ V                      # ((Q K^T) * causal mask) V
            assert _rel(o[b, seq, h], ref) < 1e-12
            assert _rel(s[b, h], K.T @ V) < 1e-12            # no decay: S_T = K^T V


@pytest.mark.parametrize("order", ORDERS)
def test_gate_zero_is_diagonal(order):
    gh, gw = 4, 6
    rng = np.random.default_rng(12)
    q, k, v, _ = _rand(rng, 1, gh * gw, 2, 5, 3)
    g = np.full_like(q, -np.inf)                            # gamma = 0: state resets every token
    o, s = oracle.recurrence(q, k, v, g, gh, gw, order)
    ref = np.einsum("bthi,bthi->bth", q, k)[..., None] * v
    assert _rel(o, ref) < 1e-14
    last = _scan_by_hand(order, gh, gw)[-1]
    ref_s = np.einsum("bhi,bhj->bhij", k[:, last], v[:, last])
    assert _rel(s, ref_s) < 1e-14
    # the chunkwise model needs finite log-decays; -1e4 is gamma = 0 in floating point
    oc, sc = oracle.chunkwise(q, k, v, np.full_like(q, -1e4), gh, gw, order, chunk=5)
    assert _rel(oc, ref) < 1e-14
    assert _rel(sc, ref_s) < 1e-14


def test_single_token():
    rng = np.random.default_rng(13)
    q, k, v, g = _rand(rng, 2, 1, 3, 4, 6)
    o, s = oracle.recurrence(q, k, v, g, 1, 1, oracle.COL_FWD)
    ref = np.einsum("bthi,bthi->bth", q, k)[..., None] * v
    assert _rel(o, ref) < 1e-14
    assert _rel(s, np.einsum("bhi,bhj->bhij", k[:, 0], v[:, 0])) < 1e-14


# --------------------------------------------------------------------------------------
# invariants
# --------------------------------------------------------------------------------------

def test_reverse_scan_is_forward_scan_on_reversed_tokens():
    gh, gw = 6, 5
    rng = np.random.default_rng(14)
    q, k, v, g = _rand(rng, 2, gh * gw, 2, 4, 3)
    o_rev, s_rev = oracle.recurrence(q, k, v, g, gh, gw, oracle.ROW_REV)
    flip = lambda a: a[:, ::-1]
    o_f, s_f = oracle.recurrence(flip(q), flip(k), flip(v), flip(g), gh, gw, oracle.ROW_FWD)
    assert _rel(o_rev, flip(o_f)) < 1e-14
    assert _rel(s_rev, s_f) < 1e-14


@pytest.mark.parametrize("col_order,row_order", [(oracle.COL_FWD, oracle.ROW_FWD),
                                                 (oracle.COL_REV, oracle.ROW_REV)])
def test_column_scan_is_row_scan_of_transposed_grid(col_order, row_order):
    gh, gw = 4, 7
    rng = np.random.default_rng(15)
    q, k, v, g = _rand(rng, 1, gh * gw, 3, 4, 5)

    def transpose(a):   # token (y, x) of a gh x gw grid -> token (x, y) of a gw x gh grid
        B, T, H, D = a.shape
        return a.reshape(B, gh, gw, H, D).transpose(0, 2, 1, 3, 4).reshape(B, T, H, D)

    o_c, s_c = oracle.recurrence(q, k, v, g, gh, gw, col_order)
    o_r, s_r = oracle.recurrence(transpose(q), transpose(k), transpose(v), transpose(g), gw, gh,
                                 row_order)
    B, T, H, Dv = o_r.shape
    back = o_r.reshape(B, gw, gh, H, Dv).transpose(0, 2, 1, 3, 4).reshape(B, T, H, Dv)
    assert _rel(o_c, back) < 1e-14
    assert _rel(s_c, s_r) < 1e-14


def test_linearity_in_q_and_v():
    gh, gw = 3, 8
    rng = np.random.default_rng(16)
    q1, k, v1, g = _rand(rng, 1, gh * gw, 2, 4, 4)
    q2 = rng.standard_normal(q1.shape)
    v2 = rng.standard_normal(v1.shape)
    a, c = 0.75, -1.5
    f = lambda qq, vv: oracle.recurrence(qq, k, vv, g, gh, gw, oracle.COL_FWD)[0]
    assert _rel(f(a * q1 + c * q2, v1), a * f(q1, v1) + c * f(q2, v1)) < 1e-13
    assert _rel(f(q1, a * v1 + c * v2), a * f(q1, v1) + c * f(q1, v2)) < 1e-13


@pytest.mark.parametrize("chunk", [1, 7, 16, 64, 150])
@pytest.mark.parametrize("wid", [2, 3])
def test_chunk_size_invariance(chunk, wid):
    """Any chunk size gives the recurrence's result (Sec. 3.3: the chunked form
    changes only the schedule), under the workloads' gate distributions --
    including workload 3's strong decay (|A| ~ 90 per 64 tokens) and workload
    2's non-decaying channels."""
    w = wl.WORKLOADS[wid]
    inp = wl.make_inputs(1, 3, 10, 15, 16, 8, "f32", seed=77, tau=w.tau, z_mean=w.z_mean,
                         frac_nodecay=0.25 if w.frac_nodecay else 0.0)
    q, k, v, g = (inp[n].astype(np.float64) for n in ("q", "k", "v", "g"))
    for order in ORDERS:
        ref_o, ref_s = oracle.recurrence(q, k, v, g, 10, 15, order)
        o, s = oracle.chunkwise(q, k, v, g, 10, 15, order, chunk=chunk)
        assert _rel(o, ref_o) < 1e-12, (order, chunk)
        assert _rel(s, ref_s) < 1e-12, (order, chunk)


def test_rejects_bad_arguments():
    q = np.zeros((1, 4, 1, 2))
    with pytest.raises(ValueError):
        oracle.recurrence(q, q, q, q, 3, 2)
    with pytest.raises(RuntimeError):
        oracle.recurrence(q, q, q, q, 2, 2, order=7)


# ----------------------------------------------------------------- output gate
def test_gated_output_hand_worked():
    """Sec. 3.1 output gate on a hand-worked head (tests/golden/gated_epilogue_1x4.json)."""
    d = json.load(open(os.path.join(GOLDEN, "gated_epilogue_1x4.json")))
    o = np.array(d["o"]).reshape(1, 1, 1, 4)
    r = np.array(d["r_pre"]).reshape(1, 1, 1, 4)
    u = oracle.gated_output(o, r, np.array(d["weight"]), d["eps"])
    np.testing.assert_allclose(u.reshape(-1), d["u"], rtol=0, atol=1e-15)


def test_gated_output_matches_library_rmsnorm_and_silu():
    """The same gate through torch's own RMSNorm and SiLU routines, in float64."""
    import torch
    rng = np.random.Generator(np.random.PCG64(31))
    o = rng.standard_normal((2, 5, 3, 16)) * 4.0
    r = rng.standard_normal((2, 5, 3, 16)) * 3.0
    w = rng.standard_normal(16)
    eps = 1e-5
    ref = (torch.nn.functional.silu(torch.from_numpy(r)) *
           torch.nn.functional.rms_norm(torch.from_numpy(o), (16,), torch.from_numpy(w), eps)).numpy()
    np.testing.assert_allclose(oracle.gated_output(o, r, w, eps), ref, rtol=1e-12, atol=1e-14)


def test_gated_output_invariants():
    rng = np.random.Generator(np.random.PCG64(32))
    o = rng.standard_normal((1, 7, 4, 8))
    r = rng.standard_normal((1, 7, 4, 8)) * 2.0
    w = rng.standard_normal(8)
    eps = 1e-3
    u = oracle.gated_output(o, r, w, eps)
    # SiLU(z) - SiLU(-z) = z  =>  u(r) - u(-r) = r * RMSNorm(o) * w  (pins the sigmoid's sign)
    rms = np.sqrt(np.mean(o * o, axis=-1, keepdims=True) + eps)
    np.testing.assert_allclose(u - oracle.gated_output(o, -r, w, eps), r * o / rms * w, rtol=1e-12,
                               atol=1e-14)
    # scale invariance: o -> c o with eps -> c^2 eps leaves u unchanged
    np.testing.assert_allclose(oracle.gated_output(3.0 * o, r, w, 9.0 * eps), u, rtol=1e-12, atol=1e-14)
    # each head is normalised on its own: changing head 0 leaves the other heads' u unchanged
    o2 = o.copy()
    o2[:, :, 0, :] *= 10.0
    np.testing.assert_array_equal(oracle.gated_output(o2, r, w, eps)[:, :, 1:, :], u[:, :, 1:, :])
    # a zero gate pre-activation closes the output (SiLU(0) = 0); a large one passes r * RMSNorm(o)
    np.testing.assert_array_equal(oracle.gated_output(o, np.zeros_like(r), w, eps), 0.0 * u)
    big = np.full_like(r, 40.0)
    np.testing.assert_allclose(oracle.gated_output(o, big, w, eps), 40.0 * o / rms * w, rtol=1e-15)


# ---------------------------------------------------------------- Spatial SwiGLU (Eq. spatial_swiglu)

def _golden_sswiglu():
    with open(os.path.join(GOLDEN, "sswiglu_dwconv_2x3.json")) as f:
        return json.load(f)


def test_sswiglu_hand_worked_2x3():
    d = _golden_sswiglu()
    gh, gw = d["grid_h"], d["grid_w"]
    v = np.array(d["value_image"], dtype=np.float64).reshape(1, gh * gw, 1)
    gate = []
    for e in d["gate"]:
        gate.append(0.0 if e[0] == "zero" else e[2] * np.log(e[1]))
    g = np.array(gate).reshape(1, gh * gw, 1)
    w = np.array(d["weight"], dtype=np.float64).reshape(1, 3, 3)
    z = oracle.sswiglu_dwconv(g, v, w, np.array([d["bias"]]), gh, gw).ravel()
    expect = np.array([c * np.log(base) for c, base in d["z_as_coefficient_of_log"]])
    np.testing.assert_allclose(z, expect, rtol=1e-14, atol=1e-14)
    # the convolution alone: gate so large that SiLU(g) = g to double precision, then divide
    big = np.full_like(g, 1e3)
    conv = oracle.sswiglu_dwconv(big, v, w, np.array([d["bias"]]), gh, gw).ravel() / 1e3
    np.testing.assert_allclose(conv, d["conv"], rtol=1e-14)


def test_sswiglu_matches_scipy_correlate2d():
    scipy_signal = pytest.importorskip("scipy.signal")
    rng = np.random.Generator(np.random.PCG64(42))
    B, gh, gw, F = 2, 7, 4, 5
    g = rng.standard_normal((B, gh * gw, F))
    v = rng.standard_normal((B, gh * gw, F))
    w = rng.standard_normal((F, 3, 3))
    bias = rng.standard_normal(F)
    z = oracle.sswiglu_dwconv(g, v, w, bias, gh, gw)
    for b in range(B):
        for f in range(F):
            img = v[b, :, f].reshape(gh, gw)
            conv = scipy_signal.correlate2d(img, w[f], mode="same", boundary="fill", fillvalue=0.0)
            silu = g[b, :, f] * scipy_expit(g[b, :, f])
            np.testing.assert_allclose(z[b, :, f], silu * (conv.ravel() + bias[f]), rtol=1e-12, atol=1e-12)


def scipy_expit(x):
    special = pytest.importorskip("scipy.special")
    return special.expit(x)


def test_sswiglu_special_cases():
    rng = np.random.Generator(np.random.PCG64(7))
    B, gh, gw, F = 1, 5, 6, 3
    g = rng.standard_normal((B, gh * gw, F))
    v = rng.standard_normal((B, gh * gw, F))
    ident = np.zeros((F, 3, 3))
    ident[:, 1, 1] = 1.0
    silu = g * scipy_expit(g)
    # identity kernel, no bias: the tokenwise SwiGLU product
    np.testing.assert_allclose(oracle.sswiglu_dwconv(g, v, ident, None, gh, gw), silu * v, rtol=1e-14)
    # zero kernel: only the bias survives, gated
    bias = np.array([0.5, -2.0, 3.0])
    np.testing.assert_allclose(oracle.sswiglu_dwconv(g, v, np.zeros((F, 3, 3)), bias, gh, gw), silu * bias,
                               rtol=1e-14)
    # all-ones kernel on a constant image: 9c inside, 6c on edges, 4c at corners
    ones = np.ones((F, 3, 3))
    big = np.full((B, gh * gw, F), 1e3)
    conv = oracle.sswiglu_dwconv(big, np.full((B, gh * gw, F), 2.0), ones, None, gh, gw)[0, :, 0] / 1e3
    img = conv.reshape(gh, gw)
    assert img[2, 2] == 18.0 and img[0, 3] == 12.0 and img[0, 0] == 8.0 and img[gh - 1, gw - 1] == 8.0
    # a 1 x 1 grid sees only the centre tap
    w = rng.standard_normal((F, 3, 3))
    np.testing.assert_allclose(oracle.sswiglu_dwconv(g[:, :1], v[:, :1], w, None, 1, 1),
                               silu[:, :1] * v[:, :1] * w[:, 1, 1], rtol=1e-14)


# ---------------------------------------------------------------- retention gate from its projection (Sec. 3.1)

def test_gate_producer_hand_worked():
    with open(os.path.join(GOLDEN, "gate_producer_2tok.json")) as f:
        d = json.load(f)
    a = np.array(d["a_low"], dtype=np.float64) * np.log(3.0)
    g = oracle.gate_producer(a, np.array(d["w2"]), np.array(d["bias"]), d["tau"])
    expect = np.array([[np.log(v) for _, v in tok] for tok in d["g"]]).reshape(1, 2, 1, 2)
    np.testing.assert_allclose(g, expect, rtol=1e-14, atol=1e-15)


def test_gate_producer_matches_scipy_log_expit():
    special = pytest.importorskip("scipy.special")
    rng = np.random.Generator(np.random.PCG64(11))
    B, T, r, H, Dk, tau = 2, 5, 16, 3, 8, 16.0
    a = rng.standard_normal((B, T, r)) * 3
    w2 = rng.standard_normal((H, r, Dk))
    b = rng.standard_normal((H, Dk))
    g = oracle.gate_producer(a, w2, b, tau)
    for h in range(H):
        z = a @ w2[h] + b[h]                              # [B, T, Dk]
        np.testing.assert_allclose(g[:, :, h, :], special.log_expit(z) / tau, rtol=1e-12, atol=1e-300)


def test_gate_producer_special_cases():
    rng = np.random.Generator(np.random.PCG64(12))
    a = rng.standard_normal((1, 4, 16))
    b = rng.standard_normal((2, 8))
    # W2 = 0: every token gets logsigmoid(b) / tau
    g = oracle.gate_producer(a, np.zeros((2, 16, 8)), b, 4.0)
    np.testing.assert_allclose(g, np.broadcast_to(-np.log1p(np.exp(-b)) / 4.0, g.shape), rtol=1e-14)
    # tau scales g; g <= 0 always (gamma in (0, 1]); extreme pre-activations stay finite
    w2 = rng.standard_normal((2, 16, 8)) * 100
    g1, g2 = oracle.gate_producer(a, w2, b, 1.0), oracle.gate_producer(a, w2, b, 16.0)
    np.testing.assert_allclose(g2, g1 / 16.0, rtol=1e-14)
    assert np.all(g1 <= 0) and np.all(np.isfinite(g1))
    # z = 0: gamma^tau = 1/2
    g0 = oracle.gate_producer(np.zeros((1, 1, 16)), w2, np.zeros((2, 8)), 2.0)
    np.testing.assert_allclose(g0, np.full(g0.shape, -np.log(2.0) / 2.0), rtol=1e-15)
