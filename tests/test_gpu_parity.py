"""GPU parity: the sm_103a kernels (through the C ABI) against the fp64 CPU oracle.

Pass rules:
  * h: |h_gpu - h_oracle| <= 1e-4 * h_oracle element-wise (exact zero where the oracle
    has zero).
  * s_g, RTN codes, packed nibbles: bit-exact.
  * refined codes and nibbles: bit-exact in every group except the oracle's near-ties
    (best and runner-up errors within 1e-6 relative); near-ties are counted and
    reported.  The search gets one fp32 h on both sides (the oracle's h rounded to
    fp32), so the comparison isolates the search.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2608_28113_gb300 as hs
from paper_2608_28113_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

H_RTOL = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    hs.load()
    oracle.set_threads(os.cpu_count() or 1)


def dev():
    return torch.device("cuda", 0)


def bits(t):
    return wl.bf16_bits(t)


def from_bits(b: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).view(torch.bfloat16)


def gpu_hessian(chunks, n):
    h = torch.zeros(n, dtype=torch.float32, device=dev())
    for x in chunks:
        hs.hscale_hessian_diag_accumulate(x, h)
    torch.cuda.synchronize()
    return h.cpu().numpy()


def oracle_hessian(chunks, n):
    h = np.zeros(n)
    for x in chunks:
        xb = bits(x)
        oracle.hessian_accumulate(xb, h, ld=xb.shape[1], n=n)
    return h


def assert_h_close(h_gpu, h_ref):
    h_gpu = h_gpu.astype(np.float64)
    zero = h_ref == 0
    assert np.all(h_gpu[zero] == 0)
    rel = np.abs(h_gpu[~zero] - h_ref[~zero]) / h_ref[~zero]
    assert rel.max(initial=0.0) <= H_RTOL, f"max rel err {rel.max():.3e}"
    return rel.max(initial=0.0)


def gpu_rtn(w):
    m, n = w.shape
    sg = torch.empty(1, dtype=torch.float32, device=dev())
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=dev())
    hs.hscale_rtn_scales(w, sg, codes, ws)
    torch.cuda.synchronize()
    return sg, codes


def gpu_refine(w, h32, sg, init, down, up, with_packed=True):
    m, n = w.shape
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    packed = torch.empty(m, n // 2, dtype=torch.uint8, device=dev()) if with_packed else None
    h = None if h32 is None else torch.from_numpy(np.ascontiguousarray(h32, np.float32)).to(dev())
    hs.hscale_refine_scales(w, h, sg, init, down, up, codes, packed)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), (packed.cpu().numpy() if with_packed else None)


def compare_search(ref, codes, packed, label=""):
    """Bit-exact outside near-ties.  Returns (groups, near_ties, mismatches_in_near_ties)."""
    nt = ref["near_tie"].astype(bool)
    diff_code = codes != ref["codes"]
    bad = diff_code & ~nt
    assert not bad.any(), f"{label}: {bad.sum()} code mismatches outside near-ties at {np.argwhere(bad)[:5]}"
    if packed is not None:
        m, ng = codes.shape
        pdiff = (packed.reshape(m, ng, 8) != ref["packed"].reshape(m, ng, 8)).any(axis=2)
        badp = pdiff & ~nt
        assert not badp.any(), f"{label}: {badp.sum()} nibble mismatches outside near-ties"
        # where the codes agree, the nibbles must agree too (final re-quantization is exact)
        assert not (pdiff & ~diff_code).any(), f"{label}: nibbles differ under an equal code"
    print(f"[parity] {label}: groups={codes.size} near_ties={int(nt.sum())} "
          f"near_tie_code_mismatches={int((diff_code & nt).sum())}")
    return codes.size, int(nt.sum()), int((diff_code & nt).sum())


def small_layer(seed=0, m=512, n=1024, sigma=0.02):
    w = wl.weight(m, n, sigma, seed, device="cpu")
    return w


# ------------------------------------------------------------------ Hessian pass

def test_hessian_single_chunk_small_layer():
    W = wl.WORKLOADS["layer-512x1024"]
    a = wl.channel_magnitudes(1024, W.sigma_a, W.outlier_channels, W.outlier_channel_mult, W.seed)
    x = wl.activation_chunk(2048, a, W.seed, 0)
    h_gpu = gpu_hessian([x.to(dev())], 1024)
    h_ref = oracle_hessian([x], 1024)
    print(f"[parity] hessian 2048x1024 max rel err {assert_h_close(h_gpu, h_ref):.3e}")


@pytest.mark.parametrize("n,tokens,chunk,pad", [
    (1040, 5000, 1536, 0),     # ragged column tile (1040 = 16 tiles + 16), chunk does not divide N
    (64, 300000, 300000, 0),   # one call longer than a launch's token limit
    (8, 3, 3, 8),              # minimum width, strided rows (ld = 16)
    (4096, 777, 256, 64),      # wide rows, ld = n + 64, ragged last chunk
    (14336, 4096, 4096, 0),    # MLP width
    (200, 9000, 4500, 8),      # last 128-channel tile 72 wide: second 64-channel box partly past n
    (136, 1000, 333, 0),       # last tile 8 wide: its second box wholly past n (not loaded)
    (4096, 8256, 8256, 0),     # chunk not a multiple of a 64-token stage per cluster CTA
])
def test_hessian_chunking_ragged_and_strided(n, tokens, chunk, pad):
    g = torch.Generator().manual_seed(n * 7 + tokens)
    base = (torch.randn(tokens, n + pad, generator=g) * torch.exp(torch.randn(n + pad, generator=g)))
    xb = base.to(torch.bfloat16)
    chunks_cpu = [xb[t:t + chunk, :n] for t in range(0, tokens, chunk)]
    xd = xb.to(dev())
    chunks_gpu = [xd[t:t + chunk, :n] for t in range(0, tokens, chunk)]
    h_gpu = gpu_hessian(chunks_gpu, n)
    h_ref = np.zeros(n)
    for c in chunks_cpu:
        cb = bits(c.contiguous())
        oracle.hessian_accumulate(cb, h_ref)
    assert_h_close(h_gpu, h_ref)


def test_hessian_closed_forms_and_empty_chunk():
    n = 192
    x = torch.full((1000, n), -1.5, dtype=torch.bfloat16, device=dev())
    h = torch.zeros(n, device=dev())
    hs.hscale_hessian_diag_accumulate(x, h)
    hs.hscale_hessian_diag_accumulate(x[:0], h)          # empty chunk: no-op
    torch.cuda.synchronize()
    assert torch.all(h == 1000 * 2.25)
    one_hot = torch.zeros(3 * n, n, dtype=torch.bfloat16, device=dev())
    idx = torch.arange(3 * n, device=dev())
    one_hot[idx, idx % n] = 2.0
    h.zero_()
    hs.hscale_hessian_diag_accumulate(one_hot, h)
    torch.cuda.synchronize()
    assert torch.all(h == 12.0)


def test_hessian_x_ready_flag_gives_the_same_bits():
    """The chunk stream with and without HSCALE_HESSIAN_X_READY (early X reads overlapping the
    previous chunk's kernel) gives the same h bit for bit, and a chunk written by the kernel
    just before the call on the same stream is read after that kernel is done."""
    g = torch.Generator().manual_seed(11)
    x = (torch.randn(8 * 4096, 1024, generator=g) * 2).to(torch.bfloat16).to(dev())
    hs_default = torch.zeros(1024, device=dev())
    hs_ready = torch.zeros(1024, device=dev())
    for c in range(8):
        hs.hscale_hessian_diag_accumulate(x[c * 4096:(c + 1) * 4096], hs_default)
    for c in range(8):
        hs.hscale_hessian_diag_accumulate_ex(x[c * 4096:(c + 1) * 4096], hs_ready, hs.HSCALE_HESSIAN_X_READY)
    torch.cuda.synchronize()
    assert torch.equal(hs_default, hs_ready)
    # producer kernel immediately before the call on the same stream
    y = torch.empty_like(x)
    h1 = torch.zeros(1024, device=dev())
    for c in range(8):
        blk = y[c * 4096:(c + 1) * 4096]
        torch.mul(x[c * 4096:(c + 1) * 4096], 1.0, out=blk)
        hs.hscale_hessian_diag_accumulate(blk, h1)
    torch.cuda.synchronize()
    assert torch.equal(h1, hs_default)
    assert hs.hscale_device_error_flags() == 0


def test_hessian_is_deterministic():
    g = torch.Generator().manual_seed(5)
    x = (torch.randn(20000, 4096, generator=g) * 3).to(torch.bfloat16).to(dev())
    outs = []
    for _ in range(3):
        h = torch.zeros(4096, device=dev())
        hs.hscale_hessian_diag_accumulate(x, h)
        outs.append(h.cpu())
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[1], outs[2])


# ------------------------------------------------------------------ global scale and RTN codes

def test_rtn_scales_match_oracle_bit_exact():
    for seed in range(4):
        w = small_layer(seed)
        sg, codes = gpu_rtn(w.to(dev()))
        s_ref, _ = oracle.global_scale(bits(w))
        assert sg.cpu().numpy()[0] == s_ref
        assert np.array_equal(codes.cpu().numpy(), oracle.rtn_codes(bits(w), s_ref))


def exact_tie_matrix():
    """Groups whose max sits exactly on each E4M3 ladder value and midpoint, under
    s_g = 2^-10 (amax = 2688 * 2^-10): RTN ties are decided by round-half-even."""
    ladder = oracle.e4m3_decode_table()[0:127]
    mids = 0.5 * (ladder[:-1] + ladder[1:])
    vs = [v for v in np.concatenate([ladder[1:], mids]) if v <= 448]
    w = np.zeros((len(vs), 32), np.float32)
    for i, v in enumerate(vs):
        w[i, 3] = 6 * v * 2.0 ** -10
        w[i, 17] = -w[i, 3] / 3.0
        w[i, 20:28] = np.linspace(-w[i, 3], w[i, 3], 8)
    w[0, 0] = 2688 * 2.0 ** -10
    return torch.from_numpy(w).to(torch.bfloat16)


def test_rtn_codes_exact_ties_and_saturation():
    w = exact_tie_matrix()
    sg, codes = gpu_rtn(w.to(dev()))
    s_ref, _ = oracle.global_scale(bits(w))
    assert sg.cpu().numpy()[0] == s_ref == np.float32(2.0 ** -10)
    assert np.array_equal(codes.cpu().numpy(), oracle.rtn_codes(bits(w), s_ref))
    sg_only = torch.empty(1, device=dev())
    ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=dev())
    hs.hscale_rtn_scales(w.to(dev()), sg_only, None, ws)   # codes = NULL: s_g only
    torch.cuda.synchronize()
    assert sg_only.item() == float(s_ref)


# ------------------------------------------------------------------ search (Algorithm 1)

def oracle_h32(seed, n, tokens=2048, sigma_a=1.0):
    a = wl.channel_magnitudes(n, sigma_a, 8, 50.0, seed)
    x = wl.activation_chunk(tokens, a, seed, 0)
    h = np.zeros(n)
    oracle.hessian_accumulate(bits(x), h)
    return h.astype(np.float32)


@pytest.mark.parametrize("down,up", [(4, 4), (9, 6), (0, 0), (1, 1), (8, 8), (16, 16), (0, 7), (125, 125)])
def test_refine_matches_oracle_small_layer(down, up):
    m, n = (512, 1024) if down + up < 40 else (64, 1024)
    w = small_layer(0, m, n)
    h32 = oracle_h32(0, n)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    ref = oracle.refine(bits(w), h32, s_ref, None, down, up)
    codes, packed = gpu_refine(wd, h32, sg, None, down, up)
    compare_search(ref, codes, packed, f"layer {m}x{n} window -{down}/+{up}")


def test_refine_with_init_codes_aliasing_and_no_packed_output():
    w = small_layer(1, 256, 512)
    h32 = oracle_h32(1, 512)
    wd = w.to(dev())
    sg, rtn = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    # arbitrary baseline codes (sign bits and off-ladder values included)
    g = np.random.default_rng(3)
    init = g.integers(0, 256, size=(256, 32)).astype(np.uint8)
    ref = oracle.refine(bits(w), h32, s_ref, init, 4, 4)
    buf = torch.from_numpy(init).to(dev())
    h = torch.from_numpy(h32).to(dev())
    packed = torch.empty(256, 256, dtype=torch.uint8, device=dev())
    hs.hscale_refine_scales(wd, h, sg, buf, 4, 4, buf, packed)   # codes_out aliases init_codes
    torch.cuda.synchronize()
    compare_search(ref, buf.cpu().numpy(), packed.cpu().numpy(), "init codes, in place")
    codes_np, _ = gpu_refine(wd, h32, sg, rtn, 4, 4, with_packed=False)
    ref2 = oracle.refine(bits(w), h32, s_ref, None, 4, 4)
    compare_search(ref2, codes_np, None, "rtn init codes, no packed output")


def test_refine_h_none_is_plain_mse_search():
    w = small_layer(2, 256, 1024)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    ref = oracle.refine(bits(w), None, s_ref, None, 9, 6)
    codes, packed = gpu_refine(wd, None, sg, None, 9, 6)
    compare_search(ref, codes, packed, "h = 1")


def test_refine_edge_groups():
    """All-zero groups, h = 0 on whole groups, the group holding amax (code 126, the
    upward walk clips), tiny groups near code 1 (the downward walk clips), -0."""
    rng = np.random.default_rng(11)
    m, n = 64, 256
    w = (rng.standard_t(4, size=(m, n)) * 0.02).astype(np.float32)
    w[0, :16] = 0.0                       # all-zero group
    w[1, :16] = -0.0                      # all negative zeros
    w[2, 16:32] *= 1e-4                   # tiny group near the bottom of the ladder
    w[3, 32:48] = 0.0
    w[3, 40] = 1e-6                       # one tiny non-zero
    w[5, 100] = 40.0                      # the tensor's amax: code 126
    w[6, 3] = 39.0
    wb = torch.from_numpy(w).to(torch.bfloat16)
    b = bits(wb)
    b[1, :16] = 0x8000
    wb = from_bits(b)
    h32 = oracle_h32(4, n)
    h32[48:64] = 0.0                      # h = 0 on a whole group column
    h32[64:80] = np.float32(1e-30)        # vanishing channel energy
    wd = wb.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(b)
    assert sg.cpu().numpy()[0] == s_ref
    for down, up in ((4, 4), (9, 6)):
        ref = oracle.refine(b, h32, s_ref, None, down, up)
        codes, packed = gpu_refine(wd, h32, sg, None, down, up)
        compare_search(ref, codes, packed, f"edge groups -{down}/+{up}")
        assert codes[5, 6] == ref["codes"][5, 6]


def test_group_amax_over_bf16_subnormals_and_signs():
    """The group amax (a packed bf16 max of magnitudes) where it decides the RTN code: every
    value a bf16 subnormal of either sign, +-0 mixes, a negative largest magnitude, under
    s_g = 2^-126 (the tensor's amax 21 * 2^-119, the smallest normal s_g), so that the
    codes of subnormal groups vary with their amax.  RTN codes, the search's own RTN start
    and the packed nibbles against the oracle."""
    rng = np.random.default_rng(17)
    m, n = 64, 512
    b = rng.integers(1, 0x80, size=(m, n), dtype=np.uint16)          # |w| subnormal
    b |= (rng.integers(0, 2, size=(m, n), dtype=np.uint16) << 15)   # random signs
    b[0, 0] = 0x0628                                                # 21 * 2^-119: the amax
    b[1, :16] = 0x8000                                              # all -0
    b[2, 16:32] = 0x0000
    b[2, 20] = 0x8045                                               # one negative subnormal
    b[3, 32:48] = 0x807F                                            # equal magnitudes, negative
    b[3, 40] = 0x007F
    for r in range(4, m):                                           # largest magnitude negative
        g = (r * 5) % (n // 16)
        b[r, 16 * g + (r % 16)] = 0x807F
    w = from_bits(b)
    wd = w.to(dev())
    sg, codes = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(b)
    assert s_ref == np.float32(2.0 ** -126) and sg.cpu().numpy()[0] == s_ref
    assert np.array_equal(codes.cpu().numpy(), oracle.rtn_codes(b, s_ref))
    h32 = oracle_h32(17, n)
    ref = oracle.refine(b, h32, s_ref, None, 4, 4)
    codes_g, packed_g = gpu_refine(wd, h32, sg, None, 4, 4)
    compare_search(ref, codes_g, packed_g, "bf16 subnormal groups")


def test_refine_inline_rtn_on_exact_e4m3_ties():
    """The search's own RTN start (init_codes = NULL) on groups whose max sits exactly on every
    E4M3 ladder value and midpoint (s_g = 2^-10): exact ties are decided half-to-even, as in
    hscale_rtn_scales; the codes below 8 (E4M3 subnormals) are included."""
    w = exact_tie_matrix()
    b = bits(w)
    m, n = w.shape
    h32 = oracle_h32(12, n)
    wd = w.to(dev())
    sg, rtn = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(b)
    assert np.array_equal(rtn.cpu().numpy(), oracle.rtn_codes(b, s_ref))
    for down, up in ((0, 0), (4, 4), (9, 6)):
        ref = oracle.refine(b, h32, s_ref, None, down, up)
        codes, packed = gpu_refine(wd, h32, sg, None, down, up)
        compare_search(ref, codes, packed, f"exact E4M3 ties -{down}/+{up}")
        if down == up == 0:
            assert np.array_equal(codes, rtn.cpu().numpy())


def test_refine_group_magnitudes_across_the_ladder():
    """Groups scaled over 2^-12 .. 2^0 of the tensor's amax, so their RTN codes cover the E4M3
    subnormals, every binade and the clipped walk at both ends of the ladder."""
    rng = np.random.default_rng(13)
    m, n = 96, 512
    w = (rng.standard_t(4, size=(m, n)) * 0.02).astype(np.float32)
    scale = 2.0 ** rng.uniform(-12, 0, size=(m, n // 16))
    w *= np.repeat(scale, 16, axis=1).astype(np.float32)
    w[0, 0] = 3.0
    wb = torch.from_numpy(w).to(torch.bfloat16)
    h32 = oracle_h32(14, n)
    wd = wb.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(wb))
    for down, up in ((4, 4), (9, 6), (16, 16)):
        ref = oracle.refine(bits(wb), h32, s_ref, None, down, up)
        codes, packed = gpu_refine(wd, h32, sg, None, down, up)
        compare_search(ref, codes, packed, f"magnitudes across the ladder -{down}/+{up}")
        assert (ref["codes"] < 8).any()


@pytest.mark.parametrize("m,n", [(1, 16), (3, 48), (33, 16 * 33), (1, 4096 * 4)])
def test_refine_tiny_and_ragged_shapes(m, n):
    w = wl.weight(m, n, 0.02, m * 1000 + n)
    h32 = oracle_h32(7, n)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    ref = oracle.refine(bits(w), h32, s_ref, None, 4, 4)
    codes, packed = gpu_refine(wd, h32, sg, None, 4, 4)
    compare_search(ref, codes, packed, f"shape {m}x{n}")


def test_refine_short_global_scale_exact_midpoint_ties():
    """amax = 2688 * 2^-7 gives s_g = 2^-7 exactly, so many |w| / (s_g l) land exactly on
    E2M1 midpoints: nibbles must follow round-half-even bit-exactly."""
    rng = np.random.default_rng(12)
    m, n = 128, 512
    grid = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 1.0, 3.0, 0.5])
    lad = oracle.e4m3_decode_table()[1:127]
    l = lad[rng.integers(40, 60, size=(m, n // 16))]
    q = grid[rng.integers(0, grid.size, size=(m, n))]
    w = (q * np.repeat(l, 16, axis=1) * 2.0 ** -7 * rng.choice([-1, 1], size=(m, n))).astype(np.float32)
    w[0, 0] = 2688 * 2.0 ** -7
    wb = torch.from_numpy(w).to(torch.bfloat16)
    b = bits(wb)
    s_ref, _ = oracle.global_scale(b)
    assert s_ref == np.float32(2.0 ** -7)
    h32 = oracle_h32(8, n)
    wd = wb.to(dev())
    sg, codes_rtn = gpu_rtn(wd)
    for down, up in ((4, 4), (0, 0)):
        ref = oracle.refine(b, h32, s_ref, None, down, up)
        codes, packed = gpu_refine(wd, h32, sg, None, down, up)
        compare_search(ref, codes, packed, f"exact midpoints -{down}/+{up}")


def test_pack_matches_oracle_bit_exact():
    w = small_layer(9, 256, 1024)
    wd = w.to(dev())
    sg, codes = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    rng = np.random.default_rng(9)
    for c in (codes.cpu().numpy(), rng.integers(0, 256, size=(256, 64)).astype(np.uint8)):
        ct = torch.from_numpy(c).to(dev())
        packed = torch.empty(256, 512, dtype=torch.uint8, device=dev())
        hs.hscale_pack_nvfp4(wd, sg, ct, packed)
        torch.cuda.synchronize()
        assert np.array_equal(packed.cpu().numpy(), oracle.pack(bits(w), s_ref, c))


def test_pack_full_size_q_proj():
    """hscale_pack_nvfp4 over the whole 4096 x 4096 q_proj matrix: with the search's own
    codes it reproduces the search's nibbles (every group), and with random codes (sign bit
    set, off-ladder bytes 0 and 127-255 clamped) it matches the oracle on sampled rows."""
    W = wl.WORKLOADS["llama8b-q_proj"]
    L = W.layers[0]
    m, n = L.out_features, L.in_features
    w = wl.weight(m, n, W.sigma_w, wl.chunk_seed(W.layer_seed(0), L.name, 0) & 0xFFFFFFFF, device=dev())
    h32 = oracle_h32(1, n, tokens=512)
    sg, _ = gpu_rtn(w)
    codes, packed = gpu_refine(w, h32, sg, None, 4, 4)
    out = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
    hs.hscale_pack_nvfp4(w, sg, torch.from_numpy(codes).to(dev()), out)
    torch.cuda.synchronize()
    assert np.array_equal(out.cpu().numpy(), packed)
    rng = np.random.default_rng(33)
    rnd = rng.integers(0, 256, size=(m, n // 16)).astype(np.uint8)
    hs.hscale_pack_nvfp4(w, sg, torch.from_numpy(rnd).to(dev()), out)
    torch.cuda.synchronize()
    rows = np.sort(rng.choice(m, size=64, replace=False))
    s_ref, _ = oracle.global_scale(bits(w))
    wb = bits(w[torch.from_numpy(rows).to(dev())])
    assert np.array_equal(out.cpu().numpy()[rows], oracle.pack(wb, s_ref, rnd[rows]))


def test_refine_launch_shape_does_not_change_results():
    """hscale_refine_scales_ex with 1, 2 or 5 resident CTAs per SM (more units per warp,
    other unit-to-warp assignment) writes the same bytes as the full launch."""
    w = small_layer(5, 512, 1024)
    h = torch.from_numpy(oracle_h32(5, 1024)).to(dev())
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    outs = []
    for k in (0, 1, 2, 5):
        codes = torch.empty(512, 64, dtype=torch.uint8, device=dev())
        packed = torch.empty(512, 512, dtype=torch.uint8, device=dev())
        hs.hscale_refine_scales_ex(wd, h, sg, None, 9, 6, codes, packed, k)
        torch.cuda.synchronize()
        outs.append((codes.cpu(), packed.cpu()))
    for c, p in outs[1:]:
        assert torch.equal(c, outs[0][0]) and torch.equal(p, outs[0][1])


def gpu_refine_ws(w, h, sg, init, fourover6, down, up, ctas_per_sm, ws):
    m, n = w.shape
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    packed = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
    hs.hscale_refine_scales_ws(w, h, sg, init, fourover6, down, up, codes, packed, ctas_per_sm, ws)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), packed.cpu().numpy()


def shared_schedule_ran(ws):
    """The work-shared kernel zeroes the workspace's first word and counts batches in it;
    the static deal leaves the workspace as it was (filled with 0xAB here)."""
    word = ws[:4].cpu().numpy()
    return not np.all(word == 0xAB)


@pytest.mark.parametrize("init", ["rtn", "given", "4over6"])
def test_search_schedules_match_oracle(init):
    """The three deals of the contiguous search on one matrix, each against the oracle on
    every group: the global work-sharing counter (hscale_refine_scales_ws, one resident CTA
    per SM, k = 8: a long search per warp), the per-SM queue (the matrix alone on the GPU,
    no workspace) and the static deal (CTAs capped at 7 per SM).  An odd row count makes
    units of consecutive queue positions straddle the end of a column chunk.  The
    workspace is reused for a second call, and all three write the same bytes."""
    m, n, down, up = 4095, 4096, 8, 8
    w = wl.weight(m, n, 0.02, 21, device="cpu")
    h32 = oracle_h32(21, n, sigma_a=1.5)
    wd, hd = w.to(dev()), torch.from_numpy(h32).to(dev())
    sg, rtn = gpu_rtn(wd)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    init_d = init_ref = None
    exclude = np.zeros((m, n // 16), np.uint8)
    if init == "given":
        init_d = rtn
        init_d[::7] = 200   # other starting codes (the sign bit is cleared on both sides)
        init_ref = init_d.cpu().numpy()
    elif init == "4over6":
        init_ref, nt = oracle.fourover6_codes(wb, s_ref)
        exclude = nt.astype(np.uint8)
    f46 = int(init == "4over6")
    ref = oracle.refine(wb, h32, s_ref, init_ref, down, up)
    ref["near_tie"] = ref["near_tie"] | exclude
    ws = torch.full((hs.hscale_refine_workspace_bytes(),), 0xAB, dtype=torch.uint8, device=dev())
    shared = gpu_refine_ws(wd, hd, sg, init_d, f46, down, up, 1, ws)
    assert shared_schedule_ran(ws)
    compare_search(ref, *shared, f"global counter {m}x{n} init {init}")
    again = gpu_refine_ws(wd, hd, sg, init_d, f46, down, up, 1, ws)
    queue = gpu_refine_ws(wd, hd, sg, init_d, f46, down, up, 0, None)
    compare_search(ref, *queue, f"per-SM queue {m}x{n} init {init}")
    static = gpu_refine_ws(wd, hd, sg, init_d, f46, down, up, 7, None)
    for other in (again, queue, static):
        assert np.array_equal(other[0], shared[0]) and np.array_equal(other[1], shared[1])


@pytest.mark.parametrize("m,n", [(1, 512 * 20000), (20000, 512)])
def test_search_schedules_on_extreme_shapes(m, n):
    """The per-SM queue (matrix alone, no workspace) and the global counter (workspace, one
    CTA per SM) where units are one row long and every unit is a new column chunk, or one
    chunk wide: against the oracle, and the same bytes as the static deal."""
    w = wl.weight(m, n, 0.02, 23, device="cpu")
    # h of 2048 tokens with the workload's channel magnitudes, in expectation (X itself would
    # be 2048 x n)
    a = wl.channel_magnitudes(n, 1.0, 8, 50.0, 23)
    h32 = (a.double() ** 2 * 2048.0).float().numpy()
    wd, hd = w.to(dev()), torch.from_numpy(h32).to(dev())
    sg, _ = gpu_rtn(wd)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    queue = gpu_refine_ws(wd, hd, sg, None, 0, 8, 8, 0, None)
    # the oracle parallelises over rows: on the single row, its first 65536 columns
    cols = n if m > 1 else 65536
    ref = oracle.refine(np.ascontiguousarray(wb[:, :cols]), h32[:cols], s_ref, None, 8, 8)
    compare_search(ref, queue[0][:, :cols // 16], queue[1][:, :cols // 2], f"per-SM queue {m}x{n} ({cols} columns)")
    ws = torch.full((16,), 0xAB, dtype=torch.uint8, device=dev())
    shared = gpu_refine_ws(wd, hd, sg, None, 0, 8, 8, 1, ws)
    assert shared_schedule_ran(ws)
    static = gpu_refine_ws(wd, hd, sg, None, 0, 8, 8, 7, None)
    for other in (shared, static):
        assert np.array_equal(other[0], queue[0]) and np.array_equal(other[1], queue[1])


def test_search_schedules_without_h():
    """h = NULL (the plain weight-MSE search of the h = 1 special case) under the three
    deals: the per-SM queue, the global counter and the static deal, against the oracle's
    unweighted search."""
    m, n, down, up = 4095, 4096, 8, 8
    w = wl.weight(m, n, 0.02, 24, device="cpu")
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    ref = oracle.refine(wb, None, s_ref, None, down, up)
    queue = gpu_refine_ws(wd, None, sg, None, 0, down, up, 0, None)
    compare_search(ref, *queue, f"per-SM queue {m}x{n} h = NULL")
    ws = torch.full((16,), 0xAB, dtype=torch.uint8, device=dev())
    shared = gpu_refine_ws(wd, None, sg, None, 0, down, up, 1, ws)
    assert shared_schedule_ran(ws)
    static = gpu_refine_ws(wd, None, sg, None, 0, down, up, 7, None)
    for other in (shared, static):
        assert np.array_equal(other[0], queue[0]) and np.array_equal(other[1], queue[1])


def test_shared_schedule_only_for_long_searches():
    """A short search (4096 x 4096 at k = 4 over every SM) keeps the static deal and leaves
    the workspace untouched; the bytes equal hscale_refine_scales'."""
    w = wl.weight(4096, 4096, 0.02, 22, device=dev())
    h = torch.from_numpy(oracle_h32(22, 4096)).to(dev())
    sg, _ = gpu_rtn(w)
    ws = torch.full((16,), 0xAB, dtype=torch.uint8, device=dev())
    codes, packed = gpu_refine_ws(w, h, sg, None, 0, 4, 4, 0, ws)
    assert not shared_schedule_ran(ws)
    ref = gpu_refine(w, h.cpu().numpy(), sg, None, 4, 4)
    assert np.array_equal(ref[0], codes) and np.array_equal(ref[1], packed)


def test_refine_is_deterministic():
    w = small_layer(3, 512, 1024)
    h32 = oracle_h32(3, 1024)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    a = gpu_refine(wd, h32, sg, None, 8, 8)
    b = gpu_refine(wd, h32, sg, None, 8, 8)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


# ------------------------------------------------------------------ 4over6 initialization (Algorithm 2)

def gpu_fourover6(w, sg):
    m, n = w.shape
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    hs.hscale_fourover6_codes(w, sg, codes)
    torch.cuda.synchronize()
    return codes.cpu().numpy()


def compare_init(ref_codes, near_tie, codes, label=""):
    """4over6 codes: bit-exact except where the two anchors' errors are a near-tie."""
    nt = near_tie.astype(bool)
    diff = codes != ref_codes
    bad = diff & ~nt
    assert not bad.any(), f"{label}: {bad.sum()} 4over6 code mismatches at {np.argwhere(bad)[:5]}"
    print(f"[parity] 4over6 {label}: groups={codes.size} anchor_near_ties={int(nt.sum())} "
          f"near_tie_mismatches={int((diff & nt).sum())}")
    return diff


@pytest.mark.parametrize("seed,m,n", [(0, 512, 1024), (1, 512, 1024), (2, 256, 4096),
                                      (5, 1, 16), (6, 3, 48), (7, 33, 16 * 33)])
def test_fourover6_codes_match_oracle(seed, m, n):
    w = wl.weight(m, n, 0.02, seed)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    ref, nt = oracle.fourover6_codes(bits(w), s_ref)
    codes = gpu_fourover6(wd, sg)
    diff = compare_init(ref, nt, codes, f"{m}x{n} seed {seed}")
    # both anchors are used on real-looking weights
    if m * n >= 512 * 1024:
        rtn = oracle.rtn_codes(bits(w), s_ref)
        assert 0.05 < float(np.mean(codes == rtn)) < 0.95
    assert not diff.all()


def test_fourover6_exact_ties_and_edge_groups():
    """s_g = 2^-7; groups whose elements sit on both anchors' grids (zero error at both
    codes: the tie keeps anchor 4), all-zero and -0 groups, tiny groups (both codes clip
    to 1), the saturated group that holds amax (both codes 126)."""
    rng = np.random.default_rng(21)
    m, n = 96, 256
    lad = oracle.e4m3_decode_table()[1:127]
    pairs = [(l6, 1.5 * l6) for l6 in lad if 1.5 * l6 in set(lad)]
    w = (rng.standard_t(4, size=(m, n)) * 0.05).astype(np.float32)
    both = np.array([0.0, 1.5, 3.0, 6.0])
    for i in range(m):
        l6, _ = pairs[i % len(pairs)]
        q = both[rng.integers(0, 4, size=16)] * rng.choice([-1, 1], size=16)
        q[rng.integers(0, 16)] = 6.0
        w[i, 16:32] = q * l6 * 2.0 ** -7
    w[0, 0] = 2688 * 2.0 ** -7            # tensor amax: s_g = 2^-7, code 126 at both anchors
    w[1, 32:48] = 0.0
    w[2, 48:64] = 1e-7                    # tiny: both anchors clip to code 1
    w[3, 64:80] = 0.0
    w[3, 70] = -3e-6
    wb = torch.from_numpy(w).to(torch.bfloat16)
    b = bits(wb)
    b[4, 32:48] = 0x8000                  # -0
    wb = from_bits(b)
    s_ref, _ = oracle.global_scale(b)
    assert s_ref == np.float32(2.0 ** -7)
    ref, nt = oracle.fourover6_codes(b, s_ref)
    wd = wb.to(dev())
    sg, _ = gpu_rtn(wd)
    codes = gpu_fourover6(wd, sg)
    compare_init(ref, nt, codes, "exact ties and edge groups")
    col = codes[:, 1]
    l6s = np.array([pairs[i % len(pairs)][0] for i in range(m)])
    expect = np.array([np.flatnonzero(lad == 1.5 * v)[0] + 1 for v in l6s])
    assert np.array_equal(col, expect), "an exact zero-error tie must keep anchor 4"
    assert codes[0, 0] == 126 and codes[1, 2] == 1 and codes[4, 2] == 1 and codes[2, 3] == 1
    # the fused pass decides the same anchors (window 0: its codes are the initial codes)
    fused, _ = gpu_refine_4over6(wd, None, sg, 0, 0)
    assert np.array_equal(fused, codes)


@pytest.mark.parametrize("down,up", [(4, 4), (9, 6), (0, 0)])
def test_fourover6_then_refine_matches_oracle(down, up):
    """Algorithm 2 end to end: 4over6 initial codes, then the search around them."""
    w = small_layer(4, 512, 1024)
    h32 = oracle_h32(4, 1024)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    init_ref, nt = oracle.fourover6_codes(bits(w), s_ref)
    init = torch.empty(512, 64, dtype=torch.uint8, device=dev())
    hs.hscale_fourover6_codes(wd, sg, init)
    diff = compare_init(init_ref, nt, init.cpu().numpy(), "512x1024 seed 4")
    codes, packed = gpu_refine(wd, h32, sg, init, down, up)
    ref = oracle.refine(bits(w), h32, s_ref, init_ref, down, up)
    ref["near_tie"] = ref["near_tie"] | diff.astype(np.uint8)
    compare_search(ref, codes, packed, f"4over6 init, window -{down}/+{up}")
    if (down, up) == (0, 0):
        assert np.array_equal(codes[~diff], init_ref[~diff])


def gpu_refine_4over6(w, h32, sg, down, up, ctas_per_sm=0):
    m, n = w.shape
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    packed = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
    h = None if h32 is None else torch.from_numpy(np.ascontiguousarray(h32, np.float32)).to(dev())
    hs.hscale_refine_scales_4over6(w, h, sg, down, up, codes, packed, ctas_per_sm)
    torch.cuda.synchronize()
    return codes.cpu().numpy(), packed.cpu().numpy()


@pytest.mark.parametrize("down,up,weighted,ctas", [(4, 4, True, 0), (9, 6, True, 4), (0, 0, True, 0),
                                                   (16, 16, True, 0), (4, 4, False, 0)])
def test_fused_fourover6_refine_matches_oracle(down, up, weighted, ctas):
    """Algorithm 2 in one pass: the 4over6 codes decided inside the search.  Against the
    oracle (its 4over6 codes, then its search), outside anchor and search near-ties; and
    bit for bit against the two-pass chain of the same library."""
    w = small_layer(4, 512, 1024)
    h32 = oracle_h32(4, 1024) if weighted else None
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    init_ref, nt = oracle.fourover6_codes(bits(w), s_ref)
    codes, packed = gpu_refine_4over6(wd, h32, sg, down, up, ctas)
    ref = oracle.refine(bits(w), h32, s_ref, init_ref, down, up)
    ref["near_tie"] = ref["near_tie"] | nt
    compare_search(ref, codes, packed, f"fused 4over6, window -{down}/+{up}, h={'x' if weighted else '1'}")
    if (down, up) == (0, 0):
        keep = ~nt.astype(bool)
        assert np.array_equal(codes[keep], init_ref[keep])
    init = torch.empty(512, 64, dtype=torch.uint8, device=dev())
    hs.hscale_fourover6_codes(wd, sg, init)
    codes2, packed2 = gpu_refine(wd, h32, sg, init, down, up)
    assert np.array_equal(codes, codes2) and np.array_equal(packed, packed2)


@pytest.mark.parametrize("seed,m,n", [(5, 1, 16), (6, 3, 48), (7, 33, 16 * 33), (8, 2, 16 * 200)])
def test_fused_fourover6_ragged_shapes(seed, m, n):
    """One row, ragged row chunks (groups per row not a multiple of the 32 lanes)."""
    w = wl.weight(m, n, 0.02, seed)
    h32 = oracle_h32(seed, n, tokens=256)
    wd = w.to(dev())
    sg, _ = gpu_rtn(wd)
    s_ref, _ = oracle.global_scale(bits(w))
    init_ref, nt = oracle.fourover6_codes(bits(w), s_ref)
    for down, up in ((4, 4), (0, 0)):
        codes, packed = gpu_refine_4over6(wd, h32, sg, down, up)
        ref = oracle.refine(bits(w), h32, s_ref, init_ref, down, up)
        ref["near_tie"] = ref["near_tie"] | nt
        compare_search(ref, codes, packed, f"fused 4over6 {m}x{n} window -{down}/+{up}")


# ------------------------------------------------------------------ 2-D views (column blocks)

@pytest.mark.parametrize("init", ["rtn", "given", "4over6"])
def test_strided_column_blocks_match_whole_matrix(init):
    """The search on column blocks of W (ragged last block, padded rows: ld_w > n), written
    into column blocks of the outputs, gives the whole-matrix call's bytes, and the
    oracle's on the block."""
    m, n, pad = 96, 16 * 136, 64
    w = small_layer(9, m, n)
    h32 = oracle_h32(9, n, tokens=512)
    buf = torch.zeros(m, n + pad, dtype=torch.bfloat16, device=dev())
    buf[:, :n] = w.to(dev())
    wd = buf[:, :n]
    sg, rtn = gpu_rtn(w.to(dev()))
    s_ref, _ = oracle.global_scale(bits(w))
    hd = torch.from_numpy(h32).to(dev())
    init_codes = rtn if init == "given" else None
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    packed = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
    if init == "4over6":
        hs.hscale_refine_scales_4over6(w.to(dev()), hd, sg, 4, 4, codes, packed)
    else:
        hs.hscale_refine_scales(w.to(dev()), hd, sg, init_codes, 4, 4, codes, packed)
    bc = torch.full((m, n // 16 + 8), 0xAB, dtype=torch.uint8, device=dev())
    bp = torch.full((m, n // 2 + 16), 0xAB, dtype=torch.uint8, device=dev())
    for c0, c1, ctas in ((0, 512, 4), (512, 1536, 2), (1536, n, 0)):
        g0, g1 = c0 // 16, c1 // 16
        hs.hscale_refine_scales_strided(wd[:, c0:c1], hd[c0:c1], sg,
                                        None if init_codes is None else init_codes[:, g0:g1],
                                        init == "4over6", 4, 4, bc[:, g0:g1], bp[:, c0 // 2:c1 // 2], ctas)
    torch.cuda.synchronize()
    assert torch.equal(bc[:, :n // 16], codes) and torch.equal(bp[:, :n // 2], packed)
    assert bool((bc[:, n // 16:] == 0xAB).all()) and bool((bp[:, n // 2:] == 0xAB).all()), "wrote past the view"
    # the middle block against the oracle on that block alone
    c0, c1 = 512, 1536
    wb = bits(w)[:, c0:c1]
    if init == "4over6":
        i_ref, nt = oracle.fourover6_codes(bits(w), s_ref)
        i_ref, nt = i_ref[:, c0 // 16:c1 // 16], nt[:, c0 // 16:c1 // 16]
    else:
        i_ref, nt = oracle.rtn_codes(wb, s_ref), np.zeros((m, (c1 - c0) // 16), np.uint8)
    ref = oracle.refine(wb, h32[c0:c1], s_ref, i_ref, 4, 4)
    ref["near_tie"] = ref["near_tie"] | nt
    compare_search(ref, bc[:, c0 // 16:c1 // 16].cpu().numpy(), bp[:, c0 // 2:c1 // 2].cpu().numpy(),
                   f"strided block {c0}:{c1}, init {init}")


def test_strided_row_slice_and_no_packed_output():
    """A row slice (one row of a larger matrix) and a view without nibbles."""
    m, n = 40, 1024
    w = small_layer(10, m, n).to(dev())
    h32 = oracle_h32(10, n, tokens=256)
    hd = torch.from_numpy(h32).to(dev())
    sg, _ = gpu_rtn(w)
    codes, packed = gpu_refine(w, h32, sg, None, 9, 6)
    c1 = torch.empty(1, n // 16, dtype=torch.uint8, device=dev())
    hs.hscale_refine_scales_strided(w[17:18], hd, sg, None, False, 9, 6, c1, None, 0)
    c2 = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    hs.hscale_refine_scales_strided(w, hd, sg, None, False, 9, 6, c2, None, 3)
    torch.cuda.synchronize()
    assert np.array_equal(c1.cpu().numpy()[0], codes[17])
    assert np.array_equal(c2.cpu().numpy(), codes)


# ------------------------------------------------------------------ the fast path's margin band

@pytest.mark.parametrize("down,up", [(4, 4), (9, 6)])
def test_search_exact_in_the_margin_band(down, up):
    """2,097,152 groups against the oracle, with the groups whose best and runner-up errors
    differ by 1e-6 to 1e-3 relative counted separately: there the fast scores cannot
    decide and the exact rescoring must (outside the 1e-6 near-tie band every code and
    nibble must be the oracle's)."""
    m, n = 4096, 8192
    w = wl.weight(m, n, 0.02, 4242, device=dev())
    h32 = oracle_h32(4242, n, tokens=1024)
    sg, _ = gpu_rtn(w)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    assert sg.cpu().numpy()[0] == s_ref
    codes, packed = gpu_refine(w, h32, sg, None, down, up)
    ref = oracle.refine(wb, h32, s_ref, None, down, up)
    compare_search(ref, codes, packed, f"2M groups -{down}/+{up}")
    with np.errstate(divide="ignore", invalid="ignore"):
        gap = (ref["e_second"] - ref["e_best"]) / ref["e_second"]
    band = (gap > 1e-6) & (gap < 1e-3)
    assert band.sum() >= 100, f"only {band.sum()} groups in the margin band"
    assert np.array_equal(codes[band], ref["codes"][band])
    rows = np.nonzero(band.any(axis=1))[0]
    for r in rows[:256]:
        cols = np.nonzero(band[r])[0]
        for c in cols:
            assert np.array_equal(packed[r, 8 * c:8 * c + 8], ref["packed"][r, 8 * c:8 * c + 8])
    print(f"[parity] margin band -{down}/+{up}: {int(band.sum())} groups with 1e-6 < gap < 1e-3, all exact")


# ------------------------------------------------------------------ offsets past 2^31 elements

def test_search_and_hessian_beyond_2_31_elements():
    """W and X of 65600 x 32768 bf16 (2.15e9 elements, 4.3 GB each): element offsets past
    2^31.  s_g against an exact maximum on the device; RTN codes, searched codes and nibbles
    of rows on both sides of the 2^31 boundary against the oracle; h of sampled channels
    against the oracle."""
    m, n = 65600, 32768
    assert m * n > 2 ** 31
    W = torch.empty(m, n, dtype=torch.bfloat16, device=dev())
    step = 4096
    for r0 in range(0, m, step):
        W[r0:r0 + step] = wl.weight(min(step, m - r0), n, 0.02, 900 + r0 // step, device=dev())
    sg, rtn = gpu_rtn(W)
    amax_bits = int((W.view(torch.int16) & 0x7FFF).max().item())
    amax = float(np.array([amax_bits << 16], dtype=np.uint32).view(np.float32)[0])
    s_ref = np.float32(amax / 2688.0)
    assert sg.cpu().numpy()[0] == s_ref
    h32 = (wl.channel_magnitudes(n, 1.0, 32, 50.0, 77).numpy().astype(np.float64) ** 2 * 1000.0).astype(np.float32)
    hd = torch.from_numpy(h32).to(dev())
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    packed = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
    hs.hscale_refine_scales(W, hd, sg, None, 4, 4, codes, packed)
    torch.cuda.synchronize()
    rows = np.array([0, 65535, 65536, 65537, m - 2, m - 1])  # row 65536 starts at element 2^31
    wb = bits(W[torch.from_numpy(rows).to(dev())])
    assert np.array_equal(rtn[torch.from_numpy(rows).to(dev())].cpu().numpy(), oracle.rtn_codes(wb, s_ref))
    ref = oracle.refine(wb, h32, s_ref, None, 4, 4)
    compare_search(ref, codes[torch.from_numpy(rows).to(dev())].cpu().numpy(),
                   packed[torch.from_numpy(rows).to(dev())].cpu().numpy(), "rows across the 2^31 element offset")
    del W, codes, packed, rtn
    torch.cuda.empty_cache()
    X = torch.empty(m, n, dtype=torch.bfloat16, device=dev())
    a = wl.channel_magnitudes(n, 1.0, 32, 50.0, 78, device=dev())
    for r0 in range(0, m, step):
        wl.activation_chunk(min(step, m - r0), a, 78, r0 // step, out=X[r0:r0 + step])
    h = torch.zeros(n, device=dev())
    hs.hscale_hessian_diag_accumulate(X, h)
    torch.cuda.synchronize()
    cols = torch.tensor([0, 1, 4095, 16384, n - 2, n - 1], device=dev())
    href = np.zeros(cols.numel())
    oracle.hessian_accumulate(bits(X[:, cols].contiguous()), href)
    err = assert_h_close(h[cols].cpu().numpy(), href)
    print(f"[parity] 65600 x 32768 (2.15e9 elements): h max rel err {err:.3e} on sampled channels")
    del X


# ------------------------------------------------------------------ output error (Eq. 3)

def oracle_codes_packed(wb, h32, s_ref, window):
    """Codes and nibbles from the CPU oracle (RTN for window None, else the search)."""
    if window is None:
        codes = oracle.rtn_codes(wb, s_ref)
        return codes, oracle.pack(wb, s_ref, codes)
    out = oracle.refine(wb, h32, s_ref, None, *window)
    return out["codes"], out["packed"]


def gpu_residual(wd, sg, codes, packed):
    m, n = wd.shape
    dw2 = torch.full((m, hs.residual_ld(n)), float("nan"), dtype=torch.bfloat16, device=dev())
    hs.hscale_dequant_residual(wd, sg, torch.from_numpy(codes).to(dev()), torch.from_numpy(packed).to(dev()), dw2)
    torch.cuda.synchronize()
    return dw2


@pytest.mark.parametrize("m,n,window", [(64, 1024, None), (48, 80, (4, 4)), (3, 16, (9, 6))])
def test_dequant_residual_matches_oracle(m, n, window):
    """hi + lo equals the oracle's dW = W - W_hat within a relative 2^-17 (one fp32 rounding
    of dW, then the bf16 split), and the padding columns are zero."""
    w = wl.weight(m, n, 0.02, 40 + n)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    codes, packed = oracle_codes_packed(wb, oracle_h32(9, n), s_ref, window)
    wd = w.to(dev())
    sg = torch.tensor([s_ref], dtype=torch.float32, device=dev())
    dw2 = gpu_residual(wd, sg, codes, packed).float().cpu().double().numpy()
    n_pad = hs.residual_ld(n) // 2
    hi, lo = dw2[:, :n], dw2[:, n_pad:n_pad + n]
    ref = oracle.dequant_residual(wb, s_ref, codes, packed)
    err = np.abs(hi + lo - ref)
    assert np.all(err <= 2.0 ** -17 * np.abs(ref) + 1e-45), f"max rel {np.max(err / (np.abs(ref) + 1e-300)):.3e}"
    assert np.all(dw2[:, n:n_pad] == 0) and np.all(dw2[:, n_pad + n:] == 0)


def gpu_output_error(xd, dw2, m):
    out = torch.zeros(1, dtype=torch.float64, device=dev())
    ws = torch.empty(max(8, hs.hscale_output_error_workspace_bytes(xd.shape[0], m)), dtype=torch.uint8, device=dev())
    hs.hscale_output_error(xd, dw2, m, out, ws)
    torch.cuda.synchronize()
    return float(out.item())


OUTPUT_ERROR_RTOL = 1e-4


@pytest.mark.parametrize("tokens,m,n", [(128, 256, 64), (300, 300, 80), (512, 512, 1024), (1000, 40, 4096),
                                        (256, 256, 14336), (2600, 2048, 64)])
def test_output_error_matches_oracle(tokens, m, n):
    """||X dW^T||_F^2 on the tensor cores against the fp64 oracle: ragged tokens, outputs
    and K (n not a multiple of 64), one tile and many, down_proj's width (K = 28672,
    14 accumulation segments; one fp32 accumulation over the whole K would drift about 2x
    past the bound there), and more tiles than SMs (21 x 8 = 168 tiles of 128 x 256: CTAs
    with two tiles, and tile-order groups of 8, 8 and 5 rows of tiles).  Tolerance: the bf16
    split of dW (2^-17 relative per element) plus fp32 accumulation over 2048-long
    segments."""
    w = wl.weight(m, n, 0.02, 50 + n)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    codes, packed = oracle_codes_packed(wb, None, s_ref, None)
    a = wl.channel_magnitudes(n, 1.0, 4, 50.0, 7)
    x = wl.activation_chunk(tokens, a, 7, n)
    ref = oracle.output_error(bits_to_f64(x), oracle.dequant_residual(wb, s_ref, codes, packed))
    wd = w.to(dev())
    sg = torch.tensor([s_ref], dtype=torch.float32, device=dev())
    dw2 = gpu_residual(wd, sg, codes, packed)
    got = gpu_output_error(x.to(dev()), dw2, m)
    print(f"[parity] output error {tokens}x{n} -> {m}: gpu {got:.9e} oracle {ref:.9e} rel {abs(got - ref) / ref:.2e}")
    assert abs(got - ref) <= OUTPUT_ERROR_RTOL * ref


def test_output_error_strided_tokens_and_accumulation():
    """x as a strided row slice of a wider buffer, two chunks accumulated into one sum."""
    m, n = 256, 512
    w = wl.weight(m, n, 0.02, 61)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    codes, packed = oracle_codes_packed(wb, None, s_ref, None)
    g = torch.Generator().manual_seed(62)
    xf = (torch.randn(384, n + 64, generator=g)).to(torch.bfloat16)
    dw = oracle.dequant_residual(wb, s_ref, codes, packed)
    ref = oracle.output_error(bits_to_f64(xf[:, :n].contiguous()), dw)
    dw2 = gpu_residual(w.to(dev()), torch.tensor([s_ref], dtype=torch.float32, device=dev()), codes, packed)
    xd = xf.to(dev())
    out = torch.zeros(1, dtype=torch.float64, device=dev())
    ws = torch.empty(hs.hscale_output_error_workspace_bytes(384, m), dtype=torch.uint8, device=dev())
    hs.hscale_output_error(xd[:200, :n], dw2, m, out, ws)
    hs.hscale_output_error(xd[200:, :n], dw2, m, out, ws)
    torch.cuda.synchronize()
    assert abs(out.item() - ref) <= OUTPUT_ERROR_RTOL * ref


def bits_to_f64(x):
    return x.float().double().numpy()


def test_full_size_output_error_q_proj():
    """The 4096 x 4096 q_proj layer at full width: RTN and searched (k = 4) quantizations
    from the oracle, ||X dW^T||^2 over 512 calibration tokens on both sides."""
    W = wl.WORKLOADS["llama8b-q_proj"]
    L = W.layers[0]
    m, n = L.out_features, L.in_features
    w = wl.weight(m, n, W.sigma_w, W.seed)
    wb = bits(w)
    s_ref, _ = oracle.global_scale(wb)
    a = wl.channel_magnitudes(n, W.sigma_a, W.outlier_channels, W.outlier_channel_mult, W.seed)
    x = wl.activation_chunk(2048, a, W.seed, 0)
    h = np.zeros(n)
    oracle.hessian_accumulate(bits(x), h)
    xe = x[:512]
    wd = w.to(dev())
    sg = torch.tensor([s_ref], dtype=torch.float32, device=dev())
    got = {}
    for name, window in (("rtn", None), ("hscale", (4, 4))):
        codes, packed = oracle_codes_packed(wb, h.astype(np.float32), s_ref, window)
        ref = oracle.output_error(bits_to_f64(xe), oracle.dequant_residual(wb, s_ref, codes, packed))
        g = gpu_output_error(xe.to(dev()), gpu_residual(wd, sg, codes, packed), m)
        assert abs(g - ref) <= OUTPUT_ERROR_RTOL * ref, (name, g, ref)
        got[name] = g
    print(f"[parity] q_proj output error over 512 tokens: rtn {got['rtn']:.6e} hscale {got['hscale']:.6e} "
          f"reduction {1 - got['hscale'] / got['rtn']:.1%}")


# ------------------------------------------------------------------ full-size workloads

BLOCK = 1024  # channels per column block of `bench.py --col-block 1024`


def full_size_check(name, sample_rows, layer_index=0, windows=None, fourover6=False):
    """A workload at its full size in the launch configuration bench.py times: h of every
    input space over every streamed chunk (all columns, against the oracle fed the same
    chunks), s_g and RTN codes over every whole matrix, and the search with packing on a
    seeded sample of rows of every matrix, for every window of the workload.  With
    ``fourover6`` the search starts from Algorithm 2's codes, checked over every whole
    matrix first."""
    W = wl.WORKLOADS[name]
    seed = W.layer_seed(layer_index)
    h_ref = {}
    for space, n in W.input_spaces():
        chunk = W.chunk_tokens[n]
        a = wl.channel_magnitudes(n, W.sigma_a, W.outlier_channels, W.outlier_channel_mult,
                                  wl.chunk_seed(seed, space, 0) & 0xFFFFFFFF, device=dev())
        h = torch.zeros(n, device=dev())
        href = np.zeros(n)
        for c in range(W.tokens // chunk):
            x = wl.activation_chunk(chunk, a, wl.chunk_seed(seed, space, 1) & 0xFFFFFFFF, c)
            hs.hscale_hessian_diag_accumulate(x, h)
            oracle.hessian_accumulate(bits(x), href)
            del x
        torch.cuda.synchronize()
        err = assert_h_close(h.cpu().numpy(), href)
        print(f"[parity] {name} {space}: h over {W.tokens} tokens x {n}: max rel err {err:.3e}")
        # the column-blocked calls of `bench.py --col-block 1024`: every token of 1024
        # channels per block, in launches of about a chunk's bytes
        x_all = torch.empty(W.tokens, n, dtype=torch.bfloat16, device=dev())
        for c in range(W.tokens // chunk):
            wl.activation_chunk(chunk, a, wl.chunk_seed(seed, space, 1) & 0xFFFFFFFF, c,
                                out=x_all[c * chunk:(c + 1) * chunk])
        hb = torch.zeros(n, device=dev())
        for c0 in range(0, n, BLOCK):
            c1 = min(n, c0 + BLOCK)
            rows = chunk if c1 - c0 == n else max(chunk, chunk * n // (c1 - c0))
            for t0 in range(0, W.tokens, rows):
                hs.hscale_hessian_diag_accumulate(x_all[t0:t0 + rows, c0:c1], hb[c0:c1])
        torch.cuda.synchronize()
        del x_all
        err = assert_h_close(hb.cpu().numpy(), href)
        print(f"[parity] {name} {space}: h in {BLOCK}-channel column blocks: max rel err {err:.3e}")
        h_ref[space] = href.astype(np.float32)
    for L in W.layers:
        m, n = L.out_features, L.in_features
        w = wl.weight(m, n, W.sigma_w, wl.chunk_seed(seed, L.name, 0) & 0xFFFFFFFF, device=dev())
        sg, codes = gpu_rtn(w)
        wb = bits(w)
        s_ref, _ = oracle.global_scale(wb)
        assert sg.cpu().numpy()[0] == s_ref
        assert np.array_equal(codes.cpu().numpy(), oracle.rtn_codes(wb, s_ref))
        rows = np.sort(np.random.default_rng(seed).choice(m, size=min(sample_rows, m), replace=False))
        init = init_ref = None
        exclude = np.zeros((rows.size, n // 16), np.uint8)
        if fourover6:
            init_ref, nt = oracle.fourover6_codes(wb, s_ref)
            init = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
            hs.hscale_fourover6_codes(w, sg, init)
            diff = compare_init(init_ref, nt, init.cpu().numpy(), f"{name} {L.name} {m}x{n}")
            init_ref, exclude = init_ref[rows], diff[rows].astype(np.uint8)
        for down, up in (windows or [(k, k) for k in W.window]):
            codes_g, packed_g = gpu_refine(w, h_ref[L.input_space], sg, init, down, up)
            ref = oracle.refine(wb[rows], h_ref[L.input_space], s_ref, init_ref, down, up)
            ref["near_tie"] = ref["near_tie"] | exclude
            compare_search(ref, codes_g[rows], packed_g[rows],
                           f"{name} {L.name} {m}x{n} window -{down}/+{up} ({rows.size} sampled rows)")
            if fourover6:
                # the one-pass form, at the launch shape the bench times it with (4 CTAs/SM)
                codes_f, packed_f = gpu_refine_4over6(w, h_ref[L.input_space], sg, down, up, 4)
                assert np.array_equal(codes_f, codes_g) and np.array_equal(packed_f, packed_g)
            # the entry point bench.py calls (work-shared schedule where the search is long),
            # alone and at 4 CTAs per SM
            hd32 = torch.from_numpy(h_ref[L.input_space]).to(dev())
            ws = torch.zeros(hs.hscale_refine_workspace_bytes(), dtype=torch.uint8, device=dev())
            for ctas in (0, 4):
                codes_w, packed_w = gpu_refine_ws(w, hd32, sg, init, 0, down, up, ctas, ws)
                assert np.array_equal(codes_w, codes_g) and np.array_equal(packed_w, packed_g)
            # the column-blocked searches of `bench.py --col-block 1024` (views, 4 CTAs/SM
            # but the last block)
            hd = torch.from_numpy(h_ref[L.input_space]).to(dev())
            bc = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
            bp = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
            for c0 in range(0, n, BLOCK):
                c1 = min(n, c0 + BLOCK)
                g0, g1 = c0 // 16, c1 // 16
                hs.hscale_refine_scales_strided(w[:, c0:c1], hd[c0:c1], sg, None if init is None else init[:, g0:g1],
                                                False, down, up, bc[:, g0:g1], bp[:, c0 // 2:c1 // 2],
                                                4 if c1 < n else 0)
            torch.cuda.synchronize()
            assert np.array_equal(bc.cpu().numpy(), codes_g) and np.array_equal(bp.cpu().numpy(), packed_g)
        del w


def test_full_size_llama8b_q_proj():
    full_size_check("llama8b-q_proj", sample_rows=512)


def test_full_size_q_proj_paper_window_and_full_grid():
    """The paper's default window (D = 9, U = 6, K = 16) and the whole E4M3 ladder."""
    full_size_check("llama8b-q_proj", sample_rows=64, windows=[(9, 6), (125, 125)])


def test_full_size_q_proj_fourover6_init():
    """Algorithm 2 at full size: 4over6 codes over the whole matrix, then the search
    around them with the paper's default window."""
    full_size_check("llama8b-q_proj", sample_rows=128, windows=[(9, 6), (4, 4)], fourover6=True)


def test_full_size_mlp_down_proj():
    full_size_check("mlp-down_proj", sample_rows=128)


def test_full_size_llama8b_decoder_layer():
    full_size_check("llama8b-decoder", sample_rows=64, layer_index=7)


def test_full_size_llama70b_mlp_window_sweep():
    full_size_check("llama70b-mlp", sample_rows=24)
