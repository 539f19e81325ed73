"""Kernel-level GPU tests: the tcgen05 dense products (all operand layouts, ragged tails,
fused epilogues, split-K accumulation) and the attention kernels against plain PyTorch
fp32 computations on the same rounded inputs."""
import math

import pytest
import torch
import torch.nn.functional as F

pytestmark = pytest.mark.gpu

jg = pytest.importorskip("paper_2607_17572_gb300")


def _rel(a, b):
    return (torch.linalg.vector_norm((a.double() - b.double())) / torch.linalg.vector_norm(b.double())).item()


def _desc(M, N, K, A, lda, a_mn, B, ldb, b_mn, dt, C, ldc, c_dt, epi=0, **kw):
    d = jg.GemmDesc()
    d.M, d.N, d.K = M, N, K
    d.A, d.lda, d.a_mn, d.a_dtype = A.data_ptr(), lda, int(a_mn), dt
    d.B, d.ldb, d.b_mn, d.b_dtype = B.data_ptr(), ldb, int(b_mn), dt
    d.epi = epi
    d.C, d.ldc, d.c_dtype = C.data_ptr(), ldc, c_dt
    d.bias_dtype = dt
    d.rows_per_seq = 1
    for k, v in kw.items():
        setattr(d, k, v.data_ptr() if isinstance(v, torch.Tensor) else v)
    return d


SHAPES = [(256, 128, 128), (300, 200, 192), (128, 64, 64), (1000, 768, 768), (5328, 2304, 768), (777, 320, 1000)]


@pytest.mark.parametrize("tile_n", [0, 64, 128, 256])
@pytest.mark.parametrize("a_mn,b_mn", [(False, False), (False, True), (True, True), (True, False)])
@pytest.mark.parametrize("M,N,K", [(300, 600, 192), (1000, 768, 520)])
def test_tcgen05_tile_widths(M, N, K, a_mn, b_mn, tile_n):
    """Every tile width on every operand layout, with a ragged last column tile, for a
    plain store, a biased bf16 store and a split-K accumulation."""
    torch.manual_seed(M + N + K + tile_n)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()
    B = (torch.randn(N, K, device=dev) / math.sqrt(K)).bfloat16()
    As = A.t().contiguous() if a_mn else A
    Bs = B.t().contiguous() if b_mn else B
    lda, ldb = (M if a_mn else K), (N if b_mn else K)
    ref = A.float() @ B.float().t()
    C = torch.full((M, N), float("nan"), device=dev)
    jg.test_gemm(_desc(M, N, K, As, lda, a_mn, Bs, ldb, b_mn, jg.DTYPE_BF16, C, N, jg.DTYPE_F32, tile_n=tile_n))
    bias = torch.randn(N, device=dev).bfloat16()
    Cb = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
    jg.test_gemm(_desc(M, N, K, As, lda, a_mn, Bs, ldb, b_mn, jg.DTYPE_BF16, Cb, N, jg.DTYPE_BF16, bias=bias,
                       tile_n=tile_n))
    G0 = torch.randn(M, N, device=dev)
    G = G0.clone()
    jg.test_gemm(_desc(M, N, K, As, lda, a_mn, Bs, ldb, b_mn, jg.DTYPE_BF16, G, N, jg.DTYPE_F32, epi=4, split_k=3,
                       tile_n=tile_n))
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    assert _rel(C, ref) < 1e-5
    assert _rel(Cb.float(), ref + bias.float()) < 5e-3
    assert _rel(G, G0 + ref) < 1e-5
    if not a_mn and b_mn:
        # the multiplier epilogue of the input-gradient products (every chunk of a warp's
        # tile at once up to 128 columns, a two-slot ring per warp at 256), bf16 output into
        # a wider buffer
        X = torch.rand(M, N, device=dev).bfloat16()
        O = torch.full((M, N + 8), 3.0, device=dev, dtype=torch.bfloat16)
        jg.test_gemm(_desc(M, N, K, As, lda, a_mn, Bs, ldb, b_mn, jg.DTYPE_BF16, O, N + 8, jg.DTYPE_BF16, epi=3,
                           aux=X, ld_aux=N, tile_n=tile_n))
        torch.cuda.synchronize()
        assert jg.device_status() == 0
        assert _rel(O[:, :N].float(), ref * X.float()) < 5e-3
        assert torch.all(O[:, N:] == 3.0)


@pytest.mark.parametrize("a_mn,b_mn", [(False, False), (False, True), (True, True), (True, False)])
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_tcgen05_gemm_layouts(M, N, K, a_mn, b_mn):
    torch.manual_seed(M * 7 + N * 3 + K)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()       # logical A[m, k]
    B = torch.randn(N, K, device=dev).bfloat16()       # logical B[n, k]
    As = A.t().contiguous() if a_mn else A
    Bs = B.t().contiguous() if b_mn else B
    lda = M if a_mn else K
    ldb = N if b_mn else K
    C = torch.full((M, N), float("nan"), device=dev)
    jg.test_gemm(_desc(M, N, K, As, lda, a_mn, Bs, ldb, b_mn, jg.DTYPE_BF16, C, N, jg.DTYPE_F32))
    ref = A.float() @ B.float().t()
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    assert _rel(C, ref) < 1e-5


@pytest.mark.parametrize("M,N,K,a_mn,b_mn,epi", [
    (56832, 16, 768, 0, 0, 0),     # stacked modulation forward: mod^T = W_mod silu(c)^T
    (768, 16, 56832, 1, 0, 4),     # d silu(c)^T = W_mod^T dmod^T, split over K
    (56832, 768, 16, 1, 1, 4),     # dW_mod += dmod^T silu(c), K = 16 rows
    (100, 30, 24, 0, 0, 0),        # every extent below one tile
    (64, 8, 40, 1, 0, 4)])
def test_tcgen05_small_extents_and_transposed_output(M, N, K, a_mn, b_mn, epi):
    """Tiles larger than the tensors (TMA zero-fills the outside), an output written
    transposed (C[n, m]) and a bias indexed by m."""
    torch.manual_seed(M + N + K)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()
    B = torch.randn(N, K, device=dev).bfloat16()
    As = A.t().contiguous() if a_mn else A
    Bs = B.t().contiguous() if b_mn else B
    bias = torch.randn(M, device=dev).bfloat16()
    C0 = torch.randn(N, M, device=dev)
    C = C0.clone()
    kw = dict(c_trans=1)
    if epi == 0:
        kw.update(bias=bias, bias_m=1)
    jg.test_gemm(_desc(M, N, K, As, M if a_mn else K, a_mn, Bs, N if b_mn else K, b_mn, jg.DTYPE_BF16, C, M,
                       jg.DTYPE_F32, epi=epi, **kw))
    ref = (A.float() @ B.float().t()).t()
    ref = ref + bias.float()[None, :] if epi == 0 else C0 + ref
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    assert _rel(C, ref) < 1e-5


@pytest.mark.parametrize("M,N,K", [(300, 200, 192), (2048, 768, 768)])
def test_gemm_epilogues(M, N, K):
    torch.manual_seed(1)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()
    B = (torch.randn(N, K, device=dev) / math.sqrt(K)).bfloat16()
    bias = torch.randn(N, device=dev).bfloat16()
    acc = A.float() @ B.float().t()
    # GELU: gelu'(u) and gelu(u) of u = acc + bias
    DU = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
    GU = torch.empty_like(DU)
    jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, DU, N, jg.DTYPE_BF16, epi=1, bias=bias, C2=GU,
                       ldc2=N))
    u = (acc + bias.float()).requires_grad_()
    gelu_u = F.gelu(u, approximate="tanh")
    gelu_u.sum().backward()
    assert _rel(GU.float(), gelu_u.detach()) < 5e-3
    assert _rel(DU.float(), u.grad) < 5e-3
    # GELU alone (no derivative output: the forwards that keep nothing), into a wider buffer
    GW = torch.full((M, N + 8), 7.0, device=dev, dtype=torch.bfloat16)
    d = _desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, DU, N, jg.DTYPE_BF16, epi=1, bias=bias, C2=GW, ldc2=N + 8)
    d.C = None
    jg.test_gemm(d)
    torch.cuda.synchronize()
    assert torch.equal(GW[:, :N], GU) and torch.all(GW[:, N:] == 7.0)
    u = u.detach()
    # gated residual: y = acc + bias; h_out = h_in + gate[seq] * y
    rows = 37
    gate = torch.randn((M + rows - 1) // rows, N + 8, device=dev)
    hin = torch.randn(M, N, device=dev)
    Y = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
    H = torch.empty(M, N, device=dev)
    jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, Y, N, jg.DTYPE_BF16, epi=2, bias=bias, C2=H, ldc2=N,
                       aux=hin, ld_aux=N, gate=gate, gate_stride=N + 8, rows_per_seq=rows))
    g = gate[torch.arange(M, device=dev) // rows, :N]
    assert _rel(H, hin + g * u) < 1e-5
    # multiply by a saved factor (the GELU derivative in the MLP backward): acc * aux
    aux = torch.randn(M, N, device=dev).bfloat16()
    O = torch.empty(M, N, device=dev, dtype=torch.bfloat16)
    jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, O, N, jg.DTYPE_BF16, epi=3, aux=aux, ld_aux=N))
    assert _rel(O.float(), acc * aux.float()) < 5e-3
    torch.cuda.synchronize()
    assert jg.device_status() == 0


@pytest.mark.parametrize("tile_n", [0, 64, 128])
@pytest.mark.parametrize("M,N,K,rows", [(300, 100, 192, 37), (1000, 768, 256, 333), (129, 264, 64, 129)])
def test_gated_residual_epilogue(M, N, K, rows, tile_n):
    """y = X W^T + b to C (bf16) and h_out = h_in + gate[seq(m)] * y (f32) to C2, with the
    residual input TMA-loaded per 32 x 32 chunk: ragged rows and columns, sequences that
    start inside a tile, outputs inside wider buffers."""
    torch.manual_seed(M + N + K + tile_n)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()
    B = (torch.randn(N, K, device=dev) / math.sqrt(K)).bfloat16()
    bias = torch.randn(N, device=dev).bfloat16()
    gate = torch.randn((M + rows - 1) // rows, N + 4, device=dev)
    hin = torch.randn(M, N + 4, device=dev)
    Y = torch.full((M, N + 8), 5.0, device=dev, dtype=torch.bfloat16)
    H = torch.full((M, N + 4), 7.0, device=dev)
    jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, Y, N + 8, jg.DTYPE_BF16, epi=2, bias=bias, C2=H,
                       ldc2=N + 4, aux=hin, ld_aux=N + 4, gate=gate, gate_stride=N + 4, rows_per_seq=rows,
                       tile_n=tile_n))
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    y = A.float() @ B.float().t() + bias.float()
    g = gate[torch.arange(M, device=dev) // rows, :N]
    assert _rel(Y[:, :N].float(), y) < 5e-3
    assert _rel(H[:, :N], hin[:, :N] + g * y) < 1e-5
    assert torch.all(Y[:, N:] == 5.0) and torch.all(H[:, N:] == 7.0)


@pytest.mark.parametrize("split", [0, 1, 3])
def test_gemm_accumulate_weight_gradient(split):
    """dW += dY^T X with both operands MN-major, accumulated into an existing f32 buffer."""
    torch.manual_seed(2)
    dev = "cuda"
    M, N, K = 5328, 768, 2304        # tokens, in, out: dW [out, in] += dY[tok, out]^T X[tok, in]
    X = torch.randn(M, N, device=dev).bfloat16()
    dY = torch.randn(M, K, device=dev).bfloat16()
    G0 = torch.randn(K, N, device=dev)
    G = G0.clone()
    jg.test_gemm(_desc(K, N, M, dY, K, 1, X, N, 1, jg.DTYPE_BF16, G, N, jg.DTYPE_F32, epi=4, split_k=split))
    ref = G0 + dY.float().t() @ X.float()
    torch.cuda.synchronize()
    assert _rel(G, ref) < 1e-5


@pytest.mark.parametrize("M,N,K", [(300, 200, 192), (77, 1000, 320), (4099, 384, 512)])
def test_gemm_outputs_inside_wider_buffers(M, N, K):
    """Outputs written as a column block of a wider buffer (row pitch > N, 16-byte aligned
    offset), the multiplier read likewise, bf16 stores with a bias and a ragged last column
    chunk, and an accumulation into a sub-block: the shared-memory-staged epilogues."""
    torch.manual_seed(M + 5 * N + K)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()
    B = (torch.randn(N, K, device=dev) / math.sqrt(K)).bfloat16()
    bias = torch.randn(N, device=dev).bfloat16()
    acc = A.float() @ B.float().t()
    pad, off = 72, 24                      # columns before and after the block (16-byte multiples)
    ld = off + N + pad
    # bf16 store with bias into columns [off, off + N) of a [M, ld] buffer
    big = torch.full((M, ld), 7.0, device=dev, dtype=torch.bfloat16)
    view = big[:, off:]
    jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, view, ld, jg.DTYPE_BF16, bias=bias))
    torch.cuda.synchronize()
    assert _rel(big[:, off:off + N].float(), acc + bias.float()) < 5e-3
    assert (big[:, :off] == 7.0).all() and (big[:, off + N:] == 7.0).all()
    # multiply by a factor that is itself a column block of a wider buffer
    auxbig = torch.randn(M, ld, device=dev).bfloat16()
    out = torch.full((M, ld), 7.0, device=dev, dtype=torch.bfloat16)
    jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, out[:, off:], ld, jg.DTYPE_BF16, epi=3,
                       aux=auxbig[:, off:], ld_aux=ld))
    torch.cuda.synchronize()
    assert _rel(out[:, off:off + N].float(), acc * auxbig[:, off:off + N].float()) < 5e-3
    assert (out[:, :off] == 7.0).all() and (out[:, off + N:] == 7.0).all()
    # f32 accumulation into a sub-block, with and without split-K
    for split in (1, 4):
        G0 = torch.randn(M, ld, device=dev)
        G = G0.clone()
        jg.test_gemm(_desc(M, N, K, A, K, 0, B, K, 0, jg.DTYPE_BF16, G[:, off:], ld, jg.DTYPE_F32, epi=4,
                           split_k=split))
        torch.cuda.synchronize()
        assert _rel(G[:, off:off + N], G0[:, off:off + N] + acc) < 1e-5
        assert torch.equal(G[:, :off], G0[:, :off]) and torch.equal(G[:, off + N:], G0[:, off + N:])
    assert jg.device_status() == 0


@pytest.mark.parametrize("M,N,K,a_mn,b_mn", [(16, 4608, 768, 0, 0), (16, 768, 56832, 0, 1), (56832, 768, 16, 1, 1),
                                              (40, 70, 33, 0, 0), (7, 9, 11, 1, 0)])
def test_simt_gemm_f32(M, N, K, a_mn, b_mn):
    torch.manual_seed(3)
    dev = "cuda"
    A = torch.randn(M, K, device=dev)
    B = torch.randn(N, K, device=dev)
    As = A.t().contiguous() if a_mn else A
    Bs = B.t().contiguous() if b_mn else B
    C0 = torch.randn(M, N, device=dev)
    C = C0.clone()
    jg.test_gemm(_desc(M, N, K, As, M if a_mn else K, a_mn, Bs, N if b_mn else K, b_mn, jg.DTYPE_F32, C, N,
                       jg.DTYPE_F32, epi=4))
    torch.cuda.synchronize()
    assert _rel(C, C0 + A.double().float() @ B.t()) < 1e-5


def _attn_ref(qkv, B, N, H, dh):
    q, k, v = qkv.float().view(B, N, 3, H, dh).permute(2, 0, 3, 1, 4)
    return q, k, v


@pytest.mark.parametrize("dtype,dh,N,B,H", [(torch.bfloat16, 64, 333, 2, 3), (torch.bfloat16, 128, 200, 1, 2),
                                            (torch.bfloat16, 64, 64, 1, 1), (torch.bfloat16, 128, 1536, 1, 2),
                                            (torch.bfloat16, 64, 24, 3, 2),
                                            (torch.float32, 16, 24, 4, 4), (torch.float32, 64, 97, 2, 2)])
def test_attention_forward_backward(dtype, dh, N, B, H):
    torch.manual_seed(N + dh)
    dev = "cuda"
    d = H * dh
    qkv = (torch.randn(B * N, 3 * d, device=dev) * 1.5).to(dtype)
    o = torch.empty(B * N, d, device=dev, dtype=dtype)
    lse = torch.empty(B, H, N, device=dev)
    jg.test_attention_fwd(qkv, B, N, H, dh, o, lse)
    q, k, v = _attn_ref(qkv, B, N, H, dh)
    q.requires_grad_(); k.requires_grad_(); v.requires_grad_()
    s = (q @ k.transpose(-1, -2)) / math.sqrt(dh)
    ref_lse = torch.logsumexp(s, -1)
    ref_o = torch.softmax(s, -1) @ v
    tol = 1e-2 if dtype == torch.bfloat16 else 1e-5
    assert _rel(o.float().view(B, N, H, dh).transpose(1, 2), ref_o) < tol
    assert (lse - ref_lse).abs().max().item() < (1e-2 if dtype == torch.bfloat16 else 1e-5)
    dO = torch.randn(B * N, d, device=dev).to(dtype)
    # reference gradient uses the kernel's own (rounded) output, as the kernel does
    ref_o.backward(dO.float().view(B, N, H, dh).transpose(1, 2))
    dqkv = torch.empty(B * N, 3 * d, device=dev, dtype=dtype)
    jg.test_attention_bwd(qkv, o, lse, dO, B, N, H, dh, dqkv)
    torch.cuda.synchronize()
    g = dqkv.float().view(B, N, 3, H, dh).permute(2, 0, 3, 1, 4)
    for i, t in enumerate((q, k, v)):
        assert _rel(g[i], t.grad) < (2e-2 if dtype == torch.bfloat16 else 1e-4), "qkv"[i]


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("dh,N,n0,B,H", [(64, 333, 333, 2, 3), (64, 256, 128, 2, 2), (64, 64, 64, 1, 1),
                                         (64, 24, 24, 3, 2), (128, 1536, 512, 1, 2), (128, 200, 200, 1, 2),
                                         (128, 700, 256, 2, 2), (128, 4608, 512, 1, 1)])
def test_attention_backward_kernels_on_two_stream_views(dh, N, n0, B, H, impl):
    """Both backward kernels (impl 1: warp-level MMA, 2: tcgen05) against PyTorch fp32 on
    one buffer (n0 = N) and on the text/image stream split of the MMDiT double blocks."""
    torch.manual_seed(N + dh + n0)
    dev = "cuda"
    d = H * dh
    qkv = (torch.randn(B * N, 3 * d, device=dev) * 1.5).bfloat16()
    o = torch.empty(B * N, d, device=dev, dtype=torch.bfloat16)
    lse = torch.empty(B, H, N, device=dev)
    jg.test_attention_fwd(qkv, B, N, H, dh, o, lse)
    q, k, v = _attn_ref(qkv, B, N, H, dh)
    q.requires_grad_(); k.requires_grad_(); v.requires_grad_()
    ref_o = torch.softmax((q @ k.transpose(-1, -2)) / math.sqrt(dh), -1) @ v
    dO = torch.randn(B * N, d, device=dev).bfloat16()
    ref_o.backward(dO.float().view(B, N, H, dh).transpose(1, 2))

    def split(x):
        x = x.view(B, N, -1)
        return x[:, :n0].contiguous(), x[:, n0:].contiguous()

    dq0 = torch.full((B, n0, 3 * d), float("nan"), device=dev, dtype=torch.bfloat16)
    dq1 = torch.full((B, N - n0, 3 * d), float("nan"), device=dev, dtype=torch.bfloat16)
    jg.test_attention_bwd_streams(split(qkv), split(o), lse, split(dO), B, N, n0, H, dh, (dq0, dq1), impl=impl)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    g = torch.cat([dq0, dq1], 1).float().view(B, N, 3, H, dh).permute(2, 0, 3, 1, 4)
    for i, t in enumerate((q, k, v)):
        assert _rel(g[i], t.grad) < 2e-2, "qkv"[i]


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("dh,N,n0,B,H", [(64, 333, 333, 2, 3), (64, 256, 128, 2, 2), (64, 64, 64, 1, 1),
                                         (64, 24, 24, 3, 2), (64, 1000, 1000, 1, 2), (128, 1536, 512, 1, 2),
                                         (128, 200, 200, 1, 2), (128, 700, 256, 2, 2), (128, 4608, 512, 1, 1)])
def test_attention_forward_kernels_on_two_stream_views(dh, N, n0, B, H, impl):
    """Both forward kernels (impl 1: warp-level MMA, 2: tcgen05) against PyTorch fp32 on one
    buffer and on the text/image stream split: output and log-sum-exp, ragged last tiles."""
    torch.manual_seed(N + dh + n0 + 1)
    dev = "cuda"
    d = H * dh
    qkv = (torch.randn(B * N, 3 * d, device=dev) * 1.5).bfloat16()
    q, k, v = _attn_ref(qkv, B, N, H, dh)
    s = (q @ k.transpose(-1, -2)) / math.sqrt(dh)
    ref_lse = torch.logsumexp(s, -1)
    ref_o = torch.softmax(s, -1) @ v

    def split(x):
        x = x.view(B, N, -1)
        return x[:, :n0].contiguous(), x[:, n0:].contiguous()

    o0 = torch.full((B, n0, d), float("nan"), device=dev, dtype=torch.bfloat16)
    o1 = torch.full((B, N - n0, d), float("nan"), device=dev, dtype=torch.bfloat16)
    lse = torch.full((B, H, N), float("nan"), device=dev)
    jg.test_attention_fwd_streams(split(qkv), (o0, o1), lse, B, N, n0, H, dh, impl=impl)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    o = torch.cat([o0, o1], 1).float().view(B, N, H, dh).transpose(1, 2)
    assert _rel(o, ref_o) < 1e-2
    assert (lse - ref_lse).abs().max().item() < 1e-2


@pytest.mark.parametrize("impl", [1, 2])
@pytest.mark.parametrize("dh", [64, 128])
def test_attention_forward_online_softmax_with_climbing_maxima(dh, impl):
    """Scores that climb along the keys at a rate that differs from row to row (a_i b_t along
    one direction u): in some rows the running maximum moves up by tens of nats over the key
    tiles, in others it is reached in the first tile, and the rows of one warp disagree on
    whether to rescale.  Output and log-sum-exp against PyTorch fp32."""
    B, N, n0, H = 1, 1536, 512, 2
    d = H * dh
    g = torch.Generator(device="cpu").manual_seed(dh + 17 * impl)
    u = torch.randn(dh, generator=g)
    u /= u.norm()
    a = torch.randn(N, H, 1, generator=g) * 2.5                        # per-row rate
    bt = (16.0 * torch.arange(N) / N * math.sqrt(dh)).view(N, 1, 1)  # per-key climb
    q = torch.randn(N, H, dh, generator=g) + a * u
    k = torch.randn(N, H, dh, generator=g) + bt * u
    v = torch.randn(N, H, dh, generator=g)
    qkv = torch.stack([q, k, v], 1).reshape(B * N, 3 * d).bfloat16().cuda()
    qf, kf, vf = _attn_ref(qkv, B, N, H, dh)
    s = (qf @ kf.transpose(-1, -2)) / math.sqrt(dh)
    climb = s.max(-1).values - s[..., :128].max(-1).values
    assert climb.max().item() > 20 and (climb == 0).float().mean().item() > 0.2
    ref_lse = torch.logsumexp(s, -1)
    ref_o = torch.softmax(s, -1) @ vf
    x = qkv.view(B, N, -1)
    o0 = torch.full((B, n0, d), float("nan"), device="cuda", dtype=torch.bfloat16)
    o1 = torch.full((B, N - n0, d), float("nan"), device="cuda", dtype=torch.bfloat16)
    lse = torch.full((B, H, N), float("nan"), device="cuda")
    jg.test_attention_fwd_streams((x[:, :n0].contiguous(), x[:, n0:].contiguous()), (o0, o1), lse, B, N, n0, H,
                                  dh, impl=impl)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    o = torch.cat([o0, o1], 1).float().view(B, N, H, dh).transpose(1, 2)
    assert _rel(o, ref_o) < 1e-2
    assert (lse - ref_lse).abs().max().item() < 2e-2


def test_tcgen05_attention_backward_rejects_unaligned_streams():
    B, N, n0, H, dh = 1, 300, 100, 2, 64
    d = H * dh
    x = lambda n, c: torch.zeros(B, n, c, device="cuda", dtype=torch.bfloat16)
    lse = torch.zeros(B, H, N, device="cuda")
    with pytest.raises(jg.JaggError):
        jg.test_attention_bwd_streams((x(n0, 3 * d), x(N - n0, 3 * d)), (x(n0, d), x(N - n0, d)), lse,
                                      (x(n0, d), x(N - n0, d)), B, N, n0, H, dh,
                                      (x(n0, 3 * d), x(N - n0, 3 * d)), impl=2)


# ------------------------------------------------------------------ bounded waits
@pytest.mark.parametrize("limit_ns", [1_000_000, 20_000_000])
def test_bounded_wait_gives_up_and_reports_timeout(limit_ns):
    """A wait on an mbarrier that nothing arrives at ends after its limit: the kernel returns,
    the device status word reads JAGG_DEV_STATUS_TIMEOUT (then clears), and the context
    stays usable for the next call."""
    assert jg.device_status() == 0
    out = torch.zeros(2, dtype=torch.int64, device="cuda")
    jg.test_wait_timeout(limit_ns, out)
    torch.cuda.synchronize()
    gave_up, waited = out.tolist()
    assert gave_up == 1
    assert limit_ns <= waited < limit_ns + 50_000_000
    assert jg.device_status() == 1          # JAGG_DEV_STATUS_TIMEOUT, cleared by the read
    assert jg.device_status() == 0
    x = torch.randn(256, 256, device="cuda")
    assert torch.isfinite(x @ x).all()      # the context still works


@pytest.mark.parametrize("d,M,rps,ln,gate,dtype", [
    (3072, 4608 * 2, 4608, True, True, torch.bfloat16),   # Flux single block: row-per-CTA kernel
    (3072, 512 * 3, 512, True, False, torch.bfloat16),    # LayerNorm only
    (3072, 1024 * 2 + 0, 1024, False, True, torch.bfloat16),  # gate only
    (3072, 333 * 3, 333, True, True, torch.bfloat16),     # sequences that straddle CTA row shares
    (3072, 40, 8, True, True, torch.float32),             # f32 y: the persistent kernel
    (768, 333 * 4, 333, True, True, torch.bfloat16),      # DiT-B width: row-in-registers kernel
    (768, 256 * 3, 256, True, False, torch.bfloat16),     # DiT-B width, LayerNorm only
    (768, 77 * 5, 77, False, True, torch.bfloat16),       # DiT-B width, gate only (persistent kernel)
    (768, 333 * 2, 333, True, True, torch.float32),       # DiT-B width, f32 y
    (1024, 300, 100, True, True, torch.bfloat16),
    (64, 24 * 4, 24, True, True, torch.float32)])
def test_ln_gate_backward_kernels(d, M, rps, ln, gate, dtype):
    """LayerNorm + modulation backward fused with the gate backward (every kernel variant the
    dispatcher picks: row per CTA at d = 3072, row in registers up to 768, the persistent
    kernel otherwise) against PyTorch fp32 on the same inputs, including the per-sequence
    column sums (dshift, dscale, dgate) and the bias gradient."""
    torch.manual_seed(d + M)
    dev = "cuda"
    S = M // rps
    f = dict(device=dev, dtype=torch.float32)
    h = torch.randn(M, d, **f) * 2 + 0.5
    mean, rstd = h.mean(1), torch.rsqrt(h.var(1, unbiased=False) + 1e-6)
    dm = torch.randn(M, d, **f)
    scale = torch.randn(S, d, **f) * 0.3
    gate_v = torch.randn(S, d, **f)
    y = torch.randn(M, d, **f).to(dtype)
    dh_in = torch.randn(M, d, **f)
    dh_out = torch.empty_like(dh_in) if ln else None
    dshift, dscale, dgate = (torch.full((S, d), 0.25, **f) for _ in range(3))
    dbias = torch.full((d,), -0.5, **f)
    dy = torch.empty(M, d, device=dev, dtype=dtype)
    kw = {}
    if ln:
        kw.update(dm=dm, h=h, mean=mean, rstd=rstd, scale=scale, dshift=dshift, dscale=dscale)
    if gate:
        kw.update(y=y, gate=gate_v, dgate=dgate, dy=dy, dbias=dbias)
    jg.test_ln_gate_bwd(M, d, rps, dh_in, dh_out, **kw)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    seq = torch.arange(M, device=dev) // rps
    xh = (h - mean[:, None]) * rstd[:, None]
    if ln:
        e = dm * (1 + scale[seq])
        dh_ref = dh_in + rstd[:, None] * (e - e.mean(1, keepdim=True) - xh * (e * xh).mean(1, keepdim=True))
        assert _rel(dh_out, dh_ref) < 1e-5
        assert _rel(dshift - 0.25, torch.zeros(S, d, **f).index_add_(0, seq, dm)) < 1e-5
        assert _rel(dscale - 0.25, torch.zeros(S, d, **f).index_add_(0, seq, dm * xh)) < 1e-5
    else:
        dh_ref = dh_in
    if gate:
        yf = y.float()
        assert _rel(dy.float(), gate_v[seq] * dh_ref) < (1e-2 if dtype == torch.bfloat16 else 1e-6)
        assert _rel(dgate - 0.25, torch.zeros(S, d, **f).index_add_(0, seq, dh_ref * yf)) < 1e-5
        sums = torch.zeros(S, d, **f).index_add_(0, seq, dh_ref)
        assert _rel(dbias + 0.5, (gate_v * sums).sum(0)) < 1e-5


def _qkn_reference(x, N, n_txt, gw, dh, scale, rope):
    """RMSNorm per head (eps 1e-6, learned scale) then 2D RoPE: the first dh/4 rotated pairs by
    the patch row, the rest by the column, pairs (2i, 2i+1), theta_i = 10000^(-2i/(dh/2)),
    text tokens (the first n_txt of each sequence) not rotated.  x [M, H, dh] f32."""
    M, H, _ = x.shape
    y = x * torch.rsqrt((x * x).mean(-1, keepdim=True) + 1e-6) * scale
    if not rope:
        return y
    n = torch.arange(M, device=x.device) % N
    tok = (n - n_txt).clamp(min=0)
    npair = dh // 4
    i = torch.arange(npair, device=x.device, dtype=torch.float32)
    theta = 10000.0 ** (-2.0 * i / (dh // 2))
    pos = torch.cat([(tok // gw)[:, None].float().expand(M, npair), (tok % gw)[:, None].float().expand(M, npair)], 1)
    ang = pos * torch.cat([theta, theta])[None, :]
    ang = torch.where((n < n_txt)[:, None], torch.zeros_like(ang), ang)
    c, s = torch.cos(ang)[:, None, :], torch.sin(ang)[:, None, :]
    y0, y1 = y[..., 0::2], y[..., 1::2]
    out = torch.empty_like(y)
    out[..., 0::2] = y0 * c - y1 * s
    out[..., 1::2] = y0 * s + y1 * c
    return out


@pytest.mark.parametrize("dh,H,N,n_txt,gw,B,dtype,rope", [
    (128, 4, 1536, 512, 32, 2, torch.bfloat16, True),   # Flux single block: vectorised kernels
    (128, 3, 1024, 0, 32, 2, torch.bfloat16, True),     # image stream of a double block
    (128, 2, 512, 512, 32, 3, torch.bfloat16, True),    # text stream: no rotation
    (128, 2, 300, 44, 16, 2, torch.bfloat16, True),     # ragged sequence, 16 x 16 grid
    (64, 3, 300, 44, 16, 2, torch.bfloat16, True),      # head dim 64: the per-element kernels
    (32, 4, 24, 8, 4, 3, torch.float32, True),
    (128, 2, 256, 0, 16, 1, torch.bfloat16, False)])
def test_qk_norm_rope_kernels(dh, H, N, n_txt, gw, B, dtype, rope):
    """Per-head RMSNorm + 2D RoPE forward (normalised, rotated q and k; 1/rms of each) and its
    backward (gradients of the raw q, k in place; the scale gradients) against PyTorch fp32
    autograd on the same inputs, in the model's layout (q, k inside a [M, 3d] buffer, the
    gradient inside a wider one)."""
    torch.manual_seed(dh + N + n_txt)
    dev = "cuda"
    d, M = H * dh, B * N
    qkv = (torch.randn(M, 3 * d, device=dev) * 2).to(dtype)
    qs, ks = (1 + 0.1 * torch.randn(dh, device=dev)).to(dtype), (1 + 0.1 * torch.randn(dh, device=dev)).to(dtype)
    qk = torch.empty(M, 2 * d, device=dev, dtype=dtype)
    rq, rk = torch.empty(M, H, device=dev), torch.empty(M, H, device=dev)
    jg.test_qk_norm_rope_fwd(qkv, M, N, H, n_txt, gw, qs, ks, qk, rq, rk, rope=rope)
    ld = 3 * d + 64
    g_up = (torch.randn(M, ld, device=dev)).to(dtype)
    dqk = g_up.clone()
    dqs, dks = torch.zeros(dh, device=dev), torch.zeros(dh, device=dev)
    jg.test_qk_norm_rope_bwd(qkv, M, N, H, n_txt, gw, qs, ks, rq, rk, dqk, dqs, dks, rope=rope)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    xq = qkv[:, :d].float().view(M, H, dh).requires_grad_()
    xk = qkv[:, d:2 * d].float().view(M, H, dh).requires_grad_()
    sq, sk = qs.float().requires_grad_(), ks.float().requires_grad_()
    yq = _qkn_reference(xq, N, n_txt, gw, dh, sq, rope)
    yk = _qkn_reference(xk, N, n_txt, gw, dh, sk, rope)
    tol = 1e-2 if dtype == torch.bfloat16 else 1e-5
    assert _rel(qk[:, :d].float(), yq.reshape(M, d)) < tol
    assert _rel(qk[:, d:].float(), yk.reshape(M, d)) < tol
    ref_r = torch.rsqrt((xq.detach() ** 2).mean(-1) + 1e-6)
    assert _rel(rq, ref_r) < 1e-5
    (yq.reshape(M, d) * g_up[:, :d].float()).sum().add((yk.reshape(M, d) * g_up[:, d:2 * d].float()).sum()).backward()
    assert _rel(dqk[:, :d].float(), xq.grad.reshape(M, d)) < 2 * tol
    assert _rel(dqk[:, d:2 * d].float(), xk.grad.reshape(M, d)) < 2 * tol
    assert torch.equal(dqk[:, 2 * d:], g_up[:, 2 * d:]), "columns past q, k changed"
    assert _rel(dqs, sq.grad) < 1e-4 and _rel(dks, sk.grad) < 1e-4


@pytest.mark.parametrize("rows,cols,ld,dtype", [(36864, 3072, 3072, torch.bfloat16), (4096, 12288, 21504, torch.bfloat16),
                                                (333, 2304, 2304, torch.bfloat16), (97, 200, 210, torch.float32)])
def test_colsum_kernels(rows, cols, ld, dtype):
    """Bias-gradient column sums (db += sum over rows, into a nonzero db) against PyTorch."""
    torch.manual_seed(rows + cols)
    X = torch.randn(rows, ld, device="cuda").to(dtype)
    db = torch.full((cols,), 0.5, device="cuda")
    jg.test_colsum(X[:, :cols], db)
    torch.cuda.synchronize()
    ref = X[:, :cols].double().sum(0) + 0.5
    assert _rel(db, ref) < 1e-5


@pytest.mark.parametrize("M,N,K", [(300, 600, 2112), (1000, 768, 3072), (128, 1280, 4096)])
def test_multiplier_epilogue_long_k(M, N, K):
    """The multiplier epilogue at long K, where the library picks 256-column tiles with the
    two-slot multiplier ring (the fc2 / lin2 input gradients at the Flux widths), ragged
    rows and column tiles, against the same product at 128 columns and PyTorch fp32."""
    torch.manual_seed(M + N + K)
    dev = "cuda"
    A = torch.randn(M, K, device=dev).bfloat16()
    B = (torch.randn(N, K, device=dev) / math.sqrt(K)).bfloat16()
    Bt = B.t().contiguous()
    X = torch.rand(M, N, device=dev).bfloat16()
    ref = (A.float() @ B.float().t()) * X.float()
    outs = []
    for tile_n in (0, 128):
        O = torch.full((M, N + 8), 3.0, device=dev, dtype=torch.bfloat16)
        jg.test_gemm(_desc(M, N, K, A, K, 0, Bt, N, 1, jg.DTYPE_BF16, O, N + 8, jg.DTYPE_BF16, epi=3, aux=X, ld_aux=N,
                           tile_n=tile_n))
        outs.append(O)
    torch.cuda.synchronize()
    assert jg.device_status() == 0
    for O in outs:
        assert _rel(O[:, :N].float(), ref) < 5e-3
        assert torch.all(O[:, N:] == 3.0)
    assert _rel(outs[0][:, :N].float(), outs[1][:, :N].float()) < 5e-3
