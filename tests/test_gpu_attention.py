"""The paged causal attention kernel (sd2_attention) against the oracle's attention (Sec. 3.2 decoder).

Each case builds a bf16 KV pool whose blocks are scattered through a random block table, row groups
at chosen positions of ragged sequences, and checks every output against oracle.model.causal_attention
evaluated in float64 on the same bf16 keys/values and bf16-rounded queries (the kernel stages queries
and probabilities in bf16). Covered: 1 to 16 context splits with empty splits, chunks of one and
several tiles, verifier-, drafter- and prompt-shaped groups, GQA ratios 1, 4 and 8, head dims 64 and
128, and the decode-step path whose cache rows below a pre-step length are read before the
programmatic wait (boundaries inside a tile, on a tile edge, on a split edge, at zero), with finite
stale rows between the last row and the planned bound; K/V rings of 2 to 4 tiles and split-merge
buffers laid over the ring. A row beyond the planned bound must raise the range bit of the error
word, not fault.
"""
import pytest
import torch

from oracle import model as oracle_model
from paper_2511_09844_gb300 import sd2

pytestmark = pytest.mark.gpu

ERR_TIMEOUT, ERR_RANGE = 2, 4


def _case(seed, seq_lens, rows_per_group, H, Hkv, hd, n_layers=2, layer=1):
    """Random pool/table/queries; group g = the last rows_per_group[g] positions of sequence g."""
    g = torch.Generator().manual_seed(seed)
    n_seq = len(seq_lens)
    bt_stride = max((L + 15) // 16 for L in seq_lens) + 1
    n_blocks = n_seq * bt_stride + 3
    pool = (torch.randn(n_layers, n_blocks, 2, Hkv, 16, hd, generator=g)).to(torch.bfloat16)
    perm = torch.randperm(n_blocks, generator=g)[: n_seq * bt_stride]
    table = perm.view(n_seq, bt_stride).to(torch.int32)
    row_pos, grp_row0, grp_nrows, grp_seq = [], [], [], []
    for s, (L, nr) in enumerate(zip(seq_lens, rows_per_group)):
        grp_row0.append(len(row_pos))
        grp_nrows.append(nr)
        grp_seq.append(s)
        row_pos += list(range(L - nr, L))
    M = len(row_pos)
    q = torch.randn(M, H, hd, generator=g) * 2.0
    return dict(pool=pool, table=table, q=q, row_pos=torch.tensor(row_pos, dtype=torch.int32),
                grp_row0=torch.tensor(grp_row0, dtype=torch.int32), grp_nrows=torch.tensor(grp_nrows, dtype=torch.int32),
                grp_seq=torch.tensor(grp_seq, dtype=torch.int32), layer=layer, seq_lens=seq_lens, H=H, hd=hd)


def _reference(c):
    """Oracle attention per sequence: dense K/V gathered through the table, queries at their positions."""
    pool, table, layer = c["pool"], c["table"], c["layer"]
    H, hd = c["H"], c["hd"]
    q_bf = c["q"].to(torch.bfloat16).double()
    out = torch.zeros(c["q"].shape[0], H * hd, dtype=torch.float64)
    for g in range(len(c["grp_row0"])):
        s, r0, nr = int(c["grp_seq"][g]), int(c["grp_row0"][g]), int(c["grp_nrows"][g])
        pos = c["row_pos"][r0:r0 + nr].tolist()
        T = max(pos) + 1
        blocks = table[s, : (T + 15) // 16].long()
        kv = pool[layer, blocks].double()                          # [nb, 2, Hkv, 16, hd]
        k = kv[:, 0].permute(0, 2, 1, 3).reshape(-1, kv.shape[2], hd)[:T]
        v = kv[:, 1].permute(0, 2, 1, 3).reshape(-1, kv.shape[2], hd)[:T]
        qf = torch.zeros(T, H, hd, dtype=torch.float64)
        for i, p in enumerate(pos):
            qf[p] = q_bf[r0 + i]
        o = oracle_model.causal_attention(qf, k, v, row_block=512)
        for i, p in enumerate(pos):
            out[r0 + i] = o[p].reshape(-1)
    return out


def _run(c, n_splits, chunk, pre_len=None, pre_stable=0, pre_fresh=0, max_rows=None):
    dev = {k: v.cuda() for k, v in c.items() if isinstance(v, torch.Tensor)}
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = sd2.attention(dev["q"].float().contiguous(), dev["pool"], dev["table"], c["layer"], dev["row_pos"],
                        dev["grp_row0"], dev["grp_nrows"], dev["grp_seq"],
                        max_rows or int(c["grp_nrows"].max()), n_splits, chunk,
                        pre_len=None if pre_len is None else torch.tensor(pre_len, dtype=torch.int32, device="cuda"),
                        pre_stable=pre_stable, pre_fresh=pre_fresh, err=err)
    torch.cuda.synchronize()
    return out.float().cpu(), int(err.item())


def _check(out, ref):
    assert torch.isfinite(out).all()
    torch.testing.assert_close(out.double(), ref, atol=1.5e-2, rtol=1e-2)


@pytest.mark.parametrize("n_splits,chunk", [(1, 1152), (9, 128), (16, 128), (5, 256), (16, 64 * 18)])
def test_verify_shaped_groups_over_splits(n_splits, chunk):
    """Verify blocks (6 rows x 4 heads per KV head, hd 128) of ragged sequences; the large-chunk
    cases leave most splits empty."""
    c = _case(1, seq_lens=[1030, 517, 70], rows_per_group=[6, 6, 6], H=32, Hkv=8, hd=128)
    out, err = _run(c, n_splits, chunk)
    assert err == 0
    _check(out, _reference(c))


@pytest.mark.parametrize("hd,H,Hkv,rows", [(64, 32, 8, [1, 2, 1]), (64, 8, 8, [2, 1, 2]), (128, 64, 8, [6, 3, 1])])
def test_drafter_and_gqa_shapes(hd, H, Hkv, rows):
    """Drafter rows (1 or 2 per sequence), GQA ratios 1, 4 and 8."""
    c = _case(2, seq_lens=[700, 129, 64], rows_per_group=rows, H=H, Hkv=Hkv, hd=hd)
    out, err = _run(c, 11, 64)
    assert err == 0
    _check(out, _reference(c))


def test_prompt_shaped_group():
    """A prompt chunk: 16 rows x 4 heads = 64 query vectors (the per-CTA maximum)."""
    c = _case(3, seq_lens=[300, 16], rows_per_group=[16, 16], H=16, Hkv=4, hd=64)
    out, err = _run(c, 3, 128)
    assert err == 0
    _check(out, _reference(c))


@pytest.mark.parametrize("stable_off", [0, 3, 6])
@pytest.mark.parametrize("lens", [[517, 1030, 7], [512, 640, 6], [1024, 200, 13]])
def test_decode_step_reads_pre_step_rows_early(lens, stable_off):
    """pre_len places the boundary inside a tile, on a tile edge, on a split edge and at zero. The rows
    between the last row and pre_len + pre_stable + pre_fresh hold finite stale values, masked."""
    k1 = 6
    c = _case(4, seq_lens=lens, rows_per_group=[k1] * 3, H=32, Hkv=8, hd=128)
    ref = _reference(c)
    # verifier convention: rows at n-1 .. n-1+k, cache [0, n-1) written before the step
    pre_len = [L - k1 + 1 - stable_off for L in lens]
    pre_len = [max(0, p) for p in pre_len]
    out, err = _run(c, 9, 128, pre_len=pre_len, pre_stable=-1, pre_fresh=k1 + stable_off + 1)
    assert err == 0
    _check(out, ref)
    # the same with more splits than the context needs and one-tile chunks
    out, err = _run(c, 16, 64 * 2, pre_len=pre_len, pre_stable=-1, pre_fresh=k1 + stable_off + 1)
    assert err == 0
    _check(out, ref)


def test_row_beyond_the_planned_bound_is_reported():
    """pre_fresh one short: each sequence's last key row is zero-filled instead of read, and the
    kernel reports the range error instead of reading outside the planned rows."""
    k1 = 6
    c = _case(5, seq_lens=[600, 300], rows_per_group=[k1, k1], H=32, Hkv=8, hd=128)
    pre_len = [600 - k1 + 1, 300 - k1 + 1]
    out, err = _run(c, 9, 128, pre_len=pre_len, pre_stable=-1, pre_fresh=k1 - 1)
    assert err & ERR_RANGE
    assert torch.isfinite(out).all()


def test_bad_arguments_are_rejected_on_the_host():
    c = _case(6, seq_lens=[100], rows_per_group=[2], H=32, Hkv=8, hd=128)
    with pytest.raises(sd2.SD2Error):
        _run(c, 17, 64)                 # more splits than a cluster takes
    with pytest.raises(sd2.SD2Error):
        _run(c, 2, 96)                  # chunk not a multiple of 64
    with pytest.raises(sd2.SD2Error):
        _run(c, 2, 64, max_rows=17)     # 17 rows x 4 heads per KV head > 64 query vectors


@pytest.mark.parametrize("hd,k1,n_splits,chunk", [(128, 9, 2, 768), (128, 9, 16, 128), (64, 2, 2, 768), (64, 1, 9, 256)])
def test_ring_depths_and_merge_over_the_ring(hd, k1, n_splits, chunk):
    """K/V rings of 2 to 4 tiles and, where two CTAs per SM fit only that way (48 query vectors at
    16 splits), the split-merge buffers laid over the ring; decode steps and plain launches."""
    lens = [1030, 517, 70]
    c = _case(7, seq_lens=lens, rows_per_group=[k1] * 3, H=32, Hkv=8, hd=hd)
    ref = _reference(c)
    pre_len = [max(0, L - k1 + 1) for L in lens]
    out, err = _run(c, n_splits, chunk, pre_len=pre_len, pre_stable=-1, pre_fresh=k1 + 1)
    assert err == 0
    _check(out, ref)
    out, err = _run(c, n_splits, chunk)
    assert err == 0
    _check(out, ref)


def test_many_sequences_four_ctas_per_sm():
    """16 drafter-shaped groups x 8 KV heads x 4 splits = 512 CTAs: the hd = 64 launch sized for four
    resident CTAs per SM (its shared-memory share), in a decode step and a plain launch."""
    lens = [70 + 61 * i for i in range(16)]
    c = _case(8, seq_lens=lens, rows_per_group=[1] * 16, H=32, Hkv=8, hd=64)
    ref = _reference(c)
    pre_len = [L - 1 for L in lens]
    out, err = _run(c, 4, 320, pre_len=pre_len, pre_stable=0, pre_fresh=1)
    assert err == 0
    _check(out, ref)
    out, err = _run(c, 4, 320)
    assert err == 0
    _check(out, ref)


def _run_flat(c, slots, max_ctx, pre_len, pre_stable, pre_fresh, workspace=None):
    dev = {k: v.cuda() for k, v in c.items() if isinstance(v, torch.Tensor)}
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = sd2.attention_flat(dev["q"].float().contiguous(), dev["pool"], dev["table"], c["layer"], dev["row_pos"],
                             dev["grp_row0"], dev["grp_nrows"], dev["grp_seq"], int(c["grp_nrows"].max()), slots,
                             max_ctx, torch.tensor(pre_len, dtype=torch.int32, device="cuda"), pre_stable=pre_stable,
                             pre_fresh=pre_fresh, workspace=workspace, err=err)
    torch.cuda.synchronize()
    return out.float().cpu(), int(err.item())


def test_flat_mode_sixty_four_ragged_sequences():
    """Flat mode (sd2_attention_flat) with the most groups a launch takes, 64 drafter-shaped groups of
    ragged lengths: groups 32..63 take the slot map's second lane half; most of the 150 slots a KV
    head has are idle. A second call on the same workspace checks that its counters reset."""
    lens = [30 + (97 * i) % 301 for i in range(64)]
    k1 = 2
    c = _case(9, seq_lens=lens, rows_per_group=[k1] * 64, H=8, Hkv=2, hd=64)
    ref = _reference(c)
    pre_len = [L - k1 for L in lens]
    ws = torch.zeros(sd2.load_library().sd2_attention_flat_workspace_bytes(2, 150, 64), dtype=torch.uint8,
                     device="cuda")
    for _ in range(2):
        out, err = _run_flat(c, 150, max(lens) + 8, pre_len, 0, k1, workspace=ws)
        assert err == 0
        _check(out, ref)


@pytest.mark.parametrize("slots", [100, 3])
def test_flat_mode_long_sequence_over_many_slots(slots):
    """Verify-shaped groups (6 rows x 4 heads, hd 128), one sequence of 2100 positions among two
    short ones. With 100 slots the per-group cap of 32 slots sets the tiles per slot (2: the long
    sequence over 17 slots); with 3 slots every group takes one."""
    lens = [2100, 70, 150]
    k1 = 6
    c = _case(10, seq_lens=lens, rows_per_group=[k1] * 3, H=8, Hkv=2, hd=128)
    ref = _reference(c)
    pre_len = [L - k1 + 1 for L in lens]      # verifier convention: rows at n-1 .. n-1+k
    out, err = _run_flat(c, slots, max(lens) + 8, pre_len, -1, k1 + 1)
    assert err == 0
    _check(out, ref)


def test_flat_mode_bad_arguments_are_rejected_on_the_host():
    c = _case(11, seq_lens=[100, 90], rows_per_group=[2, 2], H=32, Hkv=8, hd=128)
    with pytest.raises(sd2.SD2Error):
        _run_flat(c, 1, 120, [98, 88], 0, 2)       # fewer slots than groups
    with pytest.raises(sd2.SD2Error):
        _run_flat(c, 8, 64, [98, 88], 0, 2)        # a context bound of one tile
