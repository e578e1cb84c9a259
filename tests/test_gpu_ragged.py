"""Ragged and paged caches (continuous batching): every sequence of the batch
holds its own number of tokens, appends its own number of new tokens, and is
released and restarted on its own; a PAGED cache keeps each sequence's tokens
in 64-token pages of one pool.  Each sequence is checked against an
independent oracle cache of one sequence fed the same tokens (Section 3.1
coding, Sections 3.2-3.3 attention over the reconstruction):

  - its code and metadata rows, bit for bit (PAGED: gathered through the
    sequence's pages);
  - prefill attention of its newest n_b tokens and decode attention of its
    newest token, within the bf16 bound of every attention test;
  - the RoPE positions of a ragged decode step's projection, which continue
    each sequence at its own count."""
import numpy as np
import pytest
import torch

from oracle import kvq_oracle as O
from paper_2609_04263_gb300 import kvq, synth
from tests.gpu_common import require_gpu
from tests.helpers import (FORMATS, check_attention, check_projection, kv_pair, live,
                           oracle_cache, to_numpy_plane)

pytestmark = pytest.mark.gpu

PLANE_NAMES = ("k_codes", "k_scale", "k_zero", "v_codes", "v_scale", "v_zero", "k_full",
               "v_full")


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    require_gpu()


def _cache(spec, B, H, Hq, D, Tmax, layout, num_pages=0):
    from paper_2609_04263_gb300 import api
    kw = dict(spec)
    fmt = kw.pop("fmt")
    desc = api.make_desc(fmt, kw["key_bits"], kw["value_bits"], kw["group_size"], B, H, Hq, D,
                         Tmax, torch.bfloat16, residual_tokens=kw.get("residual_tokens", 0),
                         layout=layout, num_pages=num_pages)
    return api.Cache(desc)


PG = kvq.KVQ_PAGE_TOKENS


def _seq_rows(gc, name, b, T):
    """Sequence b's rows [1, H, rows, cols] of a plane (PAGED: gathered
    through its pages; KIVI's key scales and zeros hold a row per 32-token
    block, its full-precision ring stays per sequence)."""
    p = gc.planes()[name]
    if name.endswith("_full"):
        return p[b:b + 1]
    if gc.desc.layout != kvq.KVQ_LAYOUT_PAGED:
        return p[b:b + 1]
    per = PG // 32 if (gc.desc.fmt == kvq.KVQ_FMT_KIVI and name in ("k_scale", "k_zero")) else PG
    pages = gc.seq_pages(b)
    assert len(pages) == (T + PG - 1) // PG
    if not pages:
        return p[0:1, :, :0]
    return torch.cat([p[0:1, :, per * pg:per * pg + per] for pg in pages], dim=2)


def _compare_seq(gc, oc, b):
    """Bit-exact comparison of sequence b's live rows with its oracle cache."""
    T = oc.T
    assert gc.seq_tokens(b) == T
    for name in PLANE_NAMES:
        if name not in oc.planes or oc.planes[name].size == 0:
            continue
        got = live(name, to_numpy_plane(_seq_rows(gc, name, b, T).contiguous()), oc)
        ref = live(name, oc.planes[name], oc)
        assert got.shape == ref.shape, (name, got.shape, ref.shape)
        if got.dtype == np.float32:         # full-precision rows (bf16 read as fp32)
            same = np.array_equal(got, ref.astype(np.float32))
        else:
            same = np.array_equal(got.view(np.uint8), ref.view(np.uint8))
        assert same, f"sequence {b} plane {name} differs"


class Batch:
    """A ragged GPU cache and one oracle cache per sequence, fed together."""

    def __init__(self, fmt, B, H, Hq, D, Tmax, layout, num_pages=0, seed=0):
        self.spec = FORMATS[fmt]
        self.B, self.H, self.Hq, self.D, self.Tmax = B, H, Hq, D, Tmax
        self.gc = _cache(self.spec, B, H, Hq, D, Tmax, layout, num_pages)
        self.oc = [oracle_cache(self.spec, 1, H, D, Tmax, "bf16") for _ in range(B)]
        self.seed = seed
        self.step = 0
        self.n_last = [0] * B

    def append(self, n):
        L = max(max(n), 1)
        k, v, nk, nv = kv_pair(self.B, self.H, L, self.D, "bf16", seed=self.seed, stream=self.step)
        self.step += 1
        self.gc.append_ragged(k, v, n)
        for b in range(self.B):
            if n[b]:
                self.oc[b].append(nk[b:b + 1, :, :n[b]], nv[b:b + 1, :, :n[b]])
        self.n_last = list(n)
        return L

    def release(self, b):
        self.gc.seq_release(b)
        self.oc[b] = oracle_cache(self.spec, 1, self.H, self.D, self.Tmax, "bf16")
        self.n_last[b] = 0

    def check_planes(self):
        torch.cuda.synchronize()
        for b in range(self.B):
            _compare_seq(self.gc, self.oc[b], b)

    def check_prefill(self, L):
        rng = np.random.default_rng(100 + self.step)
        q = torch.from_numpy(rng.standard_normal((self.B, self.Hq, L, self.D)).astype(np.float32))
        q = q.bfloat16()
        out = self.gc.attend_prefill(q.cuda()).float().cpu().numpy()
        for b in range(self.B):
            n = self.n_last[b]
            if n == 0:
                continue
            ref = O.attend(self.oc[b], q[b:b + 1, :, :n].float().numpy())
            check_attention(out[b:b + 1, :, :n], ref, "bf16", f"prefill of sequence {b}")

    def check_decode(self):
        rng = np.random.default_rng(200 + self.step)
        q = torch.from_numpy(rng.standard_normal((self.B, self.Hq, 1, self.D)).astype(np.float32))
        q = q.bfloat16()
        out = self.gc.attend_decode(q.cuda()).float().cpu().numpy()
        for b in range(self.B):
            if self.oc[b].T == 0:
                assert np.all(out[b] == 0), "an empty sequence attends to nothing"
                continue
            ref = O.attend(self.oc[b], q[b:b + 1].float().numpy())
            check_attention(out[b:b + 1], ref, "bf16", f"decode of sequence {b}")


@pytest.mark.parametrize("layout", [kvq.KVQ_LAYOUT_RAGGED, kvq.KVQ_LAYOUT_PAGED])
@pytest.mark.parametrize("fmt,B,H,Hq,D", [("affine4", 3, 2, 8, 64), ("sym2", 4, 2, 8, 128),
                                          ("kivi2", 3, 2, 8, 128), ("kivi4", 3, 2, 4, 64)])
def test_ragged_batch_lifecycle(layout, fmt, B, H, Hq, D):
    pages = 3 * B * 2 if layout == kvq.KVQ_LAYOUT_PAGED else 0
    bt = Batch(fmt, B, H, Hq, D, 512, layout, pages, seed=D + B)
    counts = [[100, 37, 0, 64][:B], [5, 64, 130, 1][:B], [0, 3, 200, 63][:B]]
    for n in counts:                          # ragged prefill chunks
        L = bt.append(n)
        bt.check_prefill(L)
    bt.check_planes()
    for _ in range(3):                        # decode steps, one token per sequence
        bt.append([1] * B)
        bt.check_decode()
    bt.check_planes()
    # sequence 1 finishes; its slot starts a new sequence while the others run on
    bt.release(1)
    if layout == kvq.KVQ_LAYOUT_PAGED:
        held = sum((bt.oc[b].T + PG - 1) // PG for b in range(B))
        assert bt.gc.free_pages() == pages - held
    bt.check_decode()                         # the released sequence is empty
    n = [1] * B
    n[1] = 70
    L = bt.append(n)
    bt.check_prefill(L)
    bt.append([1] * B)
    bt.check_decode()
    bt.check_planes()


def test_paged_pool_exhaustion_and_reuse():
    """Appends that need more pages than the pool holds are refused whole;
    released pages serve the next sequence."""
    bt = Batch("affine4", 2, 2, 4, 64, 1024, kvq.KVQ_LAYOUT_PAGED, num_pages=4, seed=3)
    bt.append([300, 60])                      # 2 + 1 pages of 256 tokens
    assert bt.gc.free_pages() == 1
    k = torch.zeros(2, 2, 600, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(kvq.KvqError) as ei:
        bt.gc.append_ragged(k, k, [600, 0])   # would need 2 more pages
    assert ei.value.status == kvq.KVQ_ERR_CAPACITY
    assert bt.gc.free_pages() == 1 and bt.gc.seq_tokens(0) == 300
    bt.release(0)
    assert bt.gc.free_pages() == 3
    L = bt.append([700, 10])                  # the released pages come back: 3 + 0
    bt.check_prefill(L)
    bt.check_planes()
    assert bt.gc.free_pages() == 0


def test_ragged_decode_step_positions():
    """kvq_decode_step on a ragged cache: each sequence's new token is rotated
    at that sequence's own position, then appended and attended."""
    from paper_2609_04263_gb300 import api
    B, H, Hq, D, d_in = 3, 2, 8, 64, 256
    bt = Batch("affine4", B, H, Hq, D, 256, kvq.KVQ_LAYOUT_RAGGED, seed=11)
    bt.append([40, 7, 90])
    wl = synth.Workload(name="t", dtype="bf16", layers=1, d_in=d_in, n_q_heads=Hq, n_kv_heads=H,
                        head_dim=D, rope_base=10000.0, batch=B, prefill=8, decode=0, fmt=1,
                        key_bits=4, value_bits=4, group_size=32, rank=8)
    w, lora = synth.layer_weights(wl, 0, seed=5)
    tw = torch.from_numpy(w).bfloat16()
    tl = {p: tuple(torch.from_numpy(t).bfloat16() for t in lora[p]) for p in "qkv"}
    nl = {p: tuple(t.float().numpy() for t in tl[p]) for p in "qkv"}
    x = torch.from_numpy(synth.hidden_states((B, 1, d_in), outlier_frac=0.01, seed=6)).bfloat16()
    T_before = [bt.oc[b].T for b in range(B)]
    (q, k, v), out = bt.gc.decode_step(x.cuda(), tw.cuda(),
                                       {p: tuple(t.cuda() for t in tl[p]) for p in "qkv"},
                                       2.0, 10000.0)
    torch.cuda.synchronize()
    for b in range(B):
        ref = O.project_lora(x[b:b + 1].float().numpy(), tw.float().numpy(), nl, 2.0, Hq, H, D,
                             pos0=T_before[b], rope_base=10000.0)
        for got, r_, name in zip((q, k, v), ref, "qkv"):
            check_projection(got[b:b + 1].float().cpu().numpy(), r_, "bf16",
                             f"{name} of sequence {b} at position {T_before[b]}")
        bt.oc[b].append(k[b:b + 1].float().cpu().numpy(), v[b:b + 1].float().cpu().numpy())
        ref_o = O.attend(bt.oc[b], q[b:b + 1].float().cpu().numpy())
        check_attention(out[b:b + 1].float().cpu().numpy(), ref_o, "bf16", f"decode of sequence {b}")
    bt.check_planes()


@pytest.mark.parametrize("layout", [kvq.KVQ_LAYOUT_RAGGED, kvq.KVQ_LAYOUT_PAGED])
@pytest.mark.parametrize("fmt", ["sym2", "kivi2"])
def test_streaming_decode_over_ragged_sequences(layout, fmt):
    """Long ragged caches take the persistent streaming decode kernel (whose
    work split follows each sequence's own block count, and whose copies stay
    inside one page): sequences of very different lengths, one of them empty
    and one holding a single token."""
    B, H, Hq, D = 8, 4, 32, 64
    lens = [4000, 10, 0, 3000, 4096, 1, 2500, 64]
    pages = sum((t + PG - 1) // PG for t in lens) + 4
    bt = Batch(fmt, B, H, Hq, D, 4160, layout, pages if layout == kvq.KVQ_LAYOUT_PAGED else 0,
               seed=21)
    for lo in range(0, max(lens), 1024):
        bt.append([max(0, min(1024, t - lo)) for t in lens])
    bt.check_decode()
    bt.append([1, 1, 0, 1, 1, 1, 1, 1])       # one more token for all but the empty one
    bt.check_decode()
    bt.check_planes()


def test_streaming_decode_one_long_sequence():
    """One long sequence among single-token ones: the streaming decode takes
    fewer CTAs so that the long sequence's head is not split across more of
    them than its merge holds."""
    bt = Batch("affine4", 4, 1, 4, 64, 8192, kvq.KVQ_LAYOUT_PAGED, num_pages=40, seed=31)
    lens = [8000, 1, 1, 0]
    for lo in range(0, 8000, 2048):
        bt.append([max(0, min(2048, t - lo)) for t in lens])
    bt.check_decode()
