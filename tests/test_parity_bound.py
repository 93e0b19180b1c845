"""The end-to-end parity bar (CPU): the per-row perturbation bound that
parity_helpers.e2e_row_bounds derives for cache records differing within the
append tolerance really bounds the change of the exact attention output.
Records of an oracle-written cache are perturbed here on the CPU (a code
moved to its neighbour level, an fp16 ulp of a scale or a min, in keys and
values), and the oracle's decode of the perturbed cache must stay within
the bound of its decode of the original, for every row."""
import numpy as np

from oracle import oracle
from paper_2608_02691_gb300 import synth

import parity_helpers as ph


def _perturb(pool, case, rng, n):
    """n random token records of the written context get one change each;
    returns the perturbed pool and the diff mask [n_tok][h_kv]."""
    pg = pool.copy()
    cu = case["cu_ctx"].numpy()
    pos0 = case["pos0_ctx"].numpy()
    pages, slots = ph.token_slots(cu, pos0, case["block_table"])
    mask = np.zeros((len(pages), case["h_kv"]), bool)
    for _ in range(n):
        t = int(rng.integers(len(pages)))
        h = int(rng.integers(case["h_kv"]))
        kind = int(rng.integers(2))
        chunk = pg[pages[t], h]
        what = int(rng.integers(3))
        if what == 0:  # a code to a neighbouring level
            ch = int(rng.integers(128))
            byte = 512 * kind + slots[t] * 32 + ph.CODE_BYTE[ch]
            sh = ph.CODE_SHIFT[ch]
            code = (int(chunk[byte]) >> sh) & 3
            new = code + 1 if code < 3 else code - 1
            chunk[byte] = (int(chunk[byte]) & ~(3 << sh) & 0xFF) | (new << sh)
        else:  # one fp16 ulp of a scale (1) or a min (2)
            g = int(rng.integers(4))
            off = 1024 + 256 * kind + slots[t] * 16 + 4 * g + 2 * (what - 1)
            v = chunk[off:off + 2].view(np.uint16)
            v[0] = v[0] + 1 if v[0] & 0x7FFF else v[0]
        mask[t, h] = True
    return pg, mask


def test_bound_holds_for_planted_record_changes():
    oracle.build()
    c = synth.build_case(synth.workload("decode8k", 0, 1 / 64), 0)
    pool_ref, _, _ = ph.oracle_case(c)
    rng = np.random.default_rng(7)
    for trial in range(3):
        pg, mask = _perturb(pool_ref, c, rng, 40)
        bound = ph.e2e_row_bounds(c, pool_ref, pg,
                                  [(c["cu_ctx"].numpy(), c["pos0_ctx"].numpy(), mask)])
        ref = ph.oracle_decode(c, pool_ref)
        new = ph.oracle_decode(c, pg)
        diff = np.abs(new - ref).max(axis=2)
        assert np.all(diff <= bound * (1 + 1e-9) + 1e-12), trial
        # the bound is tight enough to be a real check: within 20x of the
        # actual change where something changed
        moved = diff > 0
        assert moved.any()
        assert np.median(bound[moved] / diff[moved]) < 20.0
        # rows of (sequence, KV head) groups with no changed record get no slack
        cu = c["cu_ctx"].numpy()
        touched = np.zeros(bound.shape, bool)
        for t, h in np.argwhere(mask):
            b = int(np.searchsorted(cu, t, side="right") - 1)
            touched[b, 4 * h:4 * h + 4] = True
        assert np.all(bound[~touched] == 0)
        assert np.all(diff[~touched] == 0)
        print(f"trial {trial}: median bound/change {np.median(bound[moved] / diff[moved]):.2f}")
