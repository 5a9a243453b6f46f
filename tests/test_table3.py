"""The paper's efficiency table (Table 3) reproduced from closed forms, and
the byte model the benchmark uses checked against it.

* PRCR's revisit costs 3 d_model FLOPs per (token, layer): a rotation pair
  takes 2 multiplies and an add per output element, 3 per element as the
  paper counts, over the model width. Reproduces 14.16 M ... 125.83 M.
* The raw visual store adds K and V in bf16 for every image token, layer and
  KV head: 768 x n_layers x n_kv_heads x head_dim x 2 x 2 bytes, which is
  the 108 / 192 MB printed (in MiB).
* The rebind step the kernels run moves 8 head_dim bytes per (token, layer,
  KV head) (read K and V raw, write K and V): the paper-shape workloads'
  algorithmic bytes equal that at K = 32 and 128.
"""
import os

import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "table3_efficiency.txt")


def _rows():
    out = []
    for line in open(GOLDEN):
        if line.strip() and not line.startswith("#"):
            f = line.split()
            out.append((f[0], int(f[1]), int(f[2]), int(f[3]), int(f[4]), int(f[5]), float(f[6]),
                        int(f[7])))
    return out


@pytest.mark.parametrize("row", _rows(), ids=lambda r: f"{r[0]}-K{r[5]}")
def test_table3_flops_and_memory(row):
    model, d_model, n_layers, n_kv, head_dim, K, flops_printed, mem_printed = row
    flops = 3 * d_model * n_layers * K
    assert round(flops / 1e6, 2) == round(flops_printed / 1e6, 2)
    extra = 768 * n_layers * n_kv * head_dim * 2 * 2
    assert round(extra / 2 ** 20) == mem_printed


@pytest.mark.parametrize("name,K", [("paper-8b-k32", 32), ("paper-8b-k128", 128)])
def test_paper_workloads_move_the_modelled_bytes(name, K):
    from workloads import get, make_batch
    wl = get(name)
    batch = make_batch(wl, device="cpu")
    assert batch.total_k == K and wl.n_tokens == 768
    assert batch.algorithmic_bytes() == K * wl.n_layers * wl.n_kv_heads * wl.head_dim * 8
