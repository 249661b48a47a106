"""Host logic of the multi-cycle driver (no GPU): paths of tree nodes and the
k-token contexts they are looked up with."""
import torch

from paper_2609_21827_gb300 import cycles


def test_paths_and_contexts_on_a_hand_built_tree():
    # root 0; children 1 (token 5) and 2 (token 6); node 3 (token 7) under node 1
    tok = torch.tensor([[-1, 5, 6, 7]])
    par = torch.tensor([[-1, 0, 0, 1]])
    path, length = cycles._paths(tok, par, torch.tensor([[0, 1, 2, 3]]), 3)
    assert path.tolist() == [[[0, 0, 0], [0, 0, 5], [0, 0, 6], [0, 5, 7]]]
    assert length.tolist() == [[0, 1, 1, 2]]
    win = torch.tensor([[1, 2]])
    assert cycles._contexts(win, path, length, 2).tolist() == [[[1, 2], [2, 5], [2, 6], [5, 7]]]
    assert cycles._contexts(torch.tensor([[1, 2, 3]]), path, length, 3).tolist() == \
        [[[1, 2, 3], [2, 3, 5], [2, 3, 6], [3, 5, 7]]]


def test_kgram_rows_are_indexed_by_the_last_k_tokens():
    V, k = 4, 2
    table = torch.arange(V ** k * V, dtype=torch.float32).reshape(V ** k, V)
    lm = cycles.KGramLM(table, V, k)
    ctx = torch.tensor([[3, 1], [0, 2]])
    assert torch.equal(lm.rows(ctx), table[torch.tensor([3 * V + 1, 0 * V + 2])])
