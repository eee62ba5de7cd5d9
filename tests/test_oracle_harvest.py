"""Pins for the reference harvest: cases worked by hand from the rule in
Section 3.5 (cut at the last closed tag, first 5 atoms, empty branches
omitted, nothing harvested -> nothing appended)."""
from oracle.harvest import harvest, harvest_branch

O, C = 1, 2  # open / close tag ids


def test_unfinished_unit_is_discarded():
    s = [O, 10, 11, C, O, 12]                   # second thought was cut off
    ids, src, n = harvest([s], O, C)
    assert ids == [O, 10, 11, C] and n == [1]
    assert src == [(0, 0), (0, 1), (0, 2), (0, 3)]


def test_first_five_atoms_are_kept():
    s = []
    for k in range(7):
        s += [O, 100 + k, C]
    ids, _, n = harvest([s], O, C)
    assert n == [5]
    assert ids == [O, 100, C, O, 101, C, O, 102, C, O, 103, C, O, 104, C]


def test_branch_without_a_completed_unit_is_omitted():
    ids, src, n = harvest([[O, 5, 6], [O, 7, C], [], [9, 9]], O, C)
    assert ids == [O, 7, C] and n == [0, 1, 0, 0]
    assert src == [(1, 0), (1, 1), (1, 2)]


def test_nothing_harvested_appends_nothing():
    assert harvest([[O, 3], [4, C], []], O, C) == ([], [], [0, 0, 0])


def test_branches_concatenate_in_order():
    ids, src, n = harvest([[O, 10, C], [O, 20, C, O, 30, C]], O, C)
    assert ids == [O, 10, C, O, 20, C, O, 30, C] and n == [1, 2]
    assert [b for b, _ in src] == [0, 0, 0, 1, 1, 1, 1, 1, 1]


def test_text_outside_atoms_and_stray_close_are_dropped():
    s = [7, C, 8, O, 10, C, 9, 9, C]
    assert harvest_branch(s, O, C, 5) == [[3, 4, 5]]


def test_reopen_restarts_the_atom():
    s = [O, 10, O, 11, 12, C]
    assert harvest_branch(s, O, C, 5) == [[2, 3, 4, 5]]


def test_cap_zero_and_empty_atom():
    assert harvest_branch([O, C, O, 5, C], O, C, 0) == []
    assert harvest_branch([O, C], O, C, 5) == [[0, 1]]     # "<thought></thought>" is a unit
