"""Reference thought harvest -- test infrastructure only.

Section 3.5 of the paper: when the observation arrives every branch is
cancelled and its output buffer harvested as it stands.  The buffer is cut
at its last closed </thought> tag (an unfinished unit is discarded), the
surviving thoughts are capped at 5 per branch, a branch that completed no
unit is left out, and the harvested thoughts are appended (in branch order)
after the observation.  With nothing harvested the turn is plain ReAct.

At the token level this project reads that as follows (the paper states it
on text):
* an atom is the span from an open-tag token through the next close-tag
  token, both tags included;
* an open tag inside an unfinished atom restarts the atom there (the
  unfinished part is discarded); a close tag with no open atom is ignored;
* tokens outside atoms are not harvested;
* "capped at 5" keeps the first 5 completed atoms of the branch.
"""


def harvest_branch(ids, open_id, close_id, cap):
    """Completed atoms of one branch, each as a list of token positions."""
    atoms = []
    start = None
    for i, t in enumerate(ids):
        if len(atoms) == cap:
            break
        if t == open_id:
            start = i
        elif t == close_id and start is not None:
            atoms.append(list(range(start, i + 1)))
            start = None
    return atoms


def harvest(streams, open_id, close_id, cap=5):
    """streams: list of per-branch token-id lists (generated so far).

    Returns (ids, src, atoms_per_branch): the concatenated harvested token
    ids, for each harvested token its (branch, position) source, and the
    number of atoms kept per branch.
    """
    ids, src, counts = [], [], []
    for b, stream in enumerate(streams):
        atoms = harvest_branch(stream, open_id, close_id, cap)
        counts.append(len(atoms))
        for atom in atoms:
            for pos in atom:
                ids.append(stream[pos])
                src.append((b, pos))
    return ids, src, counts
