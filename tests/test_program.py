"""Spec strings the plan runner writes (host logic, no GPU)."""
from paper_2603_08957_gb300 import program


def test_cased_and_einsum_spec():
    assert program.cased("fab", "a") == "fAb"
    assert program.einsum_spec("fab", "a", "abcd", "ac", "cdf", "c") == "fAb,AbCd->Cdf"


def test_repartition_spec():
    # promote f, keep a: keys f, a in label order, written as the input letters
    assert program.repartition_spec("fab", "a", "fa") == "fAb->fA|b"
    # demote everything
    assert program.repartition_spec("ab", "ab", "") == "AB->|AB"
    # rows to columns
    assert program.repartition_spec("ki", "k", "i") == "Ki->i|K"


class _Rel:
    def __init__(self, name):
        self.name, self.destroyed = name, False

    def destroy(self):
        assert not self.destroyed, f"{self.name} destroyed twice"
        self.destroyed = True


class _Ctx:
    """Records the calls the runner makes; fails on a destroyed operand."""

    def __init__(self):
        self.calls = []
        self.made = []

    def _use(self, *rels):
        for r in rels:
            assert not r.destroyed, f"{r.name} used after destroy"

    def einsum(self, spec, *ops, **kw):
        self._use(*ops)
        self.calls.append(("einsum", spec))
        self.made.append(_Rel(spec))
        return self.made[-1]

    def repartition(self, spec, rel):
        self._use(rel)
        self.calls.append(("repartition", spec))
        self.made.append(_Rel(spec))
        return self.made[-1]

    def drop_zero_tiles(self, rel):
        self._use(rel)
        self.made.append(_Rel("nz:" + rel.name))
        return self.made[-1]


def test_execute_dag_reuses_a_result_and_frees_it_after_its_last_use():
    # T = X Y read by two heads, the second in another split; O2 also reads X again
    verts = [{"labels": "fa"}, {"labels": "ab"}, {"labels": "fb", "left": 0, "right": 1},
             {"labels": "fg"}, {"labels": "bg", "left": 2, "right": 3},
             {"labels": "bf", "left": 2, "right": 0}]
    ups = ["a", "a", ("b", "a", "a"), "", ("b", "b", ""), ("", "", "")]
    ctx = _Ctx()
    inputs = {0: _Rel("X"), 1: _Rel("Y"), 3: _Rel("Z")}
    out = program.execute_dag(ctx, verts, ups, inputs)
    assert sorted(out) == [4, 5] and not any(r.destroyed for r in out.values())
    assert not any(r.destroyed for r in inputs.values())
    kinds = [c[0] for c in ctx.calls]
    assert kinds.count("einsum") == 3
    # T read in split "" by vertex 5 (produced in "b"), X read in "" (stored in "a")
    assert ("repartition", "fB->|fB") in ctx.calls and ("repartition", "fA->|fA") in ctx.calls
    assert ctx.calls[-1] == ("einsum", "fb,fa->bf")
    # every relation the runner made is freed, except the outputs
    assert all(r.destroyed for r in ctx.made if all(r is not o for o in out.values()))


def test_execute_dag_one_result_as_both_operands():
    verts = [{"labels": "ab"}, {"labels": "ab"}, {"labels": "ab", "left": 0, "right": 1},
             {"labels": "a", "left": 2, "right": 2}]
    ups = ["a", "a", ("a", "a", "a"), ("a", "a", "")]
    ctx = _Ctx()
    out = program.execute_dag(ctx, verts, ups, {0: _Rel("A"), 1: _Rel("B")})
    assert list(out) == [3]
    assert ("repartition", "Ab->|Ab") in ctx.calls
    assert all(r.destroyed for r in ctx.made if r is not out[3])
