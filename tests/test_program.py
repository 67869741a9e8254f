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
