"""fp64 CPU oracle for MeqMuon (test infrastructure; see meqmuon.py)."""
