"""CPU oracle for the three-stage attention path -- test infrastructure only (see oracle.py)."""
