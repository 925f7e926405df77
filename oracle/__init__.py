"""CPU oracle (test infrastructure only; see presto_oracle.py)."""
