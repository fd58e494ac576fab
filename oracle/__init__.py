"""CPU oracle for the PolyQ hot path.  Test infrastructure only: the product
library never imports it."""
