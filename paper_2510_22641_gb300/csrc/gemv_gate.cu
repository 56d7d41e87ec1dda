// ssd_wstream_kernel instantiations with the GATE_SILU epilogue, M = 1..16 rows.
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_16(gate, ssd::Epi::GATE_SILU)
