// ssd_wstream_kernel instantiations with the SILU epilogue (imitation network FC1), M = 1..16 rows (one per batched request).
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_16(silu, ssd::Epi::SILU)
