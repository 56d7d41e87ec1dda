// ssd_wstream_kernel instantiation with the SILU epilogue (imitation network FC1), M = 1.
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_1(silu, ssd::Epi::SILU)
