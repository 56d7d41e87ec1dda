// ssd_wstream_kernel instantiations with the ARGMAX epilogue, M = 1..16 rows.
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_16(head, ssd::Epi::ARGMAX)
