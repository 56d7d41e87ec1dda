// ssd_wstream_kernel instantiations with the ARGMAX epilogue, M = 1..9 rows.
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_9(head, ssd::Epi::ARGMAX)
