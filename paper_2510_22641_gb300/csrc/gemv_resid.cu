// ssd_wstream_kernel instantiations with the RESID epilogue, M = 1..16 rows.
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_16(resid, ssd::Epi::RESID)
