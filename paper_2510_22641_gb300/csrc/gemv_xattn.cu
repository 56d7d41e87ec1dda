// ssd_wstream_kernel instantiations with the XATTN epilogue (cross-q projection + folded
// cross-attention of the encoder-decoder model), M = 1..16 rows.
#include "gemv_launch.cuh"
SSD_DEFINE_GEMV_16(xattn, ssd::Epi::XATTN)
