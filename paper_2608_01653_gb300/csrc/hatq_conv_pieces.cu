// The convolution kernels whose 64-wide activation blocks arrive as two
// 32-channel TMA boxes (layers with c_in % 64 == 32), built as their own
// translation unit so that the two kernel families compile in parallel.
#define HATQ_CONV_PIECES 1
#include "hatq_conv.cu"
