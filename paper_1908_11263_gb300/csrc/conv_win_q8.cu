// Window-kernel instantiations for INT-8 layers (fp16 staging).
#define QNN_WIN_BITS 8
#include "conv_win_inst.cuh"
