// Window-kernel instantiations for INT-2 layers (e4m3 staging).
#define QNN_WIN_BITS 2
#include "conv_win_inst.cuh"
