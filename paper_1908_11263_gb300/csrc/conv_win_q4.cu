// Window-kernel instantiations for INT-4 layers (e4m3 staging).
#define QNN_WIN_BITS 4
#include "conv_win_inst.cuh"
