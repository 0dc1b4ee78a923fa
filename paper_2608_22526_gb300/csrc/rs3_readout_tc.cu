// rs3_readout_tc.cu -- tensor-core (tcgen05 / TMEM / TMA) readout for bf16.
#include "rs3_readout_common.cuh"

bool rs3_tc_supported(int d) { (void)d; return false; }
int rs3_tc_block_n(int d) { (void)d; return 128; }
rs3_status rs3_launch_tc_readout(const ReadoutArgs &a, cudaStream_t st)
{
    (void)a; (void)st;
    return RS3_EUNSUPPORTED;
}
