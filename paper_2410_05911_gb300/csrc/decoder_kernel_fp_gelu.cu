// decoder_kernel_fp_gelu.cu -- instantiations of the decoder kernel with the GELU feed-forward
// activation and full-precision (bf16) linears (the ECCT baseline, Sec. 3).
#include "decoder_kernel.cuh"

namespace aecct {

template cudaError_t launch_decode<32, 0, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, 0, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 0, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<32, 1, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, 1, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 1, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 2, 1, 1>(const DecodeParams &, cudaStream_t);
template cudaError_t prepare_decode_kernel<32, 0, 1, 1>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<64, 0, 1, 1>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 0, 1, 1>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<32, 1, 1, 1>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<64, 1, 1, 1>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 1, 1, 1>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 2, 1, 1>(int, uint32_t, int *);

}  // namespace aecct
