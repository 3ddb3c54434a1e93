// decoder_kernel.cu -- instantiations of the decoder kernel with the ReLU feed-forward activation
// (Sec. 4 item 4), AAP linears (Sec. 4.1).
#include "decoder_kernel.cuh"

namespace aecct {

template cudaError_t launch_decode<32, 0, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, 0, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 0, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<32, 1, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<64, 1, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 1, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t launch_decode<128, 2, 0, 0>(const DecodeParams &, cudaStream_t);
template cudaError_t prepare_decode_kernel<32, 0, 0, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<64, 0, 0, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 0, 0, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<32, 1, 0, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<64, 1, 0, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 1, 0, 0>(int, uint32_t, int *);
template cudaError_t prepare_decode_kernel<128, 2, 0, 0>(int, uint32_t, int *);

}  // namespace aecct
