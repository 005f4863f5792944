// K9: compaction of the kept tokens (Sec. 3.2: the kept set is the visual
// input of the subsequent decoding).  One block per kept row; 16-byte vector
// copies of the feature row, plus its position and frame.
#include "common.cuh"

namespace cp {

__global__ void __launch_bounds__(128) k_gather(const uint4* __restrict__ feats, int64_t row_vecs,
                                                const float* __restrict__ pos,
                                                const int32_t* __restrict__ frame, int N,
                                                const int64_t* __restrict__ kept, int K,
                                                uint4* __restrict__ out, float* __restrict__ pos_out,
                                                int32_t* __restrict__ frame_out, int32_t* status) {
  const int k = blockIdx.x, b = blockIdx.y;
  const int64_t idx = kept[(size_t)b * K + k];
  if (idx < 0 || idx >= N) {
    if (threadIdx.x == 0 && status) set_status(status, CP_EINVAL);
    return;
  }
  const uint4* src = feats + ((size_t)b * N + (size_t)idx) * row_vecs;
  uint4* dst = out + ((size_t)b * K + k) * row_vecs;
  for (int64_t i = threadIdx.x; i < row_vecs; i += blockDim.x) dst[i] = __ldg(src + i);
  if (threadIdx.x < 3 && pos_out)
    pos_out[((size_t)b * K + k) * 3 + threadIdx.x] = pos[((size_t)b * N + idx) * 3 + threadIdx.x];
  if (threadIdx.x == 3 && frame_out) frame_out[(size_t)b * K + k] = frame[(size_t)b * N + idx];
}

int launch_gather(const void* feats, int dtype, const float* pos, const int32_t* frame, int64_t B,
                  int64_t N, int64_t D, const int64_t* kept, int64_t K, void* feats_out,
                  float* pos_out, int32_t* frame_out, int32_t* status, cudaStream_t s) {
  const int64_t row_bytes = D * (dtype == CP_BF16 ? 2 : 4);
  dim3 grid((unsigned)K, (unsigned)B);
  k_gather<<<grid, 128, 0, s>>>((const uint4*)feats, row_bytes / 16, pos, frame, (int)N, kept,
                                (int)K, (uint4*)feats_out, pos_out, frame_out, status);
  return last_launch_status();
}

}  // namespace cp
