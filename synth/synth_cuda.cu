// Device build of the seeded synthetic input generator (definition in
// synth_gen.h).  Fills workload inputs directly in HBM so that tens of GB of
// K/V never cross the host link; the host build regenerates any slice
// bit-for-bit for the CPU oracle.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "synth_gen.h"

namespace {

__global__ void syn_fill_tokens_kernel(uint64_t seed, int dtype, float scale, uint32_t tag, int64_t n_tok,
                                       const int32_t* __restrict__ tok_t, const int32_t* __restrict__ tok_s, int H,
                                       int d, uint16_t* __restrict__ out) {
  const int64_t total = n_tok * (int64_t)H * d;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int e = (int)(i % d);
    const int64_t r = i / d;
    const int h = (int)(r % H);
    const int64_t tok = r / H;
    const float c = (float)syn_centred_sum(seed, tag, (uint32_t)tok_t[tok], (uint32_t)tok_s[tok],
                                           (uint32_t)(h * 1024 + e));
    const float x = __fmul_rn(c, scale);
    uint16_t bits;
    if (dtype == SYN_DTYPE_BF16) {
      bits = __bfloat16_as_ushort(__float2bfloat16_rn(x));
    } else {
      bits = __half_as_ushort(__float2half_rn(x));
    }
    out[i] = bits;
  }
}

}  // namespace

extern "C" {

// Same contract as the host syn_fill_tokens: out[(tok*H + h)*d + e], tok_t and
// tok_s are device arrays of n_tok entries.  Returns a cudaError_t value.
int syn_cuda_fill_tokens(uint64_t seed, int dtype, float scale, uint32_t tag, int64_t n_tok, const int32_t* tok_t,
                         const int32_t* tok_s, int H, int d, uint16_t* out, cudaStream_t stream) {
  if (n_tok <= 0) return 0;
  const int64_t total = n_tok * (int64_t)H * d;
  int64_t blocks = (total + 255) / 256;
  if (blocks > 152 * 64) blocks = 152 * 64;
  syn_fill_tokens_kernel<<<(unsigned)blocks, 256, 0, stream>>>(seed, dtype, scale, tag, n_tok, tok_t, tok_s, H, d,
                                                              out);
  return (int)cudaGetLastError();
}

}  // extern "C"
