// Kernels of the Wan-shaped model around the blocks: the timestep sinusoid, small
// matrix-vector products of the timestep MLP, and the patch (1 x 2 x 2) layout changes
// between the latent video [C, F, H, W] and the token rows [N, 4 C].  The patch embedding
// and the output head are GEMMs on K4.  All of this is memory- or latency-bound and tiny
// next to the blocks (a few MB per step).
#include "kernels.cuh"

namespace dfs {
namespace {

// e[i] = cos(t w_i), e[half + i] = sin(t w_i) with w_i = 10000^(-i / half); angles in double
__global__ void timestep_freq_kernel(float* __restrict__ e, double t, int half) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= half) return;
  const double w = exp(-log(10000.0) * static_cast<double>(i) / static_cast<double>(half));
  const double a = t * w;
  e[i] = static_cast<float>(cos(a));
  e[half + i] = static_cast<float>(sin(a));
}

// One warp per output row: out[r] = sum_c W[r, c] f(in[c]) + b[r], f = SiLU or identity.
__global__ void gemv_kernel(float* __restrict__ out_f32, bf16* __restrict__ out_bf16, const bf16* __restrict__ W,
                            const bf16* __restrict__ b, const float* __restrict__ in, int rows, int cols,
                            int silu_in) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows) return;
  const uint4* w4 = reinterpret_cast<const uint4*>(W + static_cast<long long>(warp) * cols);
  float acc = 0.f;
  for (int v = lane; v < cols / 8; v += 32) {
    float w[8];
    unpack_bf16x8(__ldg(w4 + v), w);
    const float4 x0 = __ldg(reinterpret_cast<const float4*>(in) + 2 * v);
    const float4 x1 = __ldg(reinterpret_cast<const float4*>(in) + 2 * v + 1);
    float x[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
    if (silu_in) {
#pragma unroll
      for (int i = 0; i < 8; ++i) x[i] = x[i] / (1.f + __expf(-x[i]));
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) acc = fmaf(w[i], x[i], acc);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
  if (lane == 0) {
    acc += bf16_to_f32(b[warp]);
    if (out_f32) out_f32[warp] = acc;
    if (out_bf16) out_bf16[warp] = __float2bfloat16_rn(acc);
  }
}

// Thread (n, c): the 2 x 2 patch of channel c under token n -> tok[n, 4c .. 4c + 3]
// (feature c*4 + dy*2 + dx), token n = (f * gh + y) * gw + x.
__global__ void patchify_kernel(bf16* __restrict__ tok, const bf16* __restrict__ lat, int C, int F, int gh, int gw) {
  const long long N = static_cast<long long>(F) * gh * gw;
  const long long total = N * C;
  const int W = 2 * gw;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long n = i / C;
    const int c = static_cast<int>(i - n * C);
    const int x = static_cast<int>(n % gw);
    const long long fy = n / gw;
    const int y = static_cast<int>(fy % gh);
    const int f = static_cast<int>(fy / gh);
    const bf16* src = lat + ((static_cast<long long>(c) * F + f) * (2 * gh) + 2 * y) * W + 2 * x;
    const uint32_t r0 = *reinterpret_cast<const uint32_t*>(src);      // dy = 0: dx = 0, 1
    const uint32_t r1 = *reinterpret_cast<const uint32_t*>(src + W);  // dy = 1
    *reinterpret_cast<uint2*>(tok + n * (4LL * C) + 4 * c) = make_uint2(r0, r1);
  }
}

// Thread (n, c): out[c, f, 2y + dy, 2x + dx] = (base ? base[...] : 0) + dt * tok[n, 4c + 2dy + dx]
// (fp32 arithmetic, bf16 storage; out may alias base).
__global__ void unpatchify_kernel(bf16* out, const bf16* base, const bf16* __restrict__ tok, float dt, int C, int F,
                                  int gh, int gw) {
  const long long N = static_cast<long long>(F) * gh * gw;
  const long long total = N * C;
  const int W = 2 * gw;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const long long n = i / C;
    const int c = static_cast<int>(i - n * C);
    const int x = static_cast<int>(n % gw);
    const long long fy = n / gw;
    const int y = static_cast<int>(fy % gh);
    const int f = static_cast<int>(fy / gh);
    const long long o = ((static_cast<long long>(c) * F + f) * (2 * gh) + 2 * y) * W + 2 * x;
    const uint2 v = *reinterpret_cast<const uint2*>(tok + n * (4LL * C) + 4 * c);
    const float v00 = __uint_as_float(v.x << 16), v01 = __uint_as_float(v.x & 0xFFFF0000u);
    const float v10 = __uint_as_float(v.y << 16), v11 = __uint_as_float(v.y & 0xFFFF0000u);
    float b00 = 0.f, b01 = 0.f, b10 = 0.f, b11 = 0.f;
    if (base) {
      const uint32_t r0 = *reinterpret_cast<const uint32_t*>(base + o);
      const uint32_t r1 = *reinterpret_cast<const uint32_t*>(base + o + W);
      b00 = __uint_as_float(r0 << 16); b01 = __uint_as_float(r0 & 0xFFFF0000u);
      b10 = __uint_as_float(r1 << 16); b11 = __uint_as_float(r1 & 0xFFFF0000u);
    }
    *reinterpret_cast<uint32_t*>(out + o) = pack_bf16x2(fmaf(dt, v00, b00), fmaf(dt, v01, b01));
    *reinterpret_cast<uint32_t*>(out + o + W) = pack_bf16x2(fmaf(dt, v10, b10), fmaf(dt, v11, b11));
  }
}

int blocks_for(long long work, int threads) {
  long long g = (work + threads - 1) / threads;
  const long long cap = 8LL * current_device_sms();
  if (g > cap) g = cap;
  return static_cast<int>(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t launch_timestep_freq(float* e, double t, int dim, cudaStream_t s) {
  const int half = dim / 2;
  timestep_freq_kernel<<<(half + 127) / 128, 128, 0, s>>>(e, t, half);
  return cudaGetLastError();
}

cudaError_t launch_gemv(float* out_f32, bf16* out_bf16, const bf16* W, const bf16* b, const float* in, int rows,
                        int cols, int silu_in, cudaStream_t s) {
  if (cols % 8 != 0) return cudaErrorInvalidValue;
  gemv_kernel<<<(rows * 32 + 255) / 256, 256, 0, s>>>(out_f32, out_bf16, W, b, in, rows, cols, silu_in);
  return cudaGetLastError();
}

cudaError_t launch_patchify(bf16* tok, const bf16* lat, int C, int F, int gh, int gw, cudaStream_t s) {
  const long long work = static_cast<long long>(F) * gh * gw * C;
  patchify_kernel<<<blocks_for(work, 256), 256, 0, s>>>(tok, lat, C, F, gh, gw);
  return cudaGetLastError();
}

cudaError_t launch_unpatchify(bf16* out, const bf16* base, const bf16* tok, float dt, int C, int F, int gh, int gw,
                              cudaStream_t s) {
  const long long work = static_cast<long long>(F) * gh * gw * C;
  unpatchify_kernel<<<blocks_for(work, 256), 256, 0, s>>>(out, base, tok, dt, C, F, gh, gw);
  return cudaGetLastError();
}

}  // namespace dfs
