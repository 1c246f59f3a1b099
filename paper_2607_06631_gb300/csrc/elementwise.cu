// Memory-bound kernels of the block: weight compaction (K1), adaLN LayerNorm + modulate
// and affine LayerNorm (K2 / K7), QK RMSNorm + 3D RoPE (K3), the modulation GEMV (K6),
// bias-only residual branches and the Euler update (K8).  All move 16-byte vectors and
// reduce with warp shuffles.
#include <atomic>

#include "kernels.cuh"

namespace dfs {
namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over the whole CTA (blockDim.x a multiple of 32, at most 1024); every thread gets it.
__device__ __forceinline__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
  __syncthreads();
  if (l == 0) red[w] = v;
  __syncthreads();
  float t = (l < nw) ? red[l] : 0.f;
  return warp_sum(t);
}

// Two sums over the whole CTA in one reduction (one pair of barriers); every thread gets both.
__device__ __forceinline__ float2 block_sum2(float a, float b, float (*red)[32]) {
  a = warp_sum(a);
  b = warp_sum(b);
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31, nw = blockDim.x >> 5;
  __syncthreads();
  if (l == 0) {
    red[0][w] = a;
    red[1][w] = b;
  }
  __syncthreads();
  return make_float2(warp_sum(l < nw ? red[0][l] : 0.f), warp_sum(l < nw ? red[1][l] : 0.f));
}

// Two sums over each group of TPR consecutive threads (TPR a multiple of 32 dividing blockDim.x),
// every thread getting its group's sums.  Its two barriers involve the whole CTA.
template <int TPR>
__device__ __forceinline__ float2 group_sum2(float a, float b, float (*red)[32]) {
  a = warp_sum(a);
  b = warp_sum(b);
  if constexpr (TPR == 32) return make_float2(a, b);  // one warp per group: no barrier
  constexpr int kWarps = TPR / 32;
  const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
  __syncthreads();
  if (l == 0) {
    red[0][w] = a;
    red[1][w] = b;
  }
  __syncthreads();
  const int g0 = (w / kWarps) * kWarps;
  float ta = 0.f, tb = 0.f;
#pragma unroll
  for (int i = 0; i < kWarps; ++i) {
    ta += red[0][g0 + i];
    tb += red[1][g0 + i];
  }
  return make_float2(ta, tb);
}

// ------------------------------------------------------------------ K1 compaction

__global__ void gather_rows_kernel(bf16* __restrict__ dst, long long ld_dst, const bf16* __restrict__ src,
                                   long long ld_src, const int* __restrict__ rows, int n_rows, int vec_per_row) {
  const long long total = static_cast<long long>(n_rows) * vec_per_row;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int r = static_cast<int>(i / vec_per_row);
    const int v = static_cast<int>(i - static_cast<long long>(r) * vec_per_row);
    const uint4 x = __ldg(reinterpret_cast<const uint4*>(src + rows[r] * ld_src) + v);
    reinterpret_cast<uint4*>(dst + r * ld_dst)[v] = x;
  }
}

__global__ void gather_segs_kernel(bf16* __restrict__ dst, long long ld_dst, const bf16* __restrict__ src,
                                   long long ld_src, const int* __restrict__ seg, int n_seg, int n_rows) {
  const long long total = static_cast<long long>(n_rows) * n_seg;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int r = static_cast<int>(i / n_seg);
    const int j = static_cast<int>(i - static_cast<long long>(r) * n_seg);
    const uint4 x = __ldg(reinterpret_cast<const uint4*>(src + r * ld_src) + seg[j]);
    reinterpret_cast<uint4*>(dst + r * ld_dst)[j] = x;
  }
}

// Grid-stride kernels get at most 16 CTAs per SM.
int grid_for(long long work, int threads) {
  long long g = (work + threads - 1) / threads;
  const long long cap = 16LL * current_device_sms();
  if (g > cap) g = cap;
  if (g < 1) g = 1;
  return static_cast<int>(g);
}

// ------------------------------------------------------------------ K6 modulation GEMV

__global__ void modulation_kernel(float* __restrict__ out, const bf16* __restrict__ W, const bf16* __restrict__ b,
                                  const bf16* __restrict__ e, const bf16* __restrict__ t, int rows, int cols) {
  const int warp = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= rows) return;
  const uint4* w4 = reinterpret_cast<const uint4*>(W + static_cast<long long>(warp) * cols);
  const uint4* t4 = reinterpret_cast<const uint4*>(t);
  float acc = 0.f;
  const int nv = cols / 8;
  // four 16-byte loads of W in flight per lane before their products are accumulated
  for (int v0 = lane; v0 < nv; v0 += 4 * 32) {
    uint4 wv[4], tv[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int v = v0 + 32 * u;
      if (v < nv) {
        wv[u] = __ldg(w4 + v);
        tv[u] = __ldg(t4 + v);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      if (v0 + 32 * u < nv) {
        float a[8], x[8];
        unpack_bf16x8(wv[u], a);
        unpack_bf16x8(tv[u], x);
#pragma unroll
        for (int i = 0; i < 8; ++i) acc = fmaf(a[i], x[i], acc);
      }
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) {
    float y = acc + bf16_to_f32(b[warp]);
    if (e != nullptr) y += bf16_to_f32(e[warp]);
    out[warp] = y;
  }
}

__global__ void add_table_kernel(float* out, const float* base, const bf16* e, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = base[i] + bf16_to_f32(e[i]);
}

// ------------------------------------------------------------------ K2 / K7 row LayerNorm


// A group of TPR threads per row, 256 / TPR rows per CTA (4 CTAs of 256 threads per SM), with
// the row held in registers (VPT 8-wide vectors per thread): the row is read from memory once.
// Narrow rows (the Wan-1.3B shape's 1536 columns) take 64-thread groups, so a CTA keeps four
// rows in flight.  Mean and variance come from one group reduction of two sums in the
// shifted-data form: sums of x - K and (x - K)^2 with K the row's first element, which keeps
// E[(x-K)^2] - E[x-K]^2 free of cancellation however large the row's mean.
template <bool F32IN>
__device__ __forceinline__ void load_vec8(const void* xv, long long off, float (&v)[8]) {
  if (F32IN) {
    const float4* p = reinterpret_cast<const float4*>(static_cast<const float*>(xv) + off);
    const float4 a = p[0], b = p[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  } else {
    unpack_bf16x8(*reinterpret_cast<const uint4*>(static_cast<const bf16*>(xv) + off), v);
  }
}

constexpr int kNormThreads = 256;

// Raw words of one 8-element vector of the input row: fp32 keeps 8 floats, bf16 keeps the 4
// packed words (half the registers, so more rows are in flight per SM).
template <bool F32IN>
struct RowVec {
  uint32_t w[F32IN ? 8 : 4];
};

template <bool F32IN>
__device__ __forceinline__ void load_raw8(const void* xv, long long off, RowVec<F32IN>& r) {
  if constexpr (F32IN) {
    const uint4* p = reinterpret_cast<const uint4*>(static_cast<const float*>(xv) + off);
    const uint4 a = p[0], b = p[1];
    r.w[0] = a.x; r.w[1] = a.y; r.w[2] = a.z; r.w[3] = a.w;
    r.w[4] = b.x; r.w[5] = b.y; r.w[6] = b.z; r.w[7] = b.w;
  } else {
    const uint4 a = *reinterpret_cast<const uint4*>(static_cast<const bf16*>(xv) + off);
    r.w[0] = a.x; r.w[1] = a.y; r.w[2] = a.z; r.w[3] = a.w;
  }
}

template <bool F32IN>
__device__ __forceinline__ void unpack_raw8(const RowVec<F32IN>& r, float (&v)[8]) {
  if constexpr (F32IN) {
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r.w[i]);
  } else {
    unpack_bf16x8(make_uint4(r.w[0], r.w[1], r.w[2], r.w[3]), v);
  }
}

template <bool F32IN, int VPT, int TPR>
__global__ void __launch_bounds__(kNormThreads, (F32IN ? 4 : 6) - (VPT > 5 ? 1 : 0)) row_norm_kernel(bf16* __restrict__ y, const void* __restrict__ xv,
                                                                     int rows, int cols, const float* __restrict__ mul,
                                                                     float mul_bias, const float* __restrict__ add,
                                                                     float eps) {
  __shared__ float red[2][32];
  constexpr int kRows = kNormThreads / TPR;
  const int t = threadIdx.x % TPR;
  const long long row = static_cast<long long>(blockIdx.x) * kRows + threadIdx.x / TPR;
  const bool live = row < rows;  // every thread still joins the group reduction's barriers
  const long long r0 = (live ? row : 0) * cols;
  const int nvec = cols >> 3;
  const float K = F32IN ? static_cast<const float*>(xv)[r0] : bf16_to_f32(static_cast<const bf16*>(xv)[r0]);
  RowVec<F32IN> raw[VPT];
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int c = t + k * TPR;
    if (c < nvec) load_raw8<F32IN>(xv, r0 + 8LL * c, raw[k]);
  }
  float s = 0.f, q = 0.f;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int c = t + k * TPR;
    if (c < nvec) {
      float v[8];
      unpack_raw8<F32IN>(raw[k], v);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float d = v[i] - K;
        s += d;
        q = fmaf(d, d, q);
      }
    }
  }
  const float2 sums = group_sum2<TPR>(s, q, red);
  const float ms = sums.x / cols;
  const float mean = K + ms;
  const float rstd = rsqrtf(fmaxf(sums.y / cols - ms * ms, 0.f) + eps);
  if (!live) return;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int c = t + k * TPR;
    if (c < nvec) {
      const float4* m4 = reinterpret_cast<const float4*>(mul) + 2 * c;
      const float4* a4 = reinterpret_cast<const float4*>(add) + 2 * c;
      const float4 m0 = __ldg(m4), m1 = __ldg(m4 + 1), a0 = __ldg(a4), a1 = __ldg(a4 + 1);
      const float mm[8] = {m0.x, m0.y, m0.z, m0.w, m1.x, m1.y, m1.z, m1.w};
      const float aa[8] = {a0.x, a0.y, a0.z, a0.w, a1.x, a1.y, a1.z, a1.w};
      float v[8], o[8];
      unpack_raw8<F32IN>(raw[k], v);
#pragma unroll
      for (int i = 0; i < 8; ++i) o[i] = fmaf((v[i] - mean) * rstd, mul_bias + mm[i], aa[i]);
      *reinterpret_cast<uint4*>(y + r0 + 8LL * c) = pack_bf16x8(o);
    }
  }
}

template <bool F32IN>
cudaError_t row_norm_vpt(bf16* y, const void* x, int rows, int cols, const float* mul, float mul_bias,
                         const float* add, float eps, cudaStream_t s) {
  const int nvec = cols / 8;
#define DFS_ROW_NORM(V, T)                                                                                    \
  row_norm_kernel<F32IN, V, T><<<(rows + kNormThreads / (T) - 1) / (kNormThreads / (T)), kNormThreads, 0, s>>>( \
      y, x, rows, cols, mul, mul_bias, add, eps)
  if (nvec <= 6 * 32) {  // up to 1536 columns: one warp per row, eight rows per CTA, no barrier
    switch ((nvec + 31) / 32) {
      case 1: DFS_ROW_NORM(1, 32); break;
      case 2: DFS_ROW_NORM(2, 32); break;
      case 3: DFS_ROW_NORM(3, 32); break;
      case 4: DFS_ROW_NORM(4, 32); break;
      case 5: DFS_ROW_NORM(5, 32); break;
      default: DFS_ROW_NORM(6, 32); break;
    }
  } else if (nvec <= 4 * 64) {  // up to 2048 columns: 64 threads per row, four rows per CTA
    switch ((nvec + 63) / 64) {
      case 1: DFS_ROW_NORM(1, 64); break;
      case 2: DFS_ROW_NORM(2, 64); break;
      case 3: DFS_ROW_NORM(3, 64); break;
      default: DFS_ROW_NORM(4, 64); break;
    }
  } else if (nvec <= 5 * 128) {  // up to 5120 columns: 128 threads per row
    switch ((nvec + 127) / 128) {
      case 3: DFS_ROW_NORM(3, 128); break;
      case 4: DFS_ROW_NORM(4, 128); break;
      default: DFS_ROW_NORM(5, 128); break;
    }
  } else if (nvec <= 4 * 256) {  // up to 8192 columns: one row per CTA
    switch ((nvec + 255) / 256) {
      case 3: DFS_ROW_NORM(3, 256); break;
      default: DFS_ROW_NORM(4, 256); break;
    }
  } else {
    return cudaErrorInvalidValue;  // more than 8192 columns
  }
#undef DFS_ROW_NORM
  return cudaGetLastError();
}

// ------------------------------------------------------------------ K3 QK RMSNorm + RoPE

constexpr int kQkThreads = 256;
constexpr int kQkMaxVec = 8;  // up to 256 * 8 * 8 = 16384 channels per row (q and k)

struct QkParams {
  bf16* buf;
  long long ld;
  int nq, nk;
  const bf16* gq;
  const bf16* gk;
  int head_dim, mode;
  float eps;
  int rope;
  RopeTables t;
};

// A group of TPR threads per token row, 256 / TPR rows per CTA (narrow rows, e.g. the
// Wan-1.3B shape's 3072 q + k channels, take 64-thread groups and four rows per CTA).  The row
// stays in registers as raw bf16 vectors (VPT 16-byte vectors per thread), so several rows per
// SM are in flight at once.  The rotation of the row's token (cos, sin per pair of a head, the
// same for every head) is built once per row in shared memory from the per-band tables while
// the row loads, and the q and k statistics share one reduction.
// CTAs per SM: six leave a thread about 40 registers, enough for up to five vectors of a
// 256-thread row (four of a narrower group, whose rotation table costs a few more); more
// vectors per thread take four or five CTAs per SM so that they stay in registers.
template <int VPT, int TPR>
constexpr int qk_min_blocks() {
  return VPT > 5 ? 4 : (VPT == 5 && TPR != 256) ? 5 : 6;
}

template <int VPT, int TPR>
__global__ void __launch_bounds__(kQkThreads, qk_min_blocks<VPT, TPR>()) qk_norm_rope_kernel(const QkParams p, int rows) {
  constexpr int kRows = kQkThreads / TPR;
  __shared__ float red[2][32];
  __shared__ float rcos[kRows][64], rsin[kRows][64];
  const int g = threadIdx.x / TPR, t = threadIdx.x % TPR;
  const long long row = static_cast<long long>(blockIdx.x) * kRows + g;
  const bool live = row < rows;  // every thread still joins the reductions' barriers
  bf16* base = p.buf + (live ? row : 0) * p.ld;
  const int nvq = p.nq >> 3, nv = (p.nq + p.nk) >> 3;
  const int vph = p.head_dim >> 3;  // vectors per head (8 or 16); divides 32
  uint4 raw[VPT];
  float hs[VPT];
  float sq = 0.f, sk = 0.f;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int c = t + k * TPR;
    if (c < nv) raw[k] = reinterpret_cast<const uint4*>(base)[c];
  }
  if (p.rope && t < (p.head_dim >> 1)) {
    const long long tok = live ? row : 0;
    const int hw = p.t.grid_h * p.t.grid_w;
    const int f = static_cast<int>(tok / hw);
    const int rem = static_cast<int>(tok - static_cast<long long>(f) * hw);
    const int yy = rem / p.t.grid_w, xx = rem - yy * p.t.grid_w;
    const int j = t;
    float cs, sn;
    if (j < p.t.p_t) {
      cs = __ldg(p.t.cos_t + f * p.t.p_t + j);
      sn = __ldg(p.t.sin_t + f * p.t.p_t + j);
    } else if (j < p.t.p_t + p.t.p_h) {
      const int jj = j - p.t.p_t;
      cs = __ldg(p.t.cos_h + yy * p.t.p_h + jj);
      sn = __ldg(p.t.sin_h + yy * p.t.p_h + jj);
    } else {
      const int jj = j - p.t.p_t - p.t.p_h;
      cs = __ldg(p.t.cos_w + xx * p.t.p_w + jj);
      sn = __ldg(p.t.sin_w + xx * p.t.p_w + jj);
    }
    rcos[g][j] = cs;
    rsin[g][j] = sn;
  }
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int c = t + k * TPR;
    float ss = 0.f;
    if (c < nv) {
      float v[8];
      unpack_bf16x8(raw[k], v);
#pragma unroll
      for (int i = 0; i < 8; ++i) ss = fmaf(v[i], v[i], ss);
      if (c < nvq) sq += ss; else sk += ss;
    }
    hs[k] = ss;
  }
  float rq = 0.f, rk = 0.f;
  if (p.mode == 0) {
    const float2 sums = group_sum2<TPR>(sq, sk, red);  // its barriers also publish the rotation table
    rq = p.nq > 0 ? rsqrtf(sums.x / p.nq + p.eps) : 0.f;
    rk = p.nk > 0 ? rsqrtf(sums.y / p.nk + p.eps) : 0.f;
  } else {
    // per head: the vph threads holding one head are consecutive lanes of one warp
#pragma unroll
    for (int k = 0; k < VPT; ++k) {
      float h = hs[k];
      for (int o = vph >> 1; o > 0; o >>= 1) h += __shfl_xor_sync(0xffffffffu, h, o);
      hs[k] = rsqrtf(h / p.head_dim + p.eps);
    }
    if (p.rope) __syncthreads();
  }
  if (!live) return;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int c = t + k * TPR;
    if (c < nv) {
      const bool is_q = c < nvq;
      const int ch0 = (is_q ? c : c - nvq) * 8;  // channel within the q or k part
      const float r = p.mode == 0 ? (is_q ? rq : rk) : hs[k];
      float v[8], gm[8], o[8];
      unpack_bf16x8(raw[k], v);
      unpack_bf16x8(__ldg(reinterpret_cast<const uint4*>(is_q ? p.gq : p.gk) + (ch0 >> 3)), gm);
#pragma unroll
      for (int i = 0; i < 8; ++i) o[i] = v[i] * r * gm[i];
      if (p.rope) {
        const int j0 = (ch0 % p.head_dim) >> 1;  // first rotation pair of this vector
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float cs = rcos[g][j0 + i], sn = rsin[g][j0 + i];
          const float a = o[2 * i], b = o[2 * i + 1];
          o[2 * i] = a * cs - b * sn;
          o[2 * i + 1] = a * sn + b * cs;
        }
      }
      reinterpret_cast<uint4*>(base)[c] = pack_bf16x8(o);
    }
  }
}

// ------------------------------------------------------------------ bias-only branches, Euler

template <bool RF32, bool OF32>
__global__ void bias_residual_kernel(void* out, const void* res, const float* gate, const bf16* bias, int rows,
                                     int cols) {
  const long long total = static_cast<long long>(rows) * cols;
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < total;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(i % cols);
    const float r = RF32 ? static_cast<const float*>(res)[i] : bf16_to_f32(static_cast<const bf16*>(res)[i]);
    const float g = gate ? gate[c] : 1.f;
    const float y = fmaf(g, bf16_to_f32(bias[c]), r);
    if (OF32) static_cast<float*>(out)[i] = y;
    else static_cast<bf16*>(out)[i] = __float2bfloat16_rn(y);
  }
}

__global__ void to_f32_kernel(float* out, const bf16* in, int n) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n) out[i] = bf16_to_f32(in[i]);
}

__global__ void wait_selftest_kernel(int* err) {
  __shared__ uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  // nobody arrives on `bar`: the bounded wait runs out and records the timeout
  if (threadIdx.x == 0) mbar_wait(&bar, 0, err);
  __syncthreads();
}

__global__ void euler_kernel(bf16* x, const bf16* v, float dt, long long nvec) {
  for (long long i = blockIdx.x * static_cast<long long>(blockDim.x) + threadIdx.x; i < nvec;
       i += static_cast<long long>(gridDim.x) * blockDim.x) {
    float a[8], b[8];
    unpack_bf16x8(reinterpret_cast<const uint4*>(x)[i], a);
    unpack_bf16x8(reinterpret_cast<const uint4*>(v)[i], b);
#pragma unroll
    for (int k = 0; k < 8; ++k) a[k] = fmaf(dt, b[k], a[k]);
    reinterpret_cast<uint4*>(x)[i] = pack_bf16x8(a);
  }
}

}  // namespace

cudaError_t launch_gather_rows(bf16* dst, long long ld_dst, const bf16* src, long long ld_src, const int* rows,
                               int n_rows, int cols, cudaStream_t s) {
  if (n_rows <= 0 || cols <= 0) return cudaSuccess;
  const long long work = static_cast<long long>(n_rows) * (cols / 8);
  gather_rows_kernel<<<grid_for(work, 256), 256, 0, s>>>(dst, ld_dst, src, ld_src, rows, n_rows, cols / 8);
  return cudaGetLastError();
}

cudaError_t launch_gather_segs(bf16* dst, long long ld_dst, const bf16* src, long long ld_src, const int* seg,
                               int n_seg, int n_rows, cudaStream_t s) {
  if (n_rows <= 0 || n_seg <= 0) return cudaSuccess;
  const long long work = static_cast<long long>(n_rows) * n_seg;
  gather_segs_kernel<<<grid_for(work, 256), 256, 0, s>>>(dst, ld_dst, src, ld_src, seg, n_seg, n_rows);
  return cudaGetLastError();
}

cudaError_t launch_modulation(float* out, const bf16* W, const bf16* b, const bf16* e, const bf16* t, int rows,
                              int cols, cudaStream_t s) {
  const int threads = 256;
  const int blocks = (rows * 32 + threads - 1) / threads;
  modulation_kernel<<<blocks, threads, 0, s>>>(out, W, b, e, t, rows, cols);
  return cudaGetLastError();
}

cudaError_t launch_add_table(float* out, const float* base, const bf16* e, int n, cudaStream_t s) {
  add_table_kernel<<<(n + 255) / 256, 256, 0, s>>>(out, base, e, n);
  return cudaGetLastError();
}

cudaError_t launch_row_norm(bf16* y, const void* x, int x_f32, int rows, int cols, const float* mul,
                            float mul_bias, const float* add, float eps, cudaStream_t s) {
  if (rows <= 0) return cudaSuccess;
  if (cols % 8 != 0 || cols <= 0) return cudaErrorInvalidValue;
  return x_f32 ? row_norm_vpt<true>(y, x, rows, cols, mul, mul_bias, add, eps, s)
               : row_norm_vpt<false>(y, x, rows, cols, mul, mul_bias, add, eps, s);
}

cudaError_t launch_qk_norm_rope(bf16* buf, long long ld, int rows, int nq, int nk, const bf16* gamma_q,
                                const bf16* gamma_k, int head_dim, int mode, float eps, const RopeTables* rope,
                                cudaStream_t s) {
  if (rows <= 0 || nq + nk <= 0) return cudaSuccess;
  if ((nq + nk) / 8 > kQkThreads * kQkMaxVec || nq % head_dim || nk % head_dim) return cudaErrorInvalidValue;
  QkParams p;
  p.buf = buf; p.ld = ld; p.nq = nq; p.nk = nk; p.gq = gamma_q; p.gk = gamma_k;
  p.head_dim = head_dim; p.mode = mode; p.eps = eps;
  p.rope = rope != nullptr;
  if (rope) p.t = *rope; else memset(&p.t, 0, sizeof(p.t));
  if (head_dim > 128) return cudaErrorInvalidValue;  // the rotation table holds 64 pairs
  // thread group per row: 64 threads up to 384 vectors (3072 q + k channels), 128 up to 512,
  // else 256; VPT vectors per thread
  const int nv = (nq + nk) / 8;
  const int tpr = nv <= 6 * 64 ? 64 : nv <= 4 * 128 ? 128 : 256;
  const int vpt = (nv + tpr - 1) / tpr;
  const int grid = (rows + kQkThreads / tpr - 1) / (kQkThreads / tpr);
#define DFS_QK(V, T) qk_norm_rope_kernel<V, T><<<grid, kQkThreads, 0, s>>>(p, rows)
  if (tpr == 64) {
    switch (vpt) {
      case 1: DFS_QK(1, 64); break;
      case 2: DFS_QK(2, 64); break;
      case 3: DFS_QK(3, 64); break;
      case 4: DFS_QK(4, 64); break;
      case 5: DFS_QK(5, 64); break;
      default: DFS_QK(6, 64); break;
    }
  } else if (tpr == 128) {
    switch (vpt) {
      case 1: DFS_QK(1, 128); break;
      case 2: DFS_QK(2, 128); break;
      case 3: DFS_QK(3, 128); break;
      default: DFS_QK(4, 128); break;
    }
  } else {
    switch (vpt) {
      case 1: DFS_QK(1, 256); break;
      case 2: DFS_QK(2, 256); break;
      case 3: DFS_QK(3, 256); break;
      case 4: DFS_QK(4, 256); break;
      case 5: DFS_QK(5, 256); break;
      case 6: DFS_QK(6, 256); break;
      default: DFS_QK(8, 256); break;
    }
  }
#undef DFS_QK
  return cudaGetLastError();
}

cudaError_t launch_bias_residual(void* out, int out_f32, const void* res, int res_f32, const float* gate,
                                 const bf16* bias, int rows, int cols, cudaStream_t s) {
  const long long total = static_cast<long long>(rows) * cols;
  if (total <= 0) return cudaSuccess;
  const int g = grid_for(total, 256);
  if (res_f32 && out_f32) bias_residual_kernel<true, true><<<g, 256, 0, s>>>(out, res, gate, bias, rows, cols);
  else if (res_f32) bias_residual_kernel<true, false><<<g, 256, 0, s>>>(out, res, gate, bias, rows, cols);
  else if (out_f32) bias_residual_kernel<false, true><<<g, 256, 0, s>>>(out, res, gate, bias, rows, cols);
  else bias_residual_kernel<false, false><<<g, 256, 0, s>>>(out, res, gate, bias, rows, cols);
  return cudaGetLastError();
}

cudaError_t launch_to_f32(float* out, const bf16* in, int n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  to_f32_kernel<<<(n + 255) / 256, 256, 0, s>>>(out, in, n);
  return cudaGetLastError();
}

cudaError_t launch_wait_selftest(int* err, cudaStream_t s) {
  wait_selftest_kernel<<<1, 32, 0, s>>>(err);
  return cudaGetLastError();
}

cudaError_t launch_euler(bf16* x, const bf16* v, float dt, long long n, cudaStream_t s) {
  if (n <= 0) return cudaSuccess;
  const long long nvec = n / 8;
  euler_kernel<<<grid_for(nvec, 256), 256, 0, s>>>(x, v, dt, nvec);
  return cudaGetLastError();
}

int current_device_sms() {
  constexpr int kMaxDevices = 64;
  static std::atomic<int> cache[kMaxDevices];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
  int n = dev < kMaxDevices ? cache[dev].load(std::memory_order_relaxed) : 0;
  if (n > 0) return n;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 1;
  if (dev < kMaxDevices) cache[dev].store(n, std::memory_order_relaxed);
  return n;
}

}  // namespace dfs
