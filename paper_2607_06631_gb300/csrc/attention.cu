// K5: non-causal flash attention over the retained heads only, on tcgen05 tensor cores.
//
// One CTA = two 128-row query tiles (Q0, Q1) of one head, sharing every key / value
// tile.  Per key / value block j of 128 tokens and tile i:
//   S_i = Q_i K_j^T      tcgen05.mma (M=128, N=128, K=DH), fp32 into TMEM
//   P_i = exp2(S_i * scale - m_i)   softmax warpgroup i (thread = query row), bf16 written
//                        back into the first 64 columns of S_i's TMEM region
//   O_i += P_i V_j       tcgen05.mma with A read from TMEM (M=128, N=DH, K=128)
// The single MMA thread issues  S0_j, PV1_{j-1}, S1_j, PV0_j, S0_{j+1}, PV1_j, ...  so the
// softmax of one tile runs while the tensor core works on the other tile (a window of two
// 128x128x128 MMAs).  V arrives pre-transposed (V^T [heads*DH, n_kv], written by the QKV
// projection's epilogue) so every shared-memory operand is K-major.  The running max only
// moves when it grows by more than 2^8 (exact: the same stale max enters O and the row
// sum); O is then rescaled in TMEM.  K and V sit in separate two-deep rings.
//
//   warp 0      TMA: Q0, Q1 once; K_j and V^T_j into their rings
//   warp 1      MMA issuer (single thread) + TMEM owner (512 columns: S0, S1, O0, O1)
//   warps 2..5  softmax / rescale / output of tile 0
//   warps 6..9  softmax / rescale / output of tile 1
#include "kernels.cuh"

namespace dfs {
namespace {

constexpr int kBM = 128;   // query rows per tile (two tiles per CTA)
constexpr int kBN = 128;   // key / value rows per block
constexpr int kThreads = 320;
constexpr float kRescaleThreshold = 8.f;  // log2 units

template <int DH>
struct AttnLayout {
  static constexpr int kQBytes = kBM * DH * 2;   // one query tile
  static constexpr int kKBytes = kBN * DH * 2;   // one key tile
  static constexpr int kVBytes = DH * kBN * 2;   // one V^T tile
  static constexpr int kSmem = 2 * kQBytes + 2 * kKBytes + 2 * kVBytes + 1024 + 256;
  static constexpr uint32_t kTmemCols = 512;     // S0 [0,128) S1 [128,256) O0 [256,..) O1 [384,..)
};

template <int DH>
__global__ void __launch_bounds__(kThreads, 1) attn_fwd_tcgen05(const __grid_constant__ AttnArgs p) {
  using L = AttnLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                        // tile i at i * kQBytes
  uint8_t* sK = sQ + 2 * L::kQBytes;         // ring slot b at b * kKBytes
  uint8_t* sV = sK + 2 * L::kKBytes;         // ring slot b at b * kVBytes
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + 2 * L::kVBytes);
  uint64_t* q_full = bars;                   // 1
  uint64_t* k_full = bars + 1;               // [2]
  uint64_t* k_empty = k_full + 2;            // [2]
  uint64_t* v_full = k_empty + 2;            // [2]
  uint64_t* v_empty = v_full + 2;            // [2]
  uint64_t* s_full = v_empty + 2;            // [2] per tile: S_i of the current block ready
  uint64_t* p_full = s_full + 2;             // [2] per tile: P_i written (and O_i rescaled)
  uint64_t* o_done = p_full + 2;             // [2] per tile: last P_i V accumulated
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_done + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int head = blockIdx.y;
  const int q_base = blockIdx.x * (2 * kBM);
  const int nkv = (p.n_kv + kBN - 1) / kBN;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int b = 0; b < 2; ++b) {
      mbar_init(&k_full[b], 1);
      mbar_init(&k_empty[b], 1);
      mbar_init(&v_full[b], 1);
      mbar_init(&v_empty[b], 1);
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], 128);
      mbar_init(&o_done[b], 1);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, L::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool failed = false;

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&p.tma_q);
      tma_prefetch_desc(&p.tma_k);
      tma_prefetch_desc(&p.tma_vt);
      const int qx = p.q_col0 + head * DH;
      const int kx = p.k_col0 + head * DH;
      mbar_arrive_expect_tx(q_full, 2 * L::kQBytes);
#pragma unroll
      for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int c = 0; c < DH / 64; ++c)
          tma_load_2d(sQ + i * L::kQBytes + c * (kBM * 128), &p.tma_q, q_full, qx + 64 * c, q_base + i * kBM);
      // K runs one block ahead of V: K_j is needed by S0_j long before V_j by PV0_j
      for (int j = 0; j <= nkv && !failed; ++j) {
        if (j < nkv) {
          const int b = j & 1;
          if (!mbar_wait(&k_empty[b], ((j >> 1) & 1) ^ 1, p.err)) { failed = true; break; }
          mbar_arrive_expect_tx(&k_full[b], L::kKBytes);
#pragma unroll
          for (int c = 0; c < DH / 64; ++c)
            tma_load_2d(sK + b * L::kKBytes + c * (kBN * 128), &p.tma_k, &k_full[b], kx + 64 * c, j * kBN);
        }
        if (j >= 1) {
          const int jv = j - 1, b = jv & 1;
          if (!mbar_wait(&v_empty[b], ((jv >> 1) & 1) ^ 1, p.err)) { failed = true; break; }
          mbar_arrive_expect_tx(&v_full[b], L::kVBytes);
#pragma unroll
          for (int c = 0; c < kBN / 64; ++c)
            tma_load_2d(sV + b * L::kVBytes + c * (DH * 128), &p.tma_vt, &v_full[b], jv * kBN + 64 * c,
                        head * DH);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16(kBM, kBN);
      constexpr uint32_t idesc_o = idesc_bf16(kBM, DH);
      // Descriptors are built once: the issue loop only adds constant offsets (the start
      // address field holds address >> 4), which keeps this thread's issue rate at the
      // tensor pipe's rate.
      const uint64_t dq = sw128_desc(smem_u32(sQ));
      const uint64_t dk = sw128_desc(smem_u32(sK));
      const uint64_t dv = sw128_desc(smem_u32(sV));
      // S_i(j) = Q_i K_j^T into S_i's TMEM columns
      auto issue_s = [&](int i, int j) {
        const uint64_t a = dq + static_cast<uint64_t>(i * (L::kQBytes >> 4));
        const uint64_t b = dk + static_cast<uint64_t>((j & 1) * (L::kKBytes >> 4));
        const uint32_t d = tmem + i * kBN;
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          constexpr uint32_t panel = (kBM * 128) >> 4;
          const uint64_t off = (kk / 4) * panel + (kk % 4) * 2;
          umma_bf16(d, a + off, b + off, idesc_s, kk != 0);
        }
        umma_commit(&s_full[i]);
      };
      // O_i += P_i(j) V_j with P_i read from the first 64 columns of S_i
      auto issue_pv = [&](int i, int j) {
        const uint64_t b = dv + static_cast<uint64_t>((j & 1) * (L::kVBytes >> 4));
        const uint32_t d = tmem + 256 + i * 128, a = tmem + i * kBN;
        const uint32_t first = j != 0;
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          constexpr uint32_t panel = (DH * 128) >> 4;
          const uint64_t offv = (kk / 4) * panel + (kk % 4) * 2;
          umma_bf16_tmem_a(d, a + kk * 8, b + offv, idesc_o, kk == 0 ? first : 1u);
        }
      };
      do {
        if (!mbar_wait(q_full, 0, p.err)) { failed = true; break; }
        if (!mbar_wait(&k_full[0], 0, p.err)) { failed = true; break; }
        tc_fence_after();
        issue_s(0, 0);
        issue_s(1, 0);
        umma_commit(&k_empty[0]);
        for (int j = 0; j < nkv; ++j) {
          const int b = j & 1;
          const uint32_t ph = (j >> 1) & 1;
          // PV0_j
          if (!mbar_wait(&p_full[0], j & 1, p.err) || !mbar_wait(&v_full[b], ph, p.err)) { failed = true; break; }
          tc_fence_after();
          issue_pv(0, j);
          if (j + 1 == nkv) umma_commit(&o_done[0]);
          // S0_{j+1}
          if (j + 1 < nkv) {
            if (!mbar_wait(&k_full[(j + 1) & 1], ((j + 1) >> 1) & 1, p.err)) { failed = true; break; }
            tc_fence_after();
            issue_s(0, j + 1);
          }
          // PV1_j
          if (!mbar_wait(&p_full[1], j & 1, p.err)) { failed = true; break; }
          tc_fence_after();
          issue_pv(1, j);
          umma_commit(&v_empty[b]);
          if (j + 1 == nkv) umma_commit(&o_done[1]);
          // S1_{j+1}
          if (j + 1 < nkv) {
            issue_s(1, j + 1);
            umma_commit(&k_empty[(j + 1) & 1]);
          }
        }
      } while (false);
    }
  } else {
    const int tile = (warp - 2) >> 2;        // 0: warps 2..5, 1: warps 6..9
    const int sub = warp & 3;                // TMEM lane quarter this warp may access
    const int r = sub * 32 + lane;           // query row within the tile = TMEM lane
    const uint32_t lane_addr = static_cast<uint32_t>(sub * 32) << 16;
    const uint32_t tS = tmem + tile * kBN + lane_addr;
    const uint32_t tO = tmem + 256 + tile * 128 + lane_addr;
    const int q_row = q_base + tile * kBM + r;
    const float sl2 = p.scale_log2;
    float m_run = -INFINITY;                 // running max of the scaled scores (log2 units)
    float l_run = 0.f;
    for (int j = 0; j < nkv; ++j) {
      const bool ok = mbar_wait(&s_full[tile], j & 1, p.err);
      if (!__all_sync(0xffffffffu, ok)) { failed = true; break; }
      tc_fence_after();
      float s[kBN];
      tmem_ld128(tS, s);
      const int valid = p.n_kv - j * kBN;
      if (valid < kBN) {
#pragma unroll
        for (int i = 0; i < kBN; ++i)
          if (i >= valid) s[i] = -INFINITY;
      }
      // row max: 8 independent chains of three-input maxima
      float pm[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) pm[i] = s[i];
#pragma unroll
      for (int i = 8; i < kBN; i += 16)
#pragma unroll
        for (int k = 0; k < 8; ++k) pm[k] = fmax3(pm[k], s[i + k], s[i + 8 + k]);
      const float mx = fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7])) * sl2;
      const bool move = mx > m_run + kRescaleThreshold;
      if (j == 0) {
        m_run = mx;
      } else if (__any_sync(0xffffffffu, move)) {
        // S_i(j) completing implies P_i(j-1) V_{j-1} completed: O_i is stable here
        const float alpha = move ? fast_exp2(m_run - mx) : 1.f;
        if (move) m_run = mx;
        l_run *= alpha;
#pragma unroll
        for (int c = 0; c < DH / 32; ++c) {
          float o[32];
          tmem_ld32(tO + 32 * c, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(tO + 32 * c, o);
        }
      }
      // P = exp2(s * scale - m_run) as bf16 pairs into the first 64 columns of S_i;
      // scale-and-shift and the row-sum partials run as packed pairs
      const float neg_m = -m_run;
      float ps[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ps[i] = 0.f;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        uint32_t pk[32];
#pragma unroll
        for (int c = 0; c < 32; ++c) {
          float x0, x1;
          ffma2(x0, x1, s[64 * h + 2 * c], s[64 * h + 2 * c + 1], sl2, sl2, neg_m, neg_m);
          const float e0 = fast_exp2(x0);
          const float e1 = fast_exp2(x1);
          fadd2(ps[2 * (c & 3)], ps[2 * (c & 3) + 1], e0, e1);
          pk[c] = pack_bf16x2(e0, e1);
        }
        tmem_st32u(tS + 32 * h, pk);
      }
      l_run += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      tc_fence_before();
      mbar_arrive(&p_full[tile]);
    }
    if (!failed) {
      const bool ok = mbar_wait(&o_done[tile], 0, p.err);
      if (!__all_sync(0xffffffffu, ok)) {
        failed = true;
      } else {
        tc_fence_after();
        const float inv = 1.f / l_run;
        bf16* dst = p.out + static_cast<long long>(q_row) * p.ldo + head * DH;
#pragma unroll
        for (int c = 0; c < DH / 32; ++c) {
          float o[32];
          tmem_ld32(tO + 32 * c, o);
          if (q_row < p.n_q) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              float f[8];
#pragma unroll
              for (int i = 0; i < 8; ++i) f[i] = o[8 * q + i] * inv;
              *reinterpret_cast<uint4*>(dst + 32 * c + 8 * q) = pack_bf16x8(f);
            }
          }
        }
      }
    }
  }

  if (failed) drain_after_error();
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, L::kTmemCols);
  }
}

}  // namespace

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_tcgen05<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       AttnLayout<64>::kSmem);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_fwd_tcgen05<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              AttnLayout<128>::kSmem);
}

cudaError_t launch_attention(const AttnArgs& a, int head_dim, cudaStream_t s) {
  if (a.n_q <= 0 || a.n_kv <= 0 || a.n_heads <= 0) return cudaSuccess;
  dim3 grid((a.n_q + 2 * kBM - 1) / (2 * kBM), a.n_heads);
  if (head_dim == 128) {
    attn_fwd_tcgen05<128><<<grid, kThreads, AttnLayout<128>::kSmem, s>>>(a);
  } else if (head_dim == 64) {
    attn_fwd_tcgen05<64><<<grid, kThreads, AttnLayout<64>::kSmem, s>>>(a);
  } else {
    return cudaErrorInvalidValue;
  }
  return cudaGetLastError();
}

}  // namespace dfs
