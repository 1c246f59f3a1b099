// K5: non-causal flash attention over the retained heads only, on tcgen05 tensor cores.
//
// One CTA = 128 query rows of one head.  Per key/value block j of 128 tokens:
//   S_j = Q K_j^T      tcgen05.mma (M=128, N=128, K=DH) into TMEM (two S buffers)
//   P_j = exp2(S_j * scale - m)   softmax warps, one query row per thread, bf16 into smem
//   O  += P_j V_j      tcgen05.mma (M=128, N=DH, K=128) into a TMEM accumulator
// V arrives pre-transposed (V^T [heads*DH, n_kv], written by the QKV projection's
// epilogue) so both MMAs read K-major operands.  The running max is only moved when it
// grows by more than 2^8 (exact: the same stale max enters O and the row sum); O is then
// rescaled in TMEM before the next P V.  S_{j+1} is computed while the softmax of S_j
// runs.
//
//   warp 0      TMA: Q once, then K_j and V^T_j into a 2-stage ring
//   warp 1      MMA issuer (single thread) + TMEM owner
//   warps 2..5  softmax / rescale / output, thread = query row (TMEM lane)
#include "kernels.cuh"

namespace dfs {
namespace {

constexpr int kBM = 128;   // query rows per CTA
constexpr int kBN = 128;   // key / value rows per block
constexpr int kStages = 2;
constexpr int kThreads = 192;
constexpr float kRescaleThreshold = 8.f;  // log2 units

template <int DH>
struct AttnLayout {
  static constexpr int kQBytes = kBM * DH * 2;
  static constexpr int kKBytes = kBN * DH * 2;
  static constexpr int kVBytes = DH * kBN * 2;
  static constexpr int kPBytes = kBM * kBN * 2;
  static constexpr int kStageBytes = kKBytes + kVBytes;
  static constexpr int kSmem = kQBytes + kStages * kStageBytes + kPBytes + 1024 + 256;
  static constexpr uint32_t kTmemCols = 512;  // S0 [0,128), S1 [128,256), O [256, 256+DH)
};

template <int DH>
__global__ void __launch_bounds__(kThreads, 1) attn_fwd_tcgen05(const __grid_constant__ AttnArgs p) {
  using L = AttnLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;
  uint8_t* sKV = sQ + L::kQBytes;  // stage s: K at s*kStageBytes, V^T after it
  uint8_t* sP = sKV + kStages * L::kStageBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(sP + L::kPBytes);
  uint64_t* q_full = bars;
  uint64_t* kv_full = bars + 1;              // [kStages]
  uint64_t* kv_empty = kv_full + kStages;    // [kStages]
  uint64_t* s_full = kv_empty + kStages;     // [2]
  uint64_t* p_full = s_full + 2;
  uint64_t* o_done = p_full + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_done + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int q_tile = blockIdx.x;
  const int head = blockIdx.y;
  const int nkv = (p.n_kv + kBN - 1) / kBN;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    mbar_init(&s_full[0], 1);
    mbar_init(&s_full[1], 1);
    mbar_init(p_full, 128);
    mbar_init(o_done, 1);
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
  const uint32_t tmem_o = tmem + 256;
  bool failed = false;

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&p.tma_q);
      tma_prefetch_desc(&p.tma_k);
      tma_prefetch_desc(&p.tma_vt);
      const int qx = p.q_col0 + head * DH;
      const int kx = p.k_col0 + head * DH;
      mbar_arrive_expect_tx(q_full, L::kQBytes);
#pragma unroll
      for (int c = 0; c < DH / 64; ++c)
        tma_load_2d(sQ + c * (kBM * 128), &p.tma_q, q_full, qx + 64 * c, q_tile * kBM);
      for (int j = 0; j < nkv; ++j) {
        const int s = j % kStages;
        if (!mbar_wait(&kv_empty[s], ((j / kStages) & 1) ^ 1, p.err)) { failed = true; break; }
        mbar_arrive_expect_tx(&kv_full[s], L::kStageBytes);
        uint8_t* sK = sKV + s * L::kStageBytes;
        uint8_t* sV = sK + L::kKBytes;
#pragma unroll
        for (int c = 0; c < DH / 64; ++c)
          tma_load_2d(sK + c * (kBN * 128), &p.tma_k, &kv_full[s], kx + 64 * c, j * kBN);
#pragma unroll
        for (int c = 0; c < kBN / 64; ++c)
          tma_load_2d(sV + c * (DH * 128), &p.tma_vt, &kv_full[s], j * kBN + 64 * c, head * DH);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = idesc_bf16(kBM, kBN);
      constexpr uint32_t idesc_o = idesc_bf16(kBM, DH);
      const uint32_t q0 = smem_u32(sQ);
      const uint32_t p0 = smem_u32(sP);
      // S_j = Q K_j^T into S buffer (j & 1)
      auto issue_s = [&](int j) -> bool {
        const int s = j % kStages;
        if (!mbar_wait(&kv_full[s], (j / kStages) & 1, p.err)) return false;
        tc_fence_after();
        const uint32_t k0 = smem_u32(sKV + s * L::kStageBytes);
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
          const uint32_t off = (kk / 4) * (kBM * 128) + (kk % 4) * 32;
          const uint32_t offk = (kk / 4) * (kBN * 128) + (kk % 4) * 32;
          umma_bf16(tmem + (j & 1) * kBN, sw128_desc(q0 + off), sw128_desc(k0 + offk), idesc_s, kk != 0);
        }
        umma_commit(&s_full[j & 1]);
        return true;
      };
      if (!mbar_wait(q_full, 0, p.err)) failed = true;
      if (!failed) failed = !issue_s(0);
      if (!failed && nkv > 1) failed = !issue_s(1);
      for (int j = 0; j < nkv && !failed; ++j) {
        if (!mbar_wait(p_full, j & 1, p.err)) { failed = true; break; }
        tc_fence_after();
        const int s = j % kStages;
        const uint32_t v0 = smem_u32(sKV + s * L::kStageBytes + L::kKBytes);
#pragma unroll
        for (int kk = 0; kk < kBN / 16; ++kk) {
          const uint32_t offp = (kk / 4) * (kBM * 128) + (kk % 4) * 32;
          const uint32_t offv = (kk / 4) * (DH * 128) + (kk % 4) * 32;
          umma_bf16(tmem_o, sw128_desc(p0 + offp), sw128_desc(v0 + offv), idesc_o, (j | kk) != 0);
        }
        umma_commit(&kv_empty[s]);
        umma_commit(o_done);
        if (j + 2 < nkv) failed = !issue_s(j + 2);
      }
    }
  } else {
    const int sub = warp & 3;
    const int r = sub * 32 + lane;             // query row within the tile = TMEM lane
    const uint32_t lane_addr = static_cast<uint32_t>(sub * 32) << 16;
    const int q_row = q_tile * kBM + r;
    float m_run = -INFINITY;                   // running max of the scaled scores (log2 units)
    float l_run = 0.f;
    const float sl2 = p.scale_log2;
    for (int j = 0; j < nkv; ++j) {
      const bool ok = mbar_wait(&s_full[j & 1], (j >> 1) & 1, p.err);
      if (!__all_sync(0xffffffffu, ok)) { failed = true; break; }
      tc_fence_after();
      float s[kBN];
      tmem_ld128(tmem + lane_addr + (j & 1) * kBN, s);
      const int valid = p.n_kv - j * kBN;
      if (valid < kBN) {
#pragma unroll
        for (int i = 0; i < kBN; ++i)
          if (i >= valid) s[i] = -INFINITY;
      }
      // row max with independent partial maxima (short dependency chains)
      float pm[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) pm[i] = s[i];
#pragma unroll
      for (int i = 8; i < kBN; ++i) pm[i & 7] = fmaxf(pm[i & 7], s[i]);
      const float mx = fmaxf(fmaxf(fmaxf(pm[0], pm[1]), fmaxf(pm[2], pm[3])),
                             fmaxf(fmaxf(pm[4], pm[5]), fmaxf(pm[6], pm[7]))) * sl2;

      // PV_{j-1} must be complete before O is rescaled or P is overwritten.
      if (j > 0) {
        const bool ok2 = mbar_wait(o_done, (j - 1) & 1, p.err);
        if (!__all_sync(0xffffffffu, ok2)) { failed = true; break; }
        tc_fence_after();
      }
      const bool move = mx > m_run + kRescaleThreshold;
      if (j == 0) {
        m_run = mx;
      } else if (__any_sync(0xffffffffu, move)) {
        const float alpha = move ? fast_exp2(m_run - mx) : 1.f;
        if (move) m_run = mx;
        l_run *= alpha;
        // in halves of 64 columns; the scores are re-read from TMEM afterwards so that
        // they need not stay live in registers across the rescale
#pragma unroll
        for (int c = 0; c < DH / 64; ++c) {
          float o[64];
          tmem_ld64(tmem_o + lane_addr + 64 * c, o);
#pragma unroll
          for (int i = 0; i < 64; ++i) o[i] *= alpha;
          tmem_st64(tmem_o + lane_addr + 64 * c, o);
        }
        tmem_ld128(tmem + lane_addr + (j & 1) * kBN, s);
        if (valid < kBN) {
#pragma unroll
          for (int i = 0; i < kBN; ++i)
            if (i >= valid) s[i] = -INFINITY;
        }
      }
      // P = exp2(s * scale - m_run) -> bf16 in the 128-byte swizzled K-major layout of
      // the P V operand; the row sum uses 8 independent partial sums.
      const float neg_m = -m_run;
      float ps[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) ps[i] = 0.f;
#pragma unroll
      for (int c = 0; c < kBN / 8; ++c) {
        float e[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          e[i] = fast_exp2(fmaf(s[c * 8 + i], sl2, neg_m));
          ps[i] += e[i];
        }
        const int panel = c >> 3, chunk = c & 7;
        uint8_t* dst = sP + panel * (kBM * 128) + r * 128 + ((chunk ^ (r & 7)) << 4);
        *reinterpret_cast<uint4*>(dst) = pack_bf16x8(e);
      }
      l_run += ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      fence_proxy_async_smem();
      tc_fence_before();
      mbar_arrive(p_full);
    }
    if (!failed) {
      const bool ok = mbar_wait(o_done, (nkv - 1) & 1, p.err);
      if (!__all_sync(0xffffffffu, ok)) {
        failed = true;
      } else {
        tc_fence_after();
        const float inv = 1.f / l_run;
        float o[DH];
        if constexpr (DH == 128) tmem_ld128(tmem_o + lane_addr, o); else tmem_ld64(tmem_o + lane_addr, o);
        if (q_row < p.n_q) {
          bf16* dst = p.out + static_cast<long long>(q_row) * p.ldo + head * DH;
#pragma unroll
          for (int c = 0; c < DH / 8; ++c) {
            float f[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) f[i] = o[8 * c + i] * inv;
            *reinterpret_cast<uint4*>(dst + 8 * c) = pack_bf16x8(f);
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
  dim3 grid((a.n_q + kBM - 1) / kBM, a.n_heads);
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
