// K5: non-causal flash attention over the retained heads only, on tcgen05 tensor cores,
// with CTA pairs (a cluster of 2 CTAs on two SMs) issuing 2-SM MMAs.
//
// A CTA pair covers 512 query rows of one head: CTA r (r = 0, 1 in the pair) owns rows
// [512 c + 256 r, +256) as two 128-row tiles.  Tile i of both CTAs forms one M = 256 MMA:
//   S_i = Q_i K_j^T      tcgen05.mma.cta_group::2 (M=256, N=128, K=DH) -> each CTA's TMEM
//   P_i = exp2(S_i * scale - m_i)   softmax warpgroup i of each CTA (thread = query row),
//                        bf16 written back into the first 64 columns of S_i's TMEM region
//   O_i += P_i V_j       tcgen05.mma.cta_group::2 with A read from both CTAs' TMEM
// For each 2-SM MMA each CTA holds only half of the B operand: keys [64 r, 64 r + 64) of K_j
// and V^T rows [DH/2 r, DH/2 r + DH/2), so every SM reads half as many operand bytes from
// shared memory and loads half of each K/V tile from L2.  The even CTA's single MMA thread
// issues  S0_j, PV1_{j-1}, S1_j, PV0_j, S0_{j+1}, PV1_j, ...  so either tile's softmax overlaps
// two MMAs of the other tile; its commits are multicast to both CTAs' barriers.  Both CTAs'
// TMA loads complete on the even CTA's barriers.  V arrives pre-transposed (V^T written by
// the QKV projection's epilogue) so every shared-memory operand is K-major.
//
// The softmax has no row-max pass after the first key block.  P of block j is taken with
// the running offset m (the first block's exact row max, or a later one), which is exact for
// any m because the numerator O and the row sum l share it; m only has to keep P finite and
// representable.  A row whose block sum stays within kSumLimit has every P of the block
// within it; otherwise (or for a non-finite sum) the warp redoes the block with the exact
// maximum and rescales O (in TMEM) and l.  So the exponentials start as soon as S is in
// registers, and a tile's softmax is one pass: TMEM load, exponentials and packing, P store.
//
//   warp 0      TMA: own Q0, Q1 once; own halves of K_j and V^T_j into three-deep rings
//   warp 1      TMEM allocation (collective over the pair); in the even CTA also the MMA thread
//   warps 2..3  idle (they complete warpgroup 0, whose registers go to the softmax warpgroups)
//   warps 4..7  softmax / rescale / output of tile 0
//   warps 8..11 softmax / rescale / output of tile 1
// The warpgroups split the register file unevenly (setmaxnreg): 88 registers per thread in
// warpgroup 0, 208 in the softmax warpgroups, which then hold a row's 128 scores and its
// packed P without spilling to local memory.
#include "kernels.cuh"

namespace dfs {
namespace {

constexpr int kBM = 128;   // query rows per tile (two tiles per CTA, four per pair)
constexpr int kBN = 128;   // key / value rows per block
constexpr int kStages = 3; // K and V ring depth
constexpr int kThreads = 384;
// Register split between the warpgroups (setmaxnreg): the launch gives every thread
// kRegsLaunch registers (384 threads x 168 = 64512 of the SM's 65536; ptxas reports 168 for
// this kernel); the TMA / MMA warpgroup gives part of its share to the two softmax
// warpgroups.  The shares add up to the launch's total, 128 x 88 + 256 x 208 = 384 x 168,
// and per SM sub-partition (one warp of each warpgroup) 88 + 208 + 208 = 504 registers x 32
// lanes <= its 16384.  A larger softmax share would make the increase wait forever.
constexpr int kRegsLaunch = 168, kRegsControl = 88, kRegsSoftmax = 208;
static_assert(128 * kRegsControl + 256 * kRegsSoftmax <= kThreads * kRegsLaunch, "register split exceeds the launch");
static_assert(kThreads * kRegsLaunch <= 65536, "launch registers exceed the SM");
static_assert((kRegsControl + 2 * kRegsSoftmax) * 32 <= 16384, "register split exceeds a sub-partition");
// Largest accepted row sum of one key block's P (every P of such a row is at most this):
// far from fp32 / bf16 overflow, so O and l accumulate safely with a stale offset.
constexpr float kSumLimit = 65536.f;

// Store of 32 consecutive 32-bit TMEM columns without the wait (tcgen05.wait::st follows later).
__device__ __forceinline__ void tmem_st32u_async(uint32_t taddr, const uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};\n"
      ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31])
      : "memory");
}

__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

template <int DH>
struct AttnLayout {
  static constexpr int kQBytes = kBM * DH * 2;          // one query tile
  static constexpr int kKBytes = (kBN / 2) * DH * 2;    // this CTA's half of a key tile
  static constexpr int kVBytes = (DH / 2) * kBN * 2;    // this CTA's half of a V^T tile
  static constexpr int kKPanel = (kBN / 2) * 128;       // bytes per 64-wide K panel
  static constexpr int kVPanel = (DH / 2) * 128;        // bytes per 64-wide V^T panel
  static constexpr int kSmemUsed = 2 * kQBytes + kStages * (kKBytes + kVBytes) + 1024 + 256;
  // at least 120 KB so that a second CTA can never share the SM: two pairs interleaved over
  // the same two SMs could otherwise each hold one SM's TMEM while waiting for the other's
  static constexpr int kSmem = kSmemUsed < 120 * 1024 ? 120 * 1024 : kSmemUsed;
  static constexpr uint32_t kTmemCols = 512;            // S0 [0,128) S1 [128,256) O0 [256,..) O1 [384,..)
};

template <int DH>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    attn_fwd_tcgen05(const __grid_constant__ AttnArgs p) {
  using L = AttnLayout<DH>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sQ = smem;                        // tile i at i * kQBytes
  uint8_t* sK = sQ + 2 * L::kQBytes;         // ring slot s at s * kKBytes
  uint8_t* sV = sK + kStages * L::kKBytes;   // ring slot s at s * kVBytes
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + kStages * L::kVBytes);
  uint64_t* q_full = bars;                   // 1   (even CTA's copy counts both CTAs' bytes)
  uint64_t* k_full = bars + 1;               // [kStages]
  uint64_t* k_empty = k_full + kStages;      // [kStages]
  uint64_t* v_full = k_empty + kStages;      // [kStages]
  uint64_t* v_empty = v_full + kStages;      // [kStages]
  uint64_t* s_full = v_empty + kStages;      // [2] per tile: S_i of the current block ready
  uint64_t* p_full = s_full + 2;             // [2] per tile: P_i written by all 8 warps of the pair
  uint64_t* o_done = p_full + 2;             // [2] per tile: last P_i V accumulated
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(o_done + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int head = blockIdx.y;
  const int q_base = (blockIdx.x >> 1) * (4 * kBM) + static_cast<int>(rank) * (2 * kBM);
  const int nkv = (p.n_kv + kBN - 1) / kBN;

  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], 8);
      mbar_init(&o_done[b], 1);
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(L::kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers are initialised before any cross-CTA traffic
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  bool failed = false;

  if (warp < 4) {
    // warpgroup 0 (TMA, MMA, two idle warps) hands registers to the softmax warpgroups
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsControl));
    if (warp == 0) {
      if (lane == 0) {
        tma_prefetch_desc(&p.tma_q);
        tma_prefetch_desc(&p.tma_k);
        tma_prefetch_desc(&p.tma_vt);
        const int qx = p.q_col0 + head * DH;
        const int kx = p.k_col0 + head * DH;
        const uint32_t lq = map_to_rank(q_full, 0);
        if (rank == 0) mbar_arrive_expect_tx(q_full, 2 * 2 * L::kQBytes);
#pragma unroll
        for (int i = 0; i < 2; ++i)
#pragma unroll
          for (int c = 0; c < DH / 64; ++c)
            tma_load_2d_pair(sQ + i * L::kQBytes + c * (kBM * 128), &p.tma_q, lq, qx + 64 * c, q_base + i * kBM);
        // K runs one block ahead of V: K_j is needed by S0_j long before V_j by PV0_j
        for (int j = 0; j <= nkv && !failed; ++j) {
          if (j < nkv) {
            const int s = j % kStages;
            if (!mbar_wait_cluster(&k_empty[s], ((j / kStages) & 1) ^ 1, p.err)) { failed = true; break; }
            if (rank == 0) mbar_arrive_expect_tx(&k_full[s], 2 * L::kKBytes);
            const uint32_t lk = map_to_rank(&k_full[s], 0);
#pragma unroll
            for (int c = 0; c < DH / 64; ++c)
              tma_load_2d_pair(sK + s * L::kKBytes + c * L::kKPanel, &p.tma_k, lk, kx + 64 * c,
                               j * kBN + static_cast<int>(rank) * (kBN / 2));
          }
          if (j >= 1) {
            const int jv = j - 1, s = jv % kStages;
            if (!mbar_wait_cluster(&v_empty[s], ((jv / kStages) & 1) ^ 1, p.err)) { failed = true; break; }
            if (rank == 0) mbar_arrive_expect_tx(&v_full[s], 2 * L::kVBytes);
            const uint32_t lv = map_to_rank(&v_full[s], 0);
#pragma unroll
            for (int c = 0; c < kBN / 64; ++c)
              tma_load_2d_pair(sV + s * L::kVBytes + c * L::kVPanel, &p.tma_vt, lv, jv * kBN + 64 * c,
                               head * DH + static_cast<int>(rank) * (DH / 2));
          }
        }
      }
    } else if (warp == 1) {
      if (lane == 0 && rank == 0) {
        constexpr uint32_t idesc_s = idesc_bf16(2 * kBM, kBN);
        constexpr uint32_t idesc_o = idesc_bf16(2 * kBM, DH);
        // Descriptors are built once: the issue loop only adds constant offsets (the start
        // address field holds address >> 4), which keeps this thread's issue rate at the
        // tensor pipe's rate.
        const uint64_t dq = sw128_desc(smem_u32(sQ));
        const uint64_t dk = sw128_desc(smem_u32(sK));
        const uint64_t dv = sw128_desc(smem_u32(sV));
        // S_i(j) = Q_i K_j^T into S_i's TMEM columns of both CTAs
        auto issue_s = [&](int i, int j) {
          const uint64_t a = dq + static_cast<uint64_t>(i * (L::kQBytes >> 4));
          const uint64_t b = dk + static_cast<uint64_t>((j % kStages) * (L::kKBytes >> 4));
          const uint32_t d = tmem + i * kBN;
#pragma unroll
          for (int kk = 0; kk < DH / 16; ++kk) {
            constexpr uint32_t qpanel = (kBM * 128) >> 4, kpanel = L::kKPanel >> 4;
            mma_pair_ss(d, a + (kk / 4) * qpanel + (kk % 4) * 2, b + (kk / 4) * kpanel + (kk % 4) * 2, idesc_s,
                        kk != 0);
          }
          commit_pair(&s_full[i]);
        };
        // O_i += P_i(j) V_j with P_i read from the first 64 columns of S_i in both CTAs
        auto issue_pv = [&](int i, int j) {
          const uint64_t b = dv + static_cast<uint64_t>((j % kStages) * (L::kVBytes >> 4));
          const uint32_t d = tmem + 256 + i * 128, a = tmem + i * kBN;
          const uint32_t first = j != 0;
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk) {
            constexpr uint32_t vpanel = L::kVPanel >> 4;
            mma_pair_ts(d, a + kk * 8, b + (kk / 4) * vpanel + (kk % 4) * 2, idesc_o, kk == 0 ? first : 1u);
          }
        };
        do {
          if (!mbar_wait_cluster(q_full, 0, p.err)) { failed = true; break; }
          if (!mbar_wait_cluster(&k_full[0], 0, p.err)) { failed = true; break; }
          tc_fence_after();
          issue_s(0, 0);
          issue_s(1, 0);
          commit_pair(&k_empty[0]);
          for (int j = 0; j < nkv; ++j) {
            const int s = j % kStages;
            const uint32_t ph = (j / kStages) & 1;
            // PV0_j
            if (!mbar_wait_cluster(&p_full[0], j & 1, p.err) || !mbar_wait_cluster(&v_full[s], ph, p.err)) {
              failed = true;
              break;
            }
            tc_fence_after();
            issue_pv(0, j);
            if (j + 1 == nkv) commit_pair(&o_done[0]);
            // S0_{j+1}
            if (j + 1 < nkv) {
              const int s1 = (j + 1) % kStages;
              if (!mbar_wait_cluster(&k_full[s1], ((j + 1) / kStages) & 1, p.err)) { failed = true; break; }
              tc_fence_after();
              issue_s(0, j + 1);
            }
            // PV1_j
            if (!mbar_wait_cluster(&p_full[1], j & 1, p.err)) { failed = true; break; }
            tc_fence_after();
            issue_pv(1, j);
            commit_pair(&v_empty[s]);
            if (j + 1 == nkv) commit_pair(&o_done[1]);
            // S1_{j+1}
            if (j + 1 < nkv) {
              issue_s(1, j + 1);
              commit_pair(&k_empty[(j + 1) % kStages]);
            }
          }
        } while (false);
      }
    }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsSoftmax));
    const int tile = (warp - 4) >> 2;        // 0: warps 4..7, 1: warps 8..11
    const int sub = warp & 3;                // TMEM lane quarter this warp may access
    const int r = sub * 32 + lane;           // query row within the tile = TMEM lane
    const uint32_t lane_addr = static_cast<uint32_t>(sub * 32) << 16;
    const uint32_t tS = tmem + tile * kBN + lane_addr;
    const uint32_t tO = tmem + 256 + tile * 128 + lane_addr;
    const int q_row = q_base + tile * kBM + r;
    const uint32_t p_full_leader = map_to_rank(&p_full[tile], 0);
    const float sl2 = p.scale_log2;
    float m_run = -INFINITY;                 // offset of P (log2 units): block 0's row max, raised by redone blocks
    float l_run = 0.f;
    for (int j = 0; j < nkv; ++j) {
      const bool ok = mbar_wait_cluster(&s_full[tile], j & 1, p.err);
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
      // row max of the scaled scores: 8 independent chains of three-input maxima
      auto row_max = [&]() {
        float pm[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) pm[i] = s[i];
#pragma unroll
        for (int i = 8; i < kBN; i += 16)
#pragma unroll
          for (int k = 0; k < 8; ++k) pm[k] = fmax3(pm[k], s[i + k], s[i + 8 + k]);
        return fmax3(fmax3(pm[0], pm[1], pm[2]), fmax3(pm[3], pm[4], pm[5]), fmaxf(pm[6], pm[7])) * sl2;
      };
      // P = exp2(s * scale - m_run) as bf16 pairs into the first 64 columns of S_i (the first
      // half's store overlaps the second half's arithmetic); returns the block's row sum.
      // Scale-and-shift and the row-sum partials run as packed pairs.
      auto write_p = [&]() {
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
          tmem_st32u_async(tS + 32 * h, pk);
        }
        tmem_wait_st();
        return ((ps[0] + ps[1]) + (ps[2] + ps[3])) + ((ps[4] + ps[5]) + (ps[6] + ps[7]));
      };
      // The first block sets the running max exactly.  Later blocks reuse it without a max
      // pass: their P are exact for any offset (numerator and row sum share it), and only
      // their size matters.  A block row sum within kSumLimit bounds every P of that row by
      // it; a larger (or non-finite) sum in any row of the warp makes the warp redo the block
      // with the exact maximum, rescaling O and the row sum.
      if (j == 0) m_run = row_max();
      float l_blk, alpha = 1.f;
      for (int pass = 0;; ++pass) {
        l_blk = write_p();
        if (pass == 1 || !__any_sync(0xffffffffu, !(l_blk <= kSumLimit))) break;
        const float m_new = fmaxf(m_run, row_max());
        alpha = fast_exp2(m_run - m_new);
        m_run = m_new;
      }
      if (__any_sync(0xffffffffu, alpha != 1.f)) {
        // S_i(j) completing implies P_i(j-1) V_{j-1} completed: O_i is stable here, and
        // P_i(j) V_j is issued only after this warp's arrival below
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
      l_run += l_blk;
      // The TMEM stores of P are complete (tcgen05.wait::st) and ordered before this
      // thread-sync point by the tcgen05 fence; the MMA thread orders its MMAs after its
      // wait with tcgen05.fence::after_thread_sync.  One arrival per warp: local in the
      // even CTA, remote (relaxed, cluster scope) from the odd one.
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank == 0) mbar_arrive(&p_full[tile]);
        else asm volatile("mbarrier.arrive.relaxed.cluster.shared::cluster.b64 _, [%0];" ::"r"(p_full_leader) : "memory");
      }
    }
    if (!failed) {
      const bool ok = mbar_wait_cluster(&o_done[tile], 0, p.err);
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
  cluster_sync();  // the even CTA's MMAs read this CTA's shared memory and TMEM until here
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(L::kTmemCols) : "memory");
}

}  // namespace

cudaError_t attention_prepare() {
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_tcgen05<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       AttnLayout<64>::kSmem);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(attn_fwd_tcgen05<128>, cudaFuncAttributeMaxDynamicSharedMemorySize, AttnLayout<128>::kSmem);
  if (e != cudaSuccess) return e;
  // The softmax warpgroups' setmaxnreg.inc is satisfied only by the registers warpgroup 0
  // releases, which assumes kRegsLaunch registers per thread at launch: a build that
  // allocated fewer would make the increase wait forever, so it is refused here.
  cudaFuncAttributes at64, at128;
  if ((e = cudaFuncGetAttributes(&at64, attn_fwd_tcgen05<64>)) != cudaSuccess) return e;
  if ((e = cudaFuncGetAttributes(&at128, attn_fwd_tcgen05<128>)) != cudaSuccess) return e;
  return at64.numRegs == kRegsLaunch && at128.numRegs == kRegsLaunch ? cudaSuccess : cudaErrorNotSupported;
}

cudaError_t launch_attention(const AttnArgs& a, int head_dim, cudaStream_t s) {
  if (a.n_q <= 0 || a.n_kv <= 0 || a.n_heads <= 0) return cudaSuccess;
  dim3 grid(2 * ((a.n_q + 4 * kBM - 1) / (4 * kBM)), a.n_heads);
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
