// K4: persistent, warp-specialised tcgen05 GEMM for the block's projections
// (QKV, attention output, FFN up / down), D = A * B^T with both operands K-major bf16.
//
// CTA pairs (clusters of 2 CTAs on two SMs) compute 256 x 256 output tiles with 2-SM MMAs
// (tcgen05.mma.cta_group::2, M=256, N=256, K=16): CTA r holds the A rows [128 r, 128 r + 128)
// of the tile and the B rows [128 r, 128 r + 128) (half of N), so each SM stages and reads
// half of the B operand of a 256 x 256 tile from shared memory, and the pair reads each A and
// B element from L2 once per tile.  Both CTAs' TMA loads complete on the even CTA's
// barriers; its single MMA thread's commits are multicast to both CTAs.
//
//   warp 0      TMA producer: own A rows 128x64 and own B rows 128x64 per stage, 6-stage ring;
//               B either as stored or gathered head by head from a union weight matrix.
//   warp 1      TMEM allocation (collective over the pair); in the even CTA the MMA thread,
//               issuing into one of two accumulators (2 x 256 fp32 columns per CTA), so the
//               epilogue of tile i overlaps the main loop of tile i+1.
//   warps 2..3  idle (they complete warpgroup 0, whose registers go to the epilogue warpgroups)
//   warps 4..11 epilogue of this CTA's 128 rows: tcgen05.ld 32 columns at a time, fused bias /
//               GELU / gated residual, predicated stores for the ragged M and N edges.  A
//               thread owns one output row, so every global access of a warp touches 32 rows;
//               where bases and row pitches allow, the accesses are 256-bit (one full 32-byte
//               sector per row per instruction) to halve the number of L1 / L2 transactions.
//               Short reductions use all 8 warps (two per TMEM lane quarter, 128 columns each),
//               long ones warps 4..7 only (GemmArgs::epi_warps).  The fp32 gated-residual output
//               (x1) of full tiles goes out by TMA: each warp stages its 32 x 32 chunk in shared
//               memory (128-byte swizzle) and one lane issues the tensor store, so the global
//               writes leave as whole lines instead of 32 row pieces per instruction.
// setmaxnreg splits the registers: 72 per thread in warpgroup 0, 216 in the epilogue
// warpgroups (launch 384 x 168 = 128 x 72 + 256 x 216).
// Ragged K (f_s is a multiple of 8, not of 64) is covered by TMA zero fill.
#include "kernels.cuh"

namespace dfs {
namespace {

__device__ __forceinline__ float gelu_tanh(float x) {
  // GELU, tanh form: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))
  const float u = 0.7978845608028654f * fmaf(0.044715f * x, x * x, x);
  float t;
  asm("tanh.approx.f32 %0, %1;" : "=f"(t) : "f"(u));
  return 0.5f * x * (1.f + t);
}

// Grouped raster: G M-tiles share each sweep over N so that concurrent CTA pairs reuse both
// operands from L2; the sweep direction alternates between groups (serpentine), so each group
// starts on the B bands its predecessor finished with.
__device__ __forceinline__ void tile_coords(int tile, int m_tiles, int n_tiles, int G, int& mt, int& nt) {
  const int group = tile / (G * n_tiles);
  const int first_m = group * G;
  const int gsz = min(m_tiles - first_m, G);
  const int local = tile - group * G * n_tiles;
  mt = first_m + local % gsz;
  nt = local / gsz;
  if (group & 1) nt = n_tiles - 1 - nt;
}

__device__ __forceinline__ void st_global_32B(void* dst, const uint4& a, const uint4& b);

// `wide`: dst is 32-byte aligned (one 256-bit store per 16 values instead of two 128-bit ones)
__device__ __forceinline__ void store_bf16_row(bf16* dst, const float (&v)[32], int valid, bool wide = false) {
  if (valid >= 32 && wide) {
#pragma unroll
    for (int q = 0; q < 2; ++q) {
      const uint4 a = make_uint4(pack_bf16x2(v[16 * q], v[16 * q + 1]), pack_bf16x2(v[16 * q + 2], v[16 * q + 3]),
                                 pack_bf16x2(v[16 * q + 4], v[16 * q + 5]), pack_bf16x2(v[16 * q + 6], v[16 * q + 7]));
      const uint4 b = make_uint4(pack_bf16x2(v[16 * q + 8], v[16 * q + 9]), pack_bf16x2(v[16 * q + 10], v[16 * q + 11]),
                                 pack_bf16x2(v[16 * q + 12], v[16 * q + 13]), pack_bf16x2(v[16 * q + 14], v[16 * q + 15]));
      st_global_32B(dst + 16 * q, a, b);
    }
  } else if (valid >= 32) {
    uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint4 u;
      u.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
      u.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
      u.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
      u.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
      d4[q] = u;
    }
  } else {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j < valid) dst[j] = __float2bfloat16_rn(v[j]);
  }
}

__device__ __forceinline__ void epilogue_chunk(const GemmArgs& p, int row, int col0, float (&v)[32], bool wide) {
  const int valid = min(32, p.N - col0);
  if (p.bias != nullptr) {
    if (valid >= 32) {
      const uint4* b4 = reinterpret_cast<const uint4*>(p.bias + col0);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float f[8];
        unpack_bf16x8(__ldg(b4 + q), f);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[8 * q + i] += f[i];
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j < valid) v[j] += bf16_to_f32(p.bias[col0 + j]);
    }
  }
  if (row >= p.M) return;

  if (p.mode == kEpiBias) {
    if (col0 < p.split) {
      store_bf16_row(static_cast<bf16*>(p.out) + static_cast<long long>(row) * p.ldo + col0, v, valid, wide);
    } else {
      bf16* t = p.out_t + static_cast<long long>(col0 - p.split) * p.ldt + row;
#pragma unroll
      for (int j = 0; j < 32; ++j)
        if (j < valid) t[static_cast<long long>(j) * p.ldt] = __float2bfloat16_rn(v[j]);
    }
  } else if (p.mode == kEpiBiasGelu) {
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = gelu_tanh(v[j]);
    store_bf16_row(static_cast<bf16*>(p.out) + static_cast<long long>(row) * p.ldo + col0, v, valid, wide);
  } else {  // kEpiGatedRes
    float g[32], r[32];
    if (p.gate != nullptr) {
      if (valid >= 32) {
        const float4* g4 = reinterpret_cast<const float4*>(p.gate + col0);
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 t = __ldg(g4 + q);
          g[4 * q] = t.x; g[4 * q + 1] = t.y; g[4 * q + 2] = t.z; g[4 * q + 3] = t.w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) g[j] = (j < valid) ? p.gate[col0 + j] : 0.f;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) g[j] = 1.f;
    }
    if (p.res_f32) {
      const float* rp = static_cast<const float*>(p.res) + static_cast<long long>(row) * p.ldr + col0;
      if (valid >= 32) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
          const float4 t = *reinterpret_cast<const float4*>(rp + 4 * q);
          r[4 * q] = t.x; r[4 * q + 1] = t.y; r[4 * q + 2] = t.z; r[4 * q + 3] = t.w;
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) r[j] = (j < valid) ? rp[j] : 0.f;
      }
    } else {
      const bf16* rp = static_cast<const bf16*>(p.res) + static_cast<long long>(row) * p.ldr + col0;
      if (valid >= 32) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          float f[8];
          unpack_bf16x8(*reinterpret_cast<const uint4*>(rp + 8 * q), f);
#pragma unroll
          for (int i = 0; i < 8; ++i) r[8 * q + i] = f[i];
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) r[j] = (j < valid) ? bf16_to_f32(rp[j]) : 0.f;
      }
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = fmaf(g[j], v[j], r[j]);
    if (p.out_f32) {
      float* op = static_cast<float*>(p.out) + static_cast<long long>(row) * p.ldo + col0;
      if (valid >= 32) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          *reinterpret_cast<float4*>(op + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
          if (j < valid) op[j] = v[j];
      }
    } else {
      store_bf16_row(static_cast<bf16*>(p.out) + static_cast<long long>(row) * p.ldo + col0, v, valid);
    }
  }
}

// 32 bytes at a 32-byte aligned global address as two 16-byte words (one 256-bit access).
__device__ __forceinline__ void ld_global_32B(const void* src, uint4& a, uint4& b) {
  asm volatile("ld.global.v8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
               : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
               : "l"(src));
}

__device__ __forceinline__ void st_global_32B(void* dst, const uint4& a, const uint4& b) {
  asm volatile("st.global.v8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"l"(dst), "r"(a.x), "r"(a.y), "r"(a.z),
               "r"(a.w), "r"(b.x), "r"(b.y), "r"(b.z), "r"(b.w)
               : "memory");
}

// Raw 16-byte words of one 32-column chunk of this thread's residual row (fp32: 8 words,
// bf16: the first 4), read with 256-bit accesses.
__device__ __forceinline__ void load_res_chunk(int res_f32, const char* rrow, int c, uint4 (&w)[8]) {
  if (res_f32) {
#pragma unroll
    for (int q = 0; q < 4; ++q) ld_global_32B(rrow + c * 128 + 32 * q, w[2 * q], w[2 * q + 1]);
  } else {
#pragma unroll
    for (int q = 0; q < 2; ++q) ld_global_32B(rrow + c * 64 + 32 * q, w[2 * q], w[2 * q + 1]);
  }
}

// kEpiGatedRes over one full row of a 256-column tile (row < M, all columns < N; output and
// residual 32-byte aligned with 32-byte multiple pitches): the same arithmetic as
// epilogue_chunk, with 256-bit loads and stores and the residual loads of chunk c + 2
// issued before chunk c is processed, so that each warp keeps three chunks of loads in
// flight instead of waiting out one memory latency per 32 columns.  The residual may be the
// output itself (in-place update): every element is still read by its own thread before
// that thread writes it.
template <int NCH>
__device__ __forceinline__ void epilogue_gated_row(const GemmArgs& p, int row, int colb, uint32_t taddr,
                                                   uint8_t* stage) {
  const int lane = threadIdx.x & 31;
  const bool tma_out = p.out_tma && p.out_f32;
  const char* rrow = static_cast<const char*>(p.res) +
                     (static_cast<long long>(row) * p.ldr + colb) * (p.res_f32 ? 4 : 2);
  uint4 w[3][8];
  load_res_chunk(p.res_f32, rrow, 0, w[0]);
  load_res_chunk(p.res_f32, rrow, 1, w[1]);
#pragma unroll
  for (int c = 0; c < NCH; ++c) {
    if (c + 2 < NCH) load_res_chunk(p.res_f32, rrow, c + 2, w[(c + 2) % 3]);
    const int col0 = colb + 32 * c;
    float v[32];
    tmem_ld32(taddr + 32 * c, v);
    if (p.bias != nullptr) {
      const uint4* b4 = reinterpret_cast<const uint4*>(p.bias + col0);
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float f[8];
        unpack_bf16x8(__ldg(b4 + q), f);
#pragma unroll
        for (int i = 0; i < 8; ++i) v[8 * q + i] += f[i];
      }
    }
    float g[32];
    if (p.gate != nullptr) {
      const float4* g4 = reinterpret_cast<const float4*>(p.gate + col0);
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const float4 t = __ldg(g4 + q);
        g[4 * q] = t.x; g[4 * q + 1] = t.y; g[4 * q + 2] = t.z; g[4 * q + 3] = t.w;
      }
    } else {
#pragma unroll
      for (int j = 0; j < 32; ++j) g[j] = 1.f;
    }
    float r[32];
    const uint4(&wc)[8] = w[c % 3];
    if (p.res_f32) {
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        r[4 * q] = __uint_as_float(wc[q].x); r[4 * q + 1] = __uint_as_float(wc[q].y);
        r[4 * q + 2] = __uint_as_float(wc[q].z); r[4 * q + 3] = __uint_as_float(wc[q].w);
      }
    } else {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        float f[8];
        unpack_bf16x8(wc[q], f);
#pragma unroll
        for (int i = 0; i < 8; ++i) r[8 * q + i] = f[i];
      }
    }
#pragma unroll
    for (int j = 0; j < 32; ++j) v[j] = fmaf(g[j], v[j], r[j]);
    if (tma_out) {
      // this warp's 32 rows x 32 columns through its staging buffer (128 B swizzle: 16-byte
      // piece q of row r at r * 128 + ((q ^ (r & 7)) << 4), conflict-free), stored by one TMA
      // copy; the buffer is reused once the previous copy has read it
      if (lane == 0) asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
      __syncwarp();
      const uint32_t sb = smem_u32(stage) + lane * 128;
#pragma unroll
      for (int q = 0; q < 8; ++q)
        asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};" ::"r"(sb + ((q ^ (lane & 7)) << 4)), "f"(v[4 * q]),
                     "f"(v[4 * q + 1]), "f"(v[4 * q + 2]), "f"(v[4 * q + 3])
                     : "memory");
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      __syncwarp();
      if (lane == 0) {
        asm volatile(
            "cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];\n\t"
            "cp.async.bulk.commit_group;" ::"l"(reinterpret_cast<uint64_t>(&p.tma_out)),
            "r"(col0), "r"(row - lane), "r"(smem_u32(stage))
            : "memory");
      }
    } else if (p.out_f32) {
      float* op = static_cast<float*>(p.out) + static_cast<long long>(row) * p.ldo + col0;
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const uint4 a = make_uint4(__float_as_uint(v[8 * q]), __float_as_uint(v[8 * q + 1]),
                                   __float_as_uint(v[8 * q + 2]), __float_as_uint(v[8 * q + 3]));
        const uint4 b = make_uint4(__float_as_uint(v[8 * q + 4]), __float_as_uint(v[8 * q + 5]),
                                   __float_as_uint(v[8 * q + 6]), __float_as_uint(v[8 * q + 7]));
        st_global_32B(op + 8 * q, a, b);
      }
    } else {
      bf16* op = static_cast<bf16*>(p.out) + static_cast<long long>(row) * p.ldo + col0;
#pragma unroll
      for (int q = 0; q < 2; ++q) {
        const uint4 a = make_uint4(pack_bf16x2(v[16 * q], v[16 * q + 1]), pack_bf16x2(v[16 * q + 2], v[16 * q + 3]),
                                   pack_bf16x2(v[16 * q + 4], v[16 * q + 5]), pack_bf16x2(v[16 * q + 6], v[16 * q + 7]));
        const uint4 b = make_uint4(pack_bf16x2(v[16 * q + 8], v[16 * q + 9]), pack_bf16x2(v[16 * q + 10], v[16 * q + 11]),
                                   pack_bf16x2(v[16 * q + 12], v[16 * q + 13]),
                                   pack_bf16x2(v[16 * q + 14], v[16 * q + 15]));
        st_global_32B(op + 16 * q, a, b);
      }
    }
  }
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kGemmThreads, 1)
    gemm_bf16_tcgen05(const __grid_constant__ GemmArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kGemmStages * kGemmABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kGemmStages * kGemmStageBytes + 8 * kGemmStageOut);
  uint64_t* empty = full + kGemmStages;
  uint64_t* tfull = empty + kGemmStages;
  uint64_t* tempty = tfull + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(tempty + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  const int m_tiles = (p.M + kGemmTileM - 1) / kGemmTileM;
  const int n_tiles = (p.N + kGemmBN - 1) / kGemmBN;
  const int num_tiles = m_tiles * n_tiles;
  const int kb = (p.K + kGemmBK - 1) / kGemmBK;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGemmStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 2 * p.epi_warps);  // one arrival per epilogue warp of the pair
    }
    fence_mbar_init();
  }
  if (warp == 1) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                 "r"(512)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // both CTAs' barriers are initialised before any cross-CTA traffic
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  bool failed = false;

  if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kGemmRegsControl));
  if (warp == 0) {
    if (lane == 0 && kb > 0) {
      tma_prefetch_desc(&p.tma_a);
      tma_prefetch_desc(&p.tma_b);
      int stage = 0;
      uint32_t phase = 0;
      for (int tile = pair; tile < num_tiles && !failed; tile += n_pairs) {
        int mt, nt;
        tile_coords(tile, m_tiles, n_tiles, p.group, mt, nt);
        const int nb0 = nt * kGemmBN + static_cast<int>(rank) * kGemmBRows;  // this CTA's first B row
        // kGatherRows: the union rows of this CTA's B half (one group of 128 rows, or two of
        // 64) are the same for every K block.  A TMA instruction costs the issuing thread
        // about 140 cycles (measured), so each stage issues exactly one B copy (two for
        // 64-row groups), never a predicated run of them.
        int row0 = 0, row1 = 0;
        if (p.b_gather == kGatherRows) {
          const int g0 = nb0 / p.b_group;
          row0 = p.b_idx[g0] * p.b_group;
          if (p.b_group == 64) row1 = p.b_idx[g0 + 1] * 64;
        }
        for (int k = 0; k < kb; ++k) {
          if (!mbar_wait_cluster(&empty[stage], phase ^ 1, p.err)) { failed = true; break; }
          if (rank == 0) mbar_arrive_expect_tx(&full[stage], 2 * kGemmStageBytes);
          const uint32_t lf = map_to_rank(&full[stage], 0);
          tma_load_2d_pair(sA + stage * kGemmABytes, &p.tma_a, lf, k * kGemmBK,
                           mt * kGemmTileM + static_cast<int>(rank) * kGemmBM);
          uint8_t* dB = sB + stage * kGemmBBytes;
          if (p.b_gather == kGatherNone) {
            tma_load_2d_pair(dB, &p.tma_b, lf, k * kGemmBK, nb0);
          } else if (p.b_gather == kGatherRows) {
            // 64-row groups stack in the same 128-byte swizzled layout one 128-row box
            // produces (8-row atoms of 1024 B)
            tma_load_2d_pair(dB, &p.tma_b, lf, k * kGemmBK, row0);
            if (p.b_group == 64) tma_load_2d_pair(dB + 64 * 128, &p.tma_b, lf, k * kGemmBK, row1);
          } else {  // kGatherKCols
            tma_load_2d_pair(dB, &p.tma_b, lf, p.b_idx[k] * kGemmBK, nb0);
          }
          if (++stage == kGemmStages) { stage = 0; phase ^= 1; }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && rank == 0 && kb > 0) {
      constexpr uint32_t idesc = idesc_bf16(kGemmTileM, kGemmBN);
      // descriptors built once: stages and K slices only add offsets to the start
      // address field (address >> 4), which keeps this thread's issue rate at the tensor
      // pipe's rate
      const uint64_t da = sw128_desc(smem_u32(sA)), db = sw128_desc(smem_u32(sB));
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int tile = pair; tile < num_tiles && !failed; tile += n_pairs) {
        if (!mbar_wait_cluster(&tempty[acc], acc_phase ^ 1, p.err)) { failed = true; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + acc * kGemmBN;
        for (int k = 0; k < kb; ++k) {
          if (!mbar_wait_cluster(&full[stage], phase, p.err)) { failed = true; break; }
          tc_fence_after();
          const uint64_t a0 = da + static_cast<uint64_t>(stage * (kGemmABytes >> 4));
          const uint64_t b0 = db + static_cast<uint64_t>(stage * (kGemmBBytes >> 4));
#pragma unroll
          for (int kk = 0; kk < kGemmBK / 16; ++kk)
            mma_pair_ss(d_tmem, a0 + kk * 2, b0 + kk * 2, idesc, kk == 0 ? (k != 0) : 1u);
          commit_pair(&empty[stage]);
          if (++stage == kGemmStages) { stage = 0; phase ^= 1; }
        }
        commit_pair(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1;
      }
    }
  }
  } else {
    asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kGemmRegsEpilogue));
    const int sub = warp & 3;  // TMEM lane quarter this warp may access
    // with 8 epilogue warps each lane quarter's two warps take 128 columns of every tile; with
    // 4, warps 4..7 take all 256 and warps 8..11 have no work
    const int half = (warp - 4) >> 2;
    uint8_t* stage = sB + kGemmStages * kGemmBBytes + (warp - 4) * kGemmStageOut;  // 1024-byte aligned
    const int c_lo = p.epi_warps == 8 ? 128 * half : 0, c_n = p.epi_warps == 8 ? 128 : kGemmBN;
    const bool idle = p.epi_warps != 8 && half == 1;
    const int r_in_tile = static_cast<int>(rank) * kGemmBM + sub * 32 + lane;
    // the wide epilogue reads and writes 32-byte pieces: bases and row pitches must keep them aligned
    const int osz = p.out_f32 ? 4 : 2, rsz = p.res_f32 ? 4 : 2;
    const bool wide_ok = ((reinterpret_cast<uintptr_t>(p.out) | reinterpret_cast<uintptr_t>(p.res)) & 31u) == 0 &&
                         (p.ldo * osz) % 32 == 0 && (p.ldr * rsz) % 32 == 0;
    const bool wide_out = (reinterpret_cast<uintptr_t>(p.out) & 31u) == 0 && (p.ldo * osz) % 32 == 0;
    const uint32_t tempty_leader0 = map_to_rank(&tempty[0], 0), tempty_leader1 = map_to_rank(&tempty[1], 0);
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int tile = pair; tile < num_tiles && !idle; tile += n_pairs) {
      int mt, nt;
      tile_coords(tile, m_tiles, n_tiles, p.group, mt, nt);
      const int row = mt * kGemmTileM + r_in_tile;
      if (kb > 0) {
        // every lane waits; the warp leaves together if any lane gave up, so that the
        // warp-collective TMEM loads below are never split
        const bool ok = mbar_wait_cluster(&tfull[acc], acc_phase, p.err);
        if (!__all_sync(0xffffffffu, ok)) { failed = true; break; }
        tc_fence_after();
      }
      const uint32_t tacc = tmem_base + (static_cast<uint32_t>(sub * 32) << 16) + acc * kGemmBN;
      // warp-uniform choice: the TMEM loads on both paths are warp-collective
      if (p.mode == kEpiGatedRes && kb > 0 && nt * kGemmBN + c_lo + c_n <= p.N && wide_ok &&
          __all_sync(0xffffffffu, row < p.M)) {
        for (int c = c_lo; c < c_lo + c_n; c += 128) epilogue_gated_row<4>(p, row, nt * kGemmBN + c, tacc + c, stage);
      } else {
        for (int c = c_lo; c < c_lo + c_n; c += 32) {
          const int col0 = nt * kGemmBN + c;
          if (col0 >= p.N) break;
          float v[32];
          if (kb > 0) {
            tmem_ld32(tacc + c, v);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = 0.f;
          }
          epilogue_chunk(p, row, col0, v, wide_out);
        }
      }
      if (kb > 0) {
        // this accumulator is read out: one arrival per warp on the even CTA's barrier
        tc_fence_before();
        __syncwarp();
        if (lane == 0) {
          if (rank == 0)
            mbar_arrive(&tempty[acc]);
          else
            asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(acc ? tempty_leader1 : tempty_leader0)
                         : "memory");
        }
      }
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1;
    }
    // the output copies read this warp's staging buffer: complete before the CTA exits
    if (lane == 0) asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
    __syncwarp();
  }

  if (failed) drain_after_error();
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the even CTA's MMAs read this CTA's shared memory and TMEM until here
  tc_fence_after();
  if (warp == 1)
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem_base), "r"(512) : "memory");
}

}  // namespace

cudaError_t gemm_prepare() {
  cudaError_t e = cudaFuncSetAttribute(gemm_bf16_tcgen05, cudaFuncAttributeMaxDynamicSharedMemorySize, kGemmSmem);
  if (e != cudaSuccess) return e;
  // The epilogue warpgroups' setmaxnreg.inc is satisfied only by the registers warpgroup 0
  // releases, which assumes kGemmRegsLaunch registers per thread at launch: a build that
  // allocated fewer would make the increase wait forever, so it is refused here.
  cudaFuncAttributes at;
  if ((e = cudaFuncGetAttributes(&at, gemm_bf16_tcgen05)) != cudaSuccess) return e;
  return at.numRegs == kGemmRegsLaunch ? cudaSuccess : cudaErrorNotSupported;
}

cudaError_t launch_gemm(const GemmArgs& a, int num_sms, cudaStream_t s) {
  const int m_tiles = (a.M + kGemmTileM - 1) / kGemmTileM;
  const int n_tiles = (a.N + kGemmBN - 1) / kGemmBN;
  const int tiles = m_tiles * n_tiles;
  if (tiles == 0) return cudaSuccess;
  const int pairs = tiles < num_sms / 2 ? tiles : num_sms / 2;
  if (a.epi_warps != 4 && a.epi_warps != 8) return cudaErrorInvalidValue;
  gemm_bf16_tcgen05<<<2 * pairs, kGemmThreads, kGemmSmem, s>>>(a);
  return cudaGetLastError();
}

}  // namespace dfs
