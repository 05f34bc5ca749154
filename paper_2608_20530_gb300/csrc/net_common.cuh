// Row-worker helpers shared by the scoring-network kernels (net_fused.cu, net_cluster.cu):
// shared-memory operand layouts, warp-level mma.sync products, packed fp16 arithmetic, and
// the attention core of one head for 16 queries.
#pragma once
#include "tc_ptx.cuh"

namespace lilicorr {
namespace net {
using namespace tc;

constexpr uint32_t CHUNK = 128 * 128;     // 128 rows x 64 bf16, one swizzled K chunk

// tcgen05 load / store of 16 columns (lane = row of the calling warp's quarter)
__device__ __forceinline__ void ld16f(uint32_t taddr, float (&v)[16]) {
  uint32_t u[16];
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32"
      " {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(u[0]), "=r"(u[1]), "=r"(u[2]), "=r"(u[3]), "=r"(u[4]), "=r"(u[5]), "=r"(u[6]),
        "=r"(u[7]), "=r"(u[8]), "=r"(u[9]), "=r"(u[10]), "=r"(u[11]), "=r"(u[12]), "=r"(u[13]),
        "=r"(u[14]), "=r"(u[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
  for (int j = 0; j < 16; ++j) v[j] = __uint_as_float(u[j]);
}
__device__ __forceinline__ void st16f(uint32_t taddr, const float (&v)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0],"
      " {%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
      "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
      "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
      "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
      "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
      "r"(__float_as_uint(v[15]))
      : "memory");
}

// ---- thread-block clusters: distributed shared memory and remote barrier signalling
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// address of the same shared-memory location in CTA `rank` of the cluster
__device__ __forceinline__ uint32_t peer_addr(uint32_t local, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local), "r"(rank));
  return r;
}
// 16 / 4 bytes into a peer's shared memory; the bytes count toward the transaction count
// of the peer's mbarrier `rbar` (peer address), which completes when they have landed
__device__ __forceinline__ void st_peer16(uint32_t raddr, const uint4& v, uint32_t rbar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, [%5];"
      ::"r"(raddr), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(rbar) : "memory");
}
__device__ __forceinline__ void st_peer4(uint32_t raddr, uint32_t v, uint32_t rbar) {
  asm volatile("st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];"
               ::"r"(raddr), "r"(v), "r"(rbar) : "memory");
}
// `bytes` (a multiple of 16) of this CTA's shared memory at src into a peer's shared memory
// at dst (peer address) by the bulk-copy engine, counted on the peer's mbarrier rbar (peer
// address); the writers of src must have fenced their generic-proxy writes (and synced)
__device__ __forceinline__ void bulk_to_peer(uint32_t dst, const void* src, uint32_t bytes,
                                             uint32_t rbar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      ::"r"(dst), "r"(smem_u32(src)), "r"(bytes), "r"(rbar) : "memory");
}
// wait until this thread's bulk copies have read their sources
__device__ __forceinline__ void bulk_wait_read() {
  asm volatile("cp.async.bulk.commit_group;\n cp.async.bulk.wait_group.read 0;" ::: "memory");
}
// a float of a peer's shared memory (peer address)
__device__ __forceinline__ float ld_peer_f32(uint32_t raddr) {
  float v;
  asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(raddr) : "memory");
  return v;
}
// one arrival on a peer's mbarrier (peer address), releasing this thread's prior writes
__device__ __forceinline__ void mbar_arrive_peer(uint32_t rbar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(rbar)
               : "memory");
}
// wait for a phase whose completion was signalled by other CTAs of the cluster (bounded)
__device__ __forceinline__ bool mbar_try_wait_cluster(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_cluster(uint64_t* bar, uint32_t parity, long long limit) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait_cluster(bar, parity))
    if (clock64() - t0 > limit) return false;
  return true;
}
// The same waits with a suspend-time hint: a waiting warp sleeps until the phase
// completes (or about `ns` nanoseconds pass) instead of re-polling, leaving its issue
// slots to the warps that do the work.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity, uint32_t ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(ns)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_try_wait_cluster_sleep(uint64_t* bar, uint32_t parity,
                                                            uint32_t ns) {
  uint32_t ok;
  asm volatile(
      "{\n .reg .pred p;\n mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n"
      " selp.u32 %0, 1, 0, p;\n}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(ns)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_sleep(uint64_t* bar, uint32_t parity, long long limit) {
  if (mbar_try_wait(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait_sleep(bar, parity, 20000u))
    if (clock64() - t0 > limit) return false;
  return true;
}
__device__ __forceinline__ bool mbar_wait_cluster_sleep(uint64_t* bar, uint32_t parity,
                                                        long long limit) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const long long t0 = clock64();
  while (!mbar_try_wait_cluster_sleep(bar, parity, 20000u))
    if (clock64() - t0 > limit) return false;
  return true;
}
// all threads of all CTAs of the cluster
__device__ __forceinline__ void cluster_sync() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n barrier.cluster.wait.acquire.aligned;"
               ::: "memory");
}

// q / k / v of one head: [128 rows][32] 16-bit values, 64-byte rows, pieces XOR-swizzled
// by row pair so that ldmatrix over 8 consecutive rows touches 8 distinct bank groups
__device__ __forceinline__ uint32_t qkv_off(int row, int piece) {
  return (uint32_t)(row * 64 + ((piece ^ ((row >> 1) & 3)) << 4));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t (&r)[4]) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(addr));
}
// warp-level products: S = Q K^T with bf16 operands, O += P V with fp16 operands
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                               uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                              uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, "
      "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ float ex2f(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}
// two fp32 -> fp16x2 (round to nearest), and 2^x on both halves in one instruction
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  const __half2 v = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&v);
}
__device__ __forceinline__ uint32_t ex2_h2(uint32_t x) {
  uint32_t y;
  asm("ex2.approx.f16x2 %0, %1;" : "=r"(y) : "r"(x));
  return y;
}
__device__ __forceinline__ float2 h2_to_f2(uint32_t x) {
  return __half22float2(*reinterpret_cast<const __half2*>(&x));
}
// SiLU(z) = z sigmoid(z) = z (1 + tanh(z / 2)) / 2 for two values with one packed fp16
// tanh (one MUFU operation per pair; the result feeds a bf16 operand, whose rounding is
// coarser than the fp16 tanh)
__device__ __forceinline__ void silu2(float& z0, float& z1) {
  uint32_t t;
  asm("tanh.approx.f16x2 %0, %1;" : "=r"(t) : "r"(pack_h2(0.5f * z0, 0.5f * z1)));
  const float2 tf = h2_to_f2(t);
  z0 = 0.5f * z0 * (1.0f + tf.x);
  z1 = 0.5f * z1 * (1.0f + tf.y);
}
// 16-byte asynchronous global -> shared copies (L2 only), many in flight per thread
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
// 4-byte asynchronous global -> shared copy (for gathers and transposes)
__device__ __forceinline__ void cp_async4(void* dst, const void* src) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.commit_group;\n cp.async.wait_group 0;" ::: "memory");
}

// 8 bf16 / fp16 of v[0..7] as one 16-byte piece
__device__ __forceinline__ uint4 pack8(const float* v) {
  uint4 w;
  w.x = pack_bf16x2(v[0], v[1]);
  w.y = pack_bf16x2(v[2], v[3]);
  w.z = pack_bf16x2(v[4], v[5]);
  w.w = pack_bf16x2(v[6], v[7]);
  return w;
}
__device__ __forceinline__ uint4 pack8h(const float* v) {
  uint4 w;
  w.x = pack_h2(v[0], v[1]);
  w.y = pack_h2(v[2], v[3]);
  w.z = pack_h2(v[4], v[5]);
  w.w = pack_h2(v[6], v[7]);
  return w;
}

// Write 32 values (columns c0..c0+31 of row r) as bf16 into a swizzled operand buffer
// holding 64-column chunks.
__device__ __forceinline__ void put32(uint8_t* buf, int r, int c0, const float (&v)[32]) {
  uint8_t* ch = buf + (c0 >> 6) * CHUNK;
  const int p0 = (c0 & 63) >> 3;
#pragma unroll
  for (int p = 0; p < 4; ++p) *reinterpret_cast<uint4*>(ch + swz(r, p0 + p)) = pack8(v + 8 * p);
}

__device__ __forceinline__ void ld32f(uint32_t taddr, float (&v)[32]) {
  uint32_t u[32];
  tmem_ld32(taddr, u);
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(u[j]);
}
__device__ __forceinline__ void st32f(uint32_t taddr, const float (&v)[32]) {
  uint32_t u[32];
#pragma unroll
  for (int j = 0; j < 32; ++j) u[j] = __float_as_uint(v[j]);
  tmem_st32(taddr, u);
}

// Attention core of one head (App. A: bidirectional attention over the L*K nodes with the
// signed slot-distance and same-slot biases) for the 16 queries q0..q0+15 of one warp, in
// blocks of KB (32 or 64) keys with an online softmax in log2 units; probabilities P = 2^(S - max) as
// fp16 pairs (one MUFU operation per pair). q, k (bf16) and v (fp16) of the head are at qb,
// qb + 8192 and qb + 16384 (qkv_off layout). s_slot: slot of each node; sd: the head's
// distance bias (log2 units) indexed by sj - si; same_l2: its same-slot bias (log2 units).
// Out: the unnormalised outputs o[nb][e] in the mma m16n8 fragment layout (rows
// q0 + lane/4 and q0 + lane/4 + 8, columns 8nb + 2(lane%4) + (e&1)) and the reciprocals of
// the two rows' softmax sums.
template <int KB = 64>
__device__ __forceinline__ void head_attention(uint32_t qb, int LK, int K, const uint8_t* s_slot,
                                               const float* sd, float same_l2, int q0, int lane,
                                               float (&o)[4][4], float& inv0, float& inv1) {
  const uint32_t kb = qb + 8192, vb = qb + 16384;
  const int g8 = lane >> 2, t4 = lane & 3;
  const float qscale = rsqrtf(32.f) * 1.4426950408889634f;   // 1/sqrt(head width), log2 units
  const bool k8 = (K & 7) == 0;
  uint32_t qa[2][4];
#pragma unroll
  for (int ks = 0; ks < 2; ++ks)
    ldsm_x4(qb + qkv_off(q0 + (lane & 15), ks * 2 + (lane >> 4)), qa[ks]);
  const int i0 = q0 + g8, i1 = i0 + 8;
  const int si0 = s_slot[i0], si1 = s_slot[i1];
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
#pragma unroll
  for (int nb = 0; nb < 4; ++nb) o[nb][0] = o[nb][1] = o[nb][2] = o[nb][3] = 0.f;
#pragma unroll 1
  for (int kb0 = 0; kb0 < LK; kb0 += KB) {
    constexpr int NB = KB / 8;                     // 8-key tiles of the block
    float s4[NB][4];
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) s4[nb][0] = s4[nb][1] = s4[nb][2] = s4[nb][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 2; ++ks)
#pragma unroll
      for (int nb = 0; nb < NB; nb += 2) {
        uint32_t bf[4];
        const int key = kb0 + nb * 8 + (lane & 7) + ((lane >> 4) << 3);
        ldsm_x4(kb + qkv_off(key, ks * 2 + ((lane >> 3) & 1)), bf);
        mma_bf16_16816(s4[nb], qa[ks], bf[0], bf[1]);
        mma_bf16_16816(s4[nb + 1], qa[ks], bf[2], bf[3]);
      }
    float bm0 = -INFINITY, bm1 = -INFINITY;
    if (k8) {
      // K % 8 == 0: the 8 keys of a tile share one slot, so one bias per query row
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int jt = kb0 + nb * 8;
        const bool in = jt < LK;
        const int sj = s_slot[in ? jt : 0];
        const float b0 = sd[sj - si0] + (si0 == sj ? same_l2 : 0.f);
        const float b1 = sd[sj - si1] + (si1 == sj ? same_l2 : 0.f);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float v = in ? fmaf(s4[nb][e], qscale, e < 2 ? b0 : b1) : -INFINITY;
          s4[nb][e] = v;
          if (e < 2) bm0 = fmaxf(bm0, v); else bm1 = fmaxf(bm1, v);
        }
      }
    } else {
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int j0 = kb0 + nb * 8 + 2 * t4;
        const uint32_t sp = *reinterpret_cast<const uint16_t*>(s_slot + j0);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int jj = j0 + (e & 1);
          const int sj = (e & 1) ? (int)(sp >> 8) : (int)(sp & 255u);
          const int si = e < 2 ? si0 : si1;
          const float v = jj < LK
                              ? s4[nb][e] * qscale + sd[sj - si] + (si == sj ? same_l2 : 0.f)
                              : -INFINITY;
          s4[nb][e] = v;
          if (e < 2) bm0 = fmaxf(bm0, v); else bm1 = fmaxf(bm1, v);
        }
      }
    }
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 1));
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 2));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 1));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 2));
    const float mn0 = fmaxf(m0, bm0), mn1 = fmaxf(m1, bm1);
    const float c0 = ex2f(m0 - mn0), c1 = ex2f(m1 - mn1);   // 0 on the first block
    m0 = mn0;
    m1 = mn1;
    l0 *= c0;
    l1 *= c1;
#pragma unroll
    for (int nb = 0; nb < 4; ++nb) {
      o[nb][0] *= c0; o[nb][1] *= c0;
      o[nb][2] *= c1; o[nb][3] *= c1;
    }
    uint32_t pa[NB / 2][4];
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      const uint32_t h01 = ex2_h2(pack_h2(s4[nb][0] - mn0, s4[nb][1] - mn0));
      const uint32_t h23 = ex2_h2(pack_h2(s4[nb][2] - mn1, s4[nb][3] - mn1));
      const float2 f01 = h2_to_f2(h01), f23 = h2_to_f2(h23);
      l0 += f01.x + f01.y;
      l1 += f23.x + f23.y;
      const int kk = nb >> 1;
      if ((nb & 1) == 0) {
        pa[kk][0] = h01;
        pa[kk][1] = h23;
      } else {
        pa[kk][2] = h01;
        pa[kk][3] = h23;
      }
    }
#pragma unroll
    for (int kk = 0; kk < NB / 2; ++kk)
#pragma unroll
      for (int nb = 0; nb < 4; nb += 2) {
        uint32_t vf[4];
        const int key = kb0 + kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        ldsm_x4_t(vb + qkv_off(key, nb + (lane >> 4)), vf);
        mma_f16_16816(o[nb], pa[kk], vf[0], vf[1]);
        mma_f16_16816(o[nb + 1], pa[kk], vf[2], vf[3]);
      }
  }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  inv0 = 1.0f / l0;
  inv1 = 1.0f / l1;
}


// The attention core above over a range of keys, unnormalised, for kernels that split
// the keys of one head over two warps and merge the halves afterwards: q at qb (local
// query rows q0..q0+15), k and v of every key at kb / vb (rows = key index, qkv_off
// layout), keys [key0, key0 + nkeys) with keys at or past LK masked (the first 64-key
// block of the range must hold at least one unmasked key). qoff: the node index of local
// query row 0 (for its slot). Out: o[nb][e] as above, the two rows' running maxima m0, m1
// (log2 units) and sums l0, l1 of 2^(s - m) over the range (summed over the row's lanes).
__device__ __forceinline__ void head_attention_part(uint32_t qb, uint32_t kb, uint32_t vb, int key0,
                                                    int nkeys, int LK, int K,
                                                    const uint8_t* s_slot, const float* sd,
                                                    float same_l2, int q0, int qoff, int lane,
                                                    float (&o)[4][4], float& m0, float& m1,
                                                    float& l0, float& l1) {
  constexpr int KB = 64, NB = KB / 8;
  const int g8 = lane >> 2, t4 = lane & 3;
  const float qscale = rsqrtf(32.f) * 1.4426950408889634f;   // 1/sqrt(head width), log2 units
  const bool k8 = (K & 7) == 0;
  uint32_t qa[2][4];
#pragma unroll
  for (int ks = 0; ks < 2; ++ks)
    ldsm_x4(qb + qkv_off(q0 + (lane & 15), ks * 2 + (lane >> 4)), qa[ks]);
  const int si0 = s_slot[qoff + q0 + g8], si1 = s_slot[qoff + q0 + g8 + 8];
  m0 = -INFINITY;
  m1 = -INFINITY;
  l0 = 0.f;
  l1 = 0.f;
#pragma unroll
  for (int nb = 0; nb < 4; ++nb) o[nb][0] = o[nb][1] = o[nb][2] = o[nb][3] = 0.f;
#pragma unroll 1
  for (int kb0 = key0; kb0 < key0 + nkeys; kb0 += KB) {
    float s4[NB][4];
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) s4[nb][0] = s4[nb][1] = s4[nb][2] = s4[nb][3] = 0.f;
#pragma unroll
    for (int ks = 0; ks < 2; ++ks)
#pragma unroll
      for (int nb = 0; nb < NB; nb += 2) {
        uint32_t bf[4];
        const int key = kb0 + nb * 8 + (lane & 7) + ((lane >> 4) << 3);
        ldsm_x4(kb + qkv_off(key, ks * 2 + ((lane >> 3) & 1)), bf);
        mma_bf16_16816(s4[nb], qa[ks], bf[0], bf[1]);
        mma_bf16_16816(s4[nb + 1], qa[ks], bf[2], bf[3]);
      }
    float bm0 = -INFINITY, bm1 = -INFINITY;
    if (k8) {
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int jt = kb0 + nb * 8;
        const bool in = jt < LK;
        const int sj = s_slot[in ? jt : 0];
        const float b0 = sd[sj - si0] + (si0 == sj ? same_l2 : 0.f);
        const float b1 = sd[sj - si1] + (si1 == sj ? same_l2 : 0.f);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float v = in ? fmaf(s4[nb][e], qscale, e < 2 ? b0 : b1) : -INFINITY;
          s4[nb][e] = v;
          if (e < 2) bm0 = fmaxf(bm0, v); else bm1 = fmaxf(bm1, v);
        }
      }
    } else {
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int j0 = kb0 + nb * 8 + 2 * t4;
        const uint32_t sp = *reinterpret_cast<const uint16_t*>(s_slot + j0);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int jj = j0 + (e & 1);
          const int sj = (e & 1) ? (int)(sp >> 8) : (int)(sp & 255u);
          const int si = e < 2 ? si0 : si1;
          const float v = jj < LK
                              ? s4[nb][e] * qscale + sd[sj - si] + (si == sj ? same_l2 : 0.f)
                              : -INFINITY;
          s4[nb][e] = v;
          if (e < 2) bm0 = fmaxf(bm0, v); else bm1 = fmaxf(bm1, v);
        }
      }
    }
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 1));
    bm0 = fmaxf(bm0, __shfl_xor_sync(0xffffffffu, bm0, 2));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 1));
    bm1 = fmaxf(bm1, __shfl_xor_sync(0xffffffffu, bm1, 2));
    const float mn0 = fmaxf(m0, bm0), mn1 = fmaxf(m1, bm1);
    const float c0 = ex2f(m0 - mn0), c1 = ex2f(m1 - mn1);   // 0 on the first block
    m0 = mn0;
    m1 = mn1;
    l0 *= c0;
    l1 *= c1;
#pragma unroll
    for (int nb = 0; nb < 4; ++nb) {
      o[nb][0] *= c0; o[nb][1] *= c0;
      o[nb][2] *= c1; o[nb][3] *= c1;
    }
    uint32_t pa[NB / 2][4];
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      const uint32_t h01 = ex2_h2(pack_h2(s4[nb][0] - mn0, s4[nb][1] - mn0));
      const uint32_t h23 = ex2_h2(pack_h2(s4[nb][2] - mn1, s4[nb][3] - mn1));
      const float2 f01 = h2_to_f2(h01), f23 = h2_to_f2(h23);
      l0 += f01.x + f01.y;
      l1 += f23.x + f23.y;
      const int kk = nb >> 1;
      if ((nb & 1) == 0) {
        pa[kk][0] = h01;
        pa[kk][1] = h23;
      } else {
        pa[kk][2] = h01;
        pa[kk][3] = h23;
      }
    }
#pragma unroll
    for (int kk = 0; kk < NB / 2; ++kk)
#pragma unroll
      for (int nb = 0; nb < 4; nb += 2) {
        uint32_t vf[4];
        const int key = kb0 + kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        ldsm_x4_t(vb + qkv_off(key, nb + (lane >> 4)), vf);
        mma_f16_16816(o[nb], pa[kk], vf[0], vf[1]);
        mma_f16_16816(o[nb + 1], pa[kk], vf[2], vf[3]);
      }
  }
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
}

// one 16-byte store into a peer's shared memory (peer address), ordinary (weak) semantics;
// a later release arrival on the peer's barrier publishes it
__device__ __forceinline__ void st_peer_v4(uint32_t raddr, const uint4& v) {
  asm volatile("st.shared::cluster.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(raddr), "r"(v.x),
               "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

}  // namespace net
}  // namespace lilicorr
