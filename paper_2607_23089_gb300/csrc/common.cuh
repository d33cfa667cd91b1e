// common.cuh -- shared device helpers for librowop's sm_103a kernels:
// constants of the row decomposition, inline-PTX wrappers for mbarrier,
// bulk (TMA) copies, cluster barriers and distributed shared memory, 16-byte
// chunk packing for fp32 / bf16, and warp butterfly reductions.
//
// Row decomposition used by every kernel (the row-length-dispatched family of
// §2.1: small_row_kernel / medium_row_kernel / large_row_kernel):
//   * a row is viewed through its 16-byte-aligned "window": chunk c holds the
//     16 bytes at floor16(row start) + 16c, i.e. E = 16/sizeof(T) elements;
//     h = (row start mod 16) / sizeof(T) leading elements of chunk 0 and the
//     elements past the row end in the last chunk are not part of the row;
//   * SMALL rows live in registers of a group of G lanes, lane `sub` holding
//     chunks sub, sub+G, sub+2G, ...;
//   * MEDIUM and LARGE rows are cut into tiles of 64 chunks (1 KiB); one warp
//     reduces one tile (lane l: chunks l and l+32 of the tile) to a tile
//     partial, and warp 0 combines the K tile partials of the row in a fixed
//     order (lane l takes tiles l, l+32, l+64, ... in turn, then a 5-level
//     xor butterfly).  The order depends on nothing but the row's length and
//     alignment, so which CTA or cluster rank held a tile never changes a bit
//     of the result.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace rowop {

enum OpKind : int { kSoftmax = 0, kLogSoftmax = 1, kLayerNorm = 2, kRmsNorm = 3 };

constexpr uint32_t kStatusTimeout = 1u;     // a bounded device wait ran out
constexpr uint32_t kStatusBadOffsets = 2u;  // ragged rows rejected

constexpr int kChunkBytes = 16;
constexpr int kTileChunks = 64;
constexpr int kTileBytes = kTileChunks * kChunkBytes;  // 1 KiB
constexpr int kCtaThreads = 256;
constexpr int kCtaWarps = kCtaThreads / 32;
constexpr unsigned kFullMask = 0xffffffffu;

// launch_by_rows (§2.1): bucket of a row of len elements of esize bytes --
// SMALL up to 4 KiB, MEDIUM up to 32 KiB, LARGE beyond.
constexpr int64_t kSmallMaxBytes = 4096;
constexpr int64_t kMediumMaxBytes = 32768;
enum Bucket : int { kSmall = 0, kMedium = 1, kLarge = 2 };
__host__ __device__ __forceinline__ int bucket_of(int64_t len, int esize) {
  const int64_t bytes = len * esize;
  return bytes <= kSmallMaxBytes ? kSmall : (bytes <= kMediumMaxBytes ? kMedium : kLarge);
}

// One ragged row as the classify pass lists it.
struct RowRec {
  int64_t start;  // first element of the row in the packed buffer
  int64_t n;      // its length
};

template <typename T>
struct Elem;
template <>
struct Elem<float> {
  static constexpr int kPerChunk = 4;
  static constexpr int kSize = 4;
};
template <>
struct Elem<__nv_bfloat16> {
  static constexpr int kPerChunk = 8;
  static constexpr int kSize = 2;
};
template <>
struct Elem<__half> {
  static constexpr int kPerChunk = 8;
  static constexpr int kSize = 2;
};

// ---------------------------------------------------------------------------
// fp32 <-> element conversion, whole 16-byte chunks
// ---------------------------------------------------------------------------
__device__ __forceinline__ void unpack_bf16x2(uint32_t w, float &lo, float &hi) {
  lo = __uint_as_float(w << 16);
  hi = __uint_as_float(w & 0xffff0000u);
}
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 b = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&b);
}
__device__ __forceinline__ float2 half2_bits_to_float2(uint32_t w) {
  __half2 h = *reinterpret_cast<const __half2 *>(&w);
  return __half22float2(h);
}
__device__ __forceinline__ uint32_t float2_to_half2_bits(float2 v) {
  __half2 h = __float22half2_rn(v);  // round to nearest even, .x in the low half
  return *reinterpret_cast<uint32_t *>(&h);
}

// A 16-byte chunk of T <-> its E values in fp32.
template <typename T>
__device__ __forceinline__ void unpack(const uint4 &v, float (&f)[Elem<T>::kPerChunk]);
template <typename T>
__device__ __forceinline__ uint4 pack(const float (&f)[Elem<T>::kPerChunk]);
template <>
__device__ __forceinline__ void unpack<float>(const uint4 &v, float (&f)[4]) {
  f[0] = __uint_as_float(v.x);
  f[1] = __uint_as_float(v.y);
  f[2] = __uint_as_float(v.z);
  f[3] = __uint_as_float(v.w);
}
template <>
__device__ __forceinline__ void unpack<__nv_bfloat16>(const uint4 &v, float (&f)[8]) {
  unpack_bf16x2(v.x, f[0], f[1]);
  unpack_bf16x2(v.y, f[2], f[3]);
  unpack_bf16x2(v.z, f[4], f[5]);
  unpack_bf16x2(v.w, f[6], f[7]);
}
template <>
__device__ __forceinline__ void unpack<__half>(const uint4 &v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const float2 t = half2_bits_to_float2(w[i]);
    f[2 * i] = t.x;
    f[2 * i + 1] = t.y;
  }
}
template <>
__device__ __forceinline__ uint4 pack<float>(const float (&f)[4]) {
  return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]),
                    __float_as_uint(f[2]), __float_as_uint(f[3]));
}
template <>
__device__ __forceinline__ uint4 pack<__nv_bfloat16>(const float (&f)[8]) {
  return make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]),
                    pack_bf16x2(f[4], f[5]), pack_bf16x2(f[6], f[7]));
}
template <>
__device__ __forceinline__ uint4 pack<__half>(const float (&f)[8]) {
  return make_uint4(float2_to_half2_bits(make_float2(f[0], f[1])),
                    float2_to_half2_bits(make_float2(f[2], f[3])),
                    float2_to_half2_bits(make_float2(f[4], f[5])),
                    float2_to_half2_bits(make_float2(f[6], f[7])));
}

__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }
__device__ __forceinline__ float to_f32(__half v) { return __half2float(v); }
template <typename T>
__device__ __forceinline__ T from_f32(float v);
template <>
__device__ __forceinline__ float from_f32<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float v) {
  return __float2bfloat16_rn(v);
}
template <>
__device__ __forceinline__ __half from_f32<__half>(float v) {
  return __float2half_rn(v);
}

// One element of type T read as its raw bits into an fp32 value.
template <typename T>
__device__ __forceinline__ float load_elem(const T *p) {
  return to_f32(*p);
}

// ---------------------------------------------------------------------------
// Shift of two consecutive aligned chunks (A = chunk c-1, B = chunk c) by h
// elements: returns elements [E-h, 2E-h) of the concatenation A|B, i.e. the
// values that line up with window chunk c of a row that starts h elements
// past a 16-byte boundary.  h is uniform per row; every case is unrolled so
// no register array is indexed at run time.
// ---------------------------------------------------------------------------
template <int H>
__device__ __forceinline__ uint4 shift_words(const uint4 &A, const uint4 &B) {
  // word granularity (fp32 elements, or bf16 pairs at even shifts)
  const uint32_t w[8] = {A.x, A.y, A.z, A.w, B.x, B.y, B.z, B.w};
  return make_uint4(w[4 - H], w[5 - H], w[6 - H], w[7 - H]);
}
template <int HB>  // bf16 shift by an odd number of elements: HB = (h+1)/2
__device__ __forceinline__ uint4 shift_half(const uint4 &A, const uint4 &B) {
  const uint32_t w[8] = {A.x, A.y, A.z, A.w, B.x, B.y, B.z, B.w};
  // element pair (i0, i0+1) with i0 = 8 - h + 2k odd -> high half of word
  // (i0-1)/2 and low half of word (i0+1)/2.
  return make_uint4(__byte_perm(w[4 - HB], w[5 - HB], 0x5432),
                    __byte_perm(w[5 - HB], w[6 - HB], 0x5432),
                    __byte_perm(w[6 - HB], w[7 - HB], 0x5432),
                    __byte_perm(w[7 - HB], w[8 - HB], 0x5432));
}
template <typename T>
__device__ __forceinline__ uint4 shift_chunk(const uint4 &A, const uint4 &B, int h);
template <>
__device__ __forceinline__ uint4 shift_chunk<float>(const uint4 &A, const uint4 &B, int h) {
  switch (h) {
    case 1: return shift_words<1>(A, B);
    case 2: return shift_words<2>(A, B);
    case 3: return shift_words<3>(A, B);
    default: return B;
  }
}
template <>
__device__ __forceinline__ uint4 shift_chunk<__nv_bfloat16>(const uint4 &A, const uint4 &B,
                                                            int h);
template <>
__device__ __forceinline__ uint4 shift_chunk<__half>(const uint4 &A, const uint4 &B, int h) {
  return shift_chunk<__nv_bfloat16>(A, B, h);  // both are 2-byte elements
}
template <>
__device__ __forceinline__ uint4 shift_chunk<__nv_bfloat16>(const uint4 &A, const uint4 &B,
                                                            int h) {
  switch (h) {
    case 1: return shift_half<1>(A, B);
    case 2: return shift_words<1>(A, B);
    case 3: return shift_half<2>(A, B);
    case 4: return shift_words<2>(A, B);
    case 5: return shift_half<3>(A, B);
    case 6: return shift_words<3>(A, B);
    case 7: return shift_half<4>(A, B);
    default: return B;
  }
}

// ---------------------------------------------------------------------------
// Packed fp32 pairs (Blackwell f32x2 arithmetic, float2 builtins): a pair
// holds the even element of a chunk in .x and the odd element in .y.  Every
// sum over a run of chunks accumulates even and odd elements separately and
// adds the two halves at the end, in that fixed order.
// ---------------------------------------------------------------------------
typedef float2 f2;

__device__ __forceinline__ f2 f2_make(float lo, float hi) { return make_float2(lo, hi); }
__device__ __forceinline__ float f2_lo(f2 v) { return v.x; }
__device__ __forceinline__ float f2_hi(f2 v) { return v.y; }
__device__ __forceinline__ float f2_total(f2 v) { return __fadd_rn(v.x, v.y); }
__device__ __forceinline__ f2 f2_add(f2 a, f2 b) { return __fadd2_rn(a, b); }
__device__ __forceinline__ f2 f2_mul(f2 a, f2 b) { return __fmul2_rn(a, b); }
__device__ __forceinline__ f2 f2_fma(f2 a, f2 b, f2 c) { return __ffma2_rn(a, b, c); }
__device__ __forceinline__ f2 f2_bcast(float v) { return make_float2(v, v); }
// a - b as a + (-b); callers pass the negated operand once per row
__device__ __forceinline__ f2 f2_neg(f2 v) { return make_float2(-v.x, -v.y); }
// Keeps the halves whose flag is set, the other halves become `fill`.
__device__ __forceinline__ f2 f2_select(f2 v, bool keep_lo, bool keep_hi, float fill) {
  return make_float2(keep_lo ? v.x : fill, keep_hi ? v.y : fill);
}

// 16-byte chunk of T <-> pairs.  fp32: 2 pairs, bf16 / fp16: 4 pairs.
__device__ __forceinline__ f2 bf16x2_to_pair(uint32_t w) {
  return make_float2(__uint_as_float(w << 16), __uint_as_float(w & 0xffff0000u));
}
__device__ __forceinline__ uint32_t pair_to_bf16x2(f2 v) {
  __nv_bfloat162 b = __float22bfloat162_rn(v);  // round to nearest even, .x in the low half
  return *reinterpret_cast<uint32_t *>(&b);
}
template <typename T>
__device__ __forceinline__ void chunk_to_pairs(const uint4 &v, f2 (&p)[Elem<T>::kPerChunk / 2]);
template <typename T>
__device__ __forceinline__ uint4 pairs_to_chunk(const f2 (&p)[Elem<T>::kPerChunk / 2]);
template <>
__device__ __forceinline__ void chunk_to_pairs<float>(const uint4 &v, f2 (&p)[2]) {
  p[0] = make_float2(__uint_as_float(v.x), __uint_as_float(v.y));
  p[1] = make_float2(__uint_as_float(v.z), __uint_as_float(v.w));
}
template <>
__device__ __forceinline__ void chunk_to_pairs<__nv_bfloat16>(const uint4 &v, f2 (&p)[4]) {
  p[0] = bf16x2_to_pair(v.x);
  p[1] = bf16x2_to_pair(v.y);
  p[2] = bf16x2_to_pair(v.z);
  p[3] = bf16x2_to_pair(v.w);
}
template <>
__device__ __forceinline__ void chunk_to_pairs<__half>(const uint4 &v, f2 (&p)[4]) {
  p[0] = half2_bits_to_float2(v.x);
  p[1] = half2_bits_to_float2(v.y);
  p[2] = half2_bits_to_float2(v.z);
  p[3] = half2_bits_to_float2(v.w);
}
template <>
__device__ __forceinline__ uint4 pairs_to_chunk<float>(const f2 (&p)[2]) {
  return make_uint4(__float_as_uint(p[0].x), __float_as_uint(p[0].y), __float_as_uint(p[1].x),
                    __float_as_uint(p[1].y));
}
template <>
__device__ __forceinline__ uint4 pairs_to_chunk<__nv_bfloat16>(const f2 (&p)[4]) {
  return make_uint4(pair_to_bf16x2(p[0]), pair_to_bf16x2(p[1]), pair_to_bf16x2(p[2]),
                    pair_to_bf16x2(p[3]));
}
template <>
__device__ __forceinline__ uint4 pairs_to_chunk<__half>(const f2 (&p)[4]) {
  return make_uint4(float2_to_half2_bits(p[0]), float2_to_half2_bits(p[1]),
                    float2_to_half2_bits(p[2]), float2_to_half2_bits(p[3]));
}
// element e of a chunk's pair array
template <int NP>
__device__ __forceinline__ float pair_elem(const f2 (&p)[NP], int e) {
  return (e & 1) ? p[e >> 1].y : p[e >> 1].x;
}

// e^v as 2^(v * log2 e) on the MUFU unit; v is a difference x - m <= 0 here.
constexpr float kLog2e = 1.4426950408889634f;
// 2^v, the hardware approximation, with subnormal results flushed to zero:
// they arise only for exp(x - m) < 2^-126, terms that cannot move a row sum
// of at least 1 and outputs far below every absolute tolerance.
__device__ __forceinline__ float ex2_approx(float v) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(v));
  return r;
}
// exp(x - m) for both halves of a pair, given neg_m = (-m, -m)
__device__ __forceinline__ f2 f2_exp_shifted(f2 x, f2 neg_m) {
  const f2 u = __fmul2_rn(__fadd2_rn(x, neg_m), f2_bcast(kLog2e));
  return make_float2(ex2_approx(u.x), ex2_approx(u.y));
}
__device__ __forceinline__ float exp_shifted(float x, float m) {
  return ex2_approx(__fmul_rn(__fsub_rn(x, m), kLog2e));
}

// ---------------------------------------------------------------------------
// Warp butterflies.  Every lane of a width-W group ends with the same value:
// at each level both partners combine the same two operands, and fp32
// addition and max are commutative.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float group_sum(float v, int width) {
  for (int o = width >> 1; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(kFullMask, v, o));
  return v;
}
__device__ __forceinline__ float group_max(float v, int width) {
  for (int o = width >> 1; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFullMask, v, o));
  return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = __fadd_rn(v, __shfl_xor_sync(kFullMask, v, o));
  return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(kFullMask, v, o));
  return v;
}

// Merge of two (max, sum-of-exp) softmax partials; symmetric in its operands.
__device__ __forceinline__ void softmax_merge(float &m, float &s, float m2, float s2) {
  if (m2 == -INFINITY) return;
  if (m == -INFINITY) {
    m = m2;
    s = s2;
    return;
  }
  const float M = fmaxf(m, m2);
  s = __fadd_rn(__fmul_rn(s, expf(__fsub_rn(m, M))), __fmul_rn(s2, expf(__fsub_rn(m2, M))));
  m = M;
}
__device__ __forceinline__ void warp_softmax_merge(float &m, float &s) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float m2 = __shfl_xor_sync(kFullMask, m, o);
    const float s2 = __shfl_xor_sync(kFullMask, s, o);
    softmax_merge(m, s, m2, s2);
  }
}

// ---------------------------------------------------------------------------
// PTX wrappers: shared-memory addresses, mbarrier, bulk copy, cluster
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint64_t global_timer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile(
      "{\n\t.reg .b64 st;\n\t"
      "mbarrier.arrive.shared::cta.b64 st, [%0];\n\t}" ::"r"(bar)
      : "memory");
}
// A waiting thread is suspended until the phase completes or this many
// nanoseconds pass, whichever comes first, instead of re-polling.
constexpr uint32_t kWaitSuspendNs = 1000000;
// pause between two polls of a barrier that is not yet complete
#ifndef ROWOP_WAIT_BACKOFF_NS
#define ROWOP_WAIT_BACKOFF_NS 64
#endif
constexpr uint32_t kWaitBackoffNs = ROWOP_WAIT_BACKOFF_NS;

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(kWaitSuspendNs)
      : "memory");
  return ok != 0;
}
// Waits for phase `parity` of the barrier for at most limit_ns nanoseconds.
// Returns false when the limit ran out (the caller records a timeout).
__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (;;) {
    // a retry only after a pause, so that a waiting warp leaves the issue
    // slots to the warps that have work
    __nanosleep(kWaitBackoffNs);
    if (mbar_try_wait(bar, parity)) return true;
    if (global_timer_ns() - t0 > limit_ns) return false;
  }
}
__device__ __forceinline__ uint64_t l2_evict_first_policy() {
  uint64_t pol;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
  return pol;
}
// Bulk (non-tensor TMA) copy global -> this CTA's shared memory; completion
// is signalled as transaction bytes on the mbarrier.  dst, src and bytes must
// be multiples of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void *src, uint32_t bytes,
                                         uint32_t bar, uint64_t policy) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;" ::"r"(dst),
      "l"(src), "r"(bytes), "r"(bar), "l"(policy)
      : "memory");
}

__device__ __forceinline__ uint32_t cluster_ctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_nctarank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_nctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_count_x() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%nclusterid.x;" : "=r"(r));
  return r;
}
// Full cluster barrier: every thread of every CTA of the cluster arrives
// (release) and waits (acquire); also a superset of __syncthreads().
__device__ __forceinline__ void cluster_sync() {
  asm volatile(
      "barrier.cluster.arrive.release.aligned;\n\t"
      "barrier.cluster.wait.acquire.aligned;" ::
          : "memory");
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t local_smem, uint32_t rank) {
  uint32_t r;
  asm("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(local_smem), "r"(rank));
  return r;
}
// Load from a peer CTA's shared memory.  Volatile, so it stays after the
// (volatile) barrier wait that publishes the data, but without a memory
// clobber, so independent loads issue back to back before their results are
// stored anywhere.
__device__ __forceinline__ float4 ld_dsmem_f4(uint32_t addr) {
  float4 v;
  asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
               : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
               : "r"(addr));
  return v;
}

// Named barrier over `nthreads` threads (a multiple of 32) of the CTA.
__device__ __forceinline__ void named_sync(uint32_t id, uint32_t nthreads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(nthreads) : "memory");
}
// Named barrier that also ORs a predicate over the participating threads.
__device__ __forceinline__ bool named_sync_or(uint32_t id, uint32_t nthreads, bool pred) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(pred)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
// Arrive, with release at cluster scope, on the barrier at the same shared
// memory offset in the CTA of the given cluster rank.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t local_bar, uint32_t rank) {
  const uint32_t remote = map_to_rank(local_bar, rank);
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(remote)
               : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(kWaitSuspendNs)
      : "memory");
  return ok != 0;
}
// Bounded wait with acquire at cluster scope (for barriers peers arrive on).
__device__ __forceinline__ bool mbar_wait_cluster_bounded(uint32_t bar, uint32_t parity,
                                                          uint64_t limit_ns) {
  if (mbar_try_wait_cluster(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (;;) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    if (global_timer_ns() - t0 > limit_ns) return false;
  }
}
__device__ __forceinline__ void fence_cluster() {
  asm volatile("fence.acq_rel.cluster;" ::: "memory");
}

// Streaming 16-byte global load / store (evict-first in L1/L2).
__device__ __forceinline__ uint4 ldg_stream(const void *p) {
  return __ldcs(reinterpret_cast<const uint4 *>(p));
}
__device__ __forceinline__ void stg_stream(void *p, const uint4 &v) {
  __stcs(reinterpret_cast<uint4 *>(p), v);
}

}  // namespace rowop
