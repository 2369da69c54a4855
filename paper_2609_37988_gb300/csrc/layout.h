// layout.h -- stored layout of one anchor's cache (host and device).
//
// Every (position, KV head) of a GQA anchor is one contiguous, 16-byte
// aligned RECORD:
//
//     [ K section | V section | K meta (per-token keys) | V meta ]
//
//   K/V section  head_dim codes at `bits` (16 = bf16 values, 8 = one code per
//                byte, 4 = two codes per byte), in the fragment order below;
//   meta         one float2 (scale, zero) per group of `group` channels,
//                natural group order, padded to 16 bytes.
//
// Per-channel keys (KIVI layout) keep the K codes in the record and store
// (scale, zero) per (group of `group` positions, channel) in a separate
// group-meta plane; positions of a not-yet-full group stay bf16 in a
// residual plane (row = position mod group) in the bf16 K fragment order.
//
// Records are stored [batch][kv head][position] with `cap` positions per
// (batch, kv head) slab, so a run of positions is one contiguous block (one
// copy per tile when streaming) and one position is 1-2 cache lines (few
// sectors per kept position when gathering an eviction list).
//
// Fragment order.  The decode kernel multiplies with mma.m16n8k16: for
// scores, A = keys (16 positions x 16 channels); for the value product,
// A = V^T (16 channels x 16 positions).  Channels are permuted on write so
// that the bytes one lane needs for its A fragments are contiguous:
//
//   K: channel ch -> k-step j = ch/16, slot s = ch%16, lane column
//      c = (s%8)/2, element n = 4j + r with r = (s%2) + 2*(s/8), i.e. lane c
//      holds slots {2c, 2c+1, 2c+8, 2c+9} of every k-step.  Lane c's segment
//      (head_dim/4 elements) is split into 16-byte chunks; chunk i of lane c
//      sits at chunk index 4i + c.  For 4-bit keys each 32-bit word holds
//      k-steps (2w, 2w+1) with nibbles ordered so that masking with
//      0x000F000F / 0x00F000F0 (and again after >> 8) yields the f16 pairs of
//      the a0 / a2 registers directly.
//   V, bf16: channel ch -> M-block m = ch/16, row rr = ch%16, lane row
//      g = rr%8, e = rr/8; lane g's segment (head_dim/8 elements) holds
//      (m, e) at element 2m + e.
//   V, codes: laid out for ldmatrix.trans over 8 positions x 16 bytes: the
//      16-bit element g of 16-byte chunk k is lane row g's pair of bytes for
//      M-blocks (2k, 2k+1) (4-bit: byte 16k + 2g + (m%2) holds row g in the
//      low nibble, row g+8 in the high nibble) or for M-block k (8-bit: byte
//      16k + 2g + e).  The chunks of position t are rotated by v_rot(t), so
//      that eight consecutive records' copies of one chunk fall in eight
//      distinct 16-byte bank slots of shared memory.
//
// Symmetric per-vector scheme (the paper's own quantiser, Appendix C.3: one
// bf16 scale per token-head row, no zero point, codes in [-q, q] with
// q = 2^(b-1) - 1, b = 2, 4 or 8).  Codes are stored offset by q (u = code +
// q, unsigned) in the same fragment orders as above, 2-bit codes as below.
// The record holds only [K section | V section]; the two bf16 scales of a
// (position, KV head) sit in a scale plane [slab][cap] as one 32-bit word
// (K scale in the low half, V scale in the high half).  The record's 16-byte
// chunks are rotated as a whole: logical chunk u of position t sits at chunk
// (u + sym_rot(t)) mod nch.  With 64-byte records (2-bit) the rotation is
// (t/2) mod 4, with 128- or 256-byte records t mod 8; either way the key
// fragments of eight consecutive positions and the ldmatrix rows of one value
// chunk fall on distinct shared-memory bank slots.
//
//   2-bit K: lane c's segment is 8 bytes (two 32-bit words); word w holds
//      k-steps 4w..4w+3.  In each 16-bit half (low half: slots 2c and 2c+8,
//      high half: 2c+1 and 2c+9) byte jj/2 of k-step jj = j % 4 holds four
//      2-bit fields: field 2 (jj % 2) + a for a = 0 (a0 register) or 1 (a2),
//      so a mask of 0x00030003 << (4 (jj % 2)) (a0) or 0x000C000C << ...
//      (a2), after >> 8 for jj >= 2, yields the f16 pair at weight 4^field.
//   2-bit V: the 16-bit element g of 16-byte chunk k holds lane row g's
//      fields of M-blocks 4k..4k+3: byte (m/2) % 2, field 2 (m % 2) + e for
//      row g + 8e.
//
// An MLA anchor stores [c[:width] | k^R] in bf16, natural order, one record
// per (batch, position).
#pragma once
#include <stdint.h>

#if defined(__CUDACC__)
#define KVK_HD __host__ __device__ __forceinline__
#else
#define KVK_HD inline
#endif

namespace kvk {

constexpr int kTile = 64;  // positions per decode tile

// quantisation schemes of a GQA anchor
constexpr int kSchemeGrouped = 0;    // asymmetric, (scale, zero) per group
constexpr int kSchemeSym = 1;        // symmetric, one bf16 scale per row

KVK_HD int sec_bytes(int bits, int D) { return D * bits / 8; }
KVK_HD int meta_bytes(int D, int g) { return (((D / g) * 8) + 15) & ~15; }

struct RecLayout {
  int k_off, v_off, km_off, vm_off, rec;
};

// key_axis: 0 = per token, 1 = per channel.
KVK_HD RecLayout rec_layout(int bits, int D, int g, int key_axis) {
  RecLayout L;
  const int s = sec_bytes(bits, D);
  L.k_off = 0;
  L.v_off = s;
  int off = 2 * s;
  if (bits == 16) {
    L.km_off = -1;
    L.vm_off = -1;
    L.rec = off;
    return L;
  }
  if (key_axis == 0) {
    L.km_off = off;
    off += meta_bytes(D, g);
  } else {
    L.km_off = -1;
  }
  L.vm_off = off;
  off += meta_bytes(D, g);
  L.rec = off;
  return L;
}

// Position of channel `ch` inside the K section: byte offset, and for 4-bit
// codes whether it is the high nibble.
KVK_HD void k_pos(int ch, int bits, int D, int *byte, int *hi) {
  const int j = ch >> 4, s = ch & 15;
  const int c = (s & 7) >> 1;
  const int r = (s & 1) | ((s >> 3) << 1);
  const int n = 4 * j + r;
  const int seg = D * bits / 32;  // bytes per lane segment
  int bp;
  *hi = 0;
  if (bits == 16) {
    bp = 2 * n;
  } else if (bits == 8) {
    bp = n;
  } else {
    const int w = j >> 1, jj = j & 1;
    const int nib = (r & 1) * 4 + (r >> 1) + 2 * jj;
    bp = 4 * w + (nib >> 1);
    *hi = nib & 1;
  }
  *byte = (seg >= 16) ? 16 * (4 * (bp >> 4) + c) + (bp & 15) : seg * c + bp;
}

// Chunk rotation of the V section of position t (records of rec_bytes, nc
// 16-byte chunks, nc a power of two).  With R = rec_bytes / 16 the natural
// bank slot of record t is R t mod 8: all distinct for odd R, period 4 for
// R = 2 mod 4, period 2 for R = 4 mod 8, constant for R = 0 mod 8.
KVK_HD int v_rot(int t, int rec_bytes, int nc) {
  const int R = rec_bytes >> 4;
  const int r = (R & 1) ? 0 : ((R & 3) == 2) ? (t >> 2) : ((R & 7) == 4) ? (t >> 1) : t;
  return r & (nc - 1);
}

// Position of channel `ch` inside the V section of position t.
KVK_HD void v_pos(int ch, int bits, int D, int t, int rec_bytes, int *byte, int *hi) {
  const int m = ch >> 4, rr = ch & 15;
  const int g = rr & 7, e = rr >> 3;
  *hi = 0;
  if (bits == 16) {
    *byte = (D / 4) * g + 2 * (2 * m + e);
    return;
  }
  int bl;  // logical byte
  if (bits == 8) {
    bl = 16 * m + 2 * g + e;
  } else {
    bl = 16 * (m >> 1) + 2 * g + (m & 1);
    *hi = e;
  }
  const int nc = D * bits / 128;
  *byte = 16 * (((bl >> 4) + v_rot(t, rec_bytes, nc)) & (nc - 1)) + (bl & 15);
}

// ---- symmetric per-vector records ------------------------------------------
KVK_HD int sym_levels(int bits) { return (1 << (bits - 1)) - 1; }
KVK_HD int sym_rec_bytes(int bits, int D) { return 2 * sec_bytes(bits, D); }
KVK_HD int sym_rot(int t, int nch) { return nch == 4 ? ((t >> 1) & 3) : (t & 7); }

// Logical bit offset of channel `ch` inside the K section (before rotation).
KVK_HD int sym_k_bit(int ch, int bits, int D) {
  if (bits == 2) {
    const int j = ch >> 4, s = ch & 15;
    const int c = (s & 7) >> 1;
    const int r = (s & 1) | ((s >> 3) << 1);
    const int w = j >> 2, jj = j & 3, h = r & 1, a = r >> 1;
    return 64 * c + 32 * w + 16 * h + 8 * (jj >> 1) + 2 * (2 * (jj & 1) + a);
  }
  int byte, hi;
  k_pos(ch, bits, D, &byte, &hi);
  return 8 * byte + 4 * hi;
}

// Logical bit offset of channel `ch` inside the V section (before rotation).
KVK_HD int sym_v_bit(int ch, int bits, int D) {
  const int m = ch >> 4, rr = ch & 15;
  const int g = rr & 7, e = rr >> 3;
  if (bits == 2) return 8 * (16 * (m >> 2) + 2 * g + ((m >> 1) & 1)) + 2 * (2 * (m & 1) + e);
  if (bits == 8) return 8 * (16 * m + 2 * g + e);
  (void)D;
  return 8 * (16 * (m >> 1) + 2 * g + (m & 1)) + 4 * e;
}

// Physical byte of logical record byte `lb` of position t.
KVK_HD int sym_phys(int lb, int t, int rec_bytes) {
  const int nch = rec_bytes >> 4;
  return 16 * (((lb >> 4) + sym_rot(t, nch)) & (nch - 1)) + (lb & 15);
}

KVK_HD int64_t align256(int64_t x) { return (x + 255) & ~(int64_t)255; }

// ---- quantised MLA latents --------------------------------------------------
// A position of a quantised MLA anchor stores two vectors, the kept latent
// c[:width] and the positional key k^R, as unsigned codes (symmetric: code +
// q; grouped: the code), in one record of (width + rope) * bits / 8 bytes:
// coordinate k of the concatenation [c[:width] | k^R] in chunk k / 8 of
// `bits` bytes, within which code k % 8 = 2 p + h sits at
//   8 bits: byte 2 p + h;
//   4 bits: bits 4 p + 16 h of the chunk's 32-bit word;
//   2 bits: bits 2 p + 8 h of the chunk's 16-bit half-word;
// so that the f16 pair (code 2p, code 2p+1) is one byte permute (8 bits) or
// one shift and mask (4 and 2 bits) away.  Beside the records, a plane of
// per-position metadata: symmetric, one 32-bit word (bf16 scale of the
// latent, bf16 scale of k^R in the high half); grouped, a float4 (latent
// scale, latent zero, k^R scale, k^R zero).
KVK_HD int mla_q_rec_bytes(int width, int rope, int bits) { return (width + rope) * bits / 8; }
KVK_HD int mla_q_meta_bytes(int scheme) { return scheme == kSchemeSym ? 4 : 16; }
// bit offset of code k (0..7) inside its chunk
KVK_HD int mla_q_bit(int k, int bits) {
  const int p = k >> 1, h = k & 1;
  return bits == 8 ? 8 * (2 * p + h) : bits == 4 ? 4 * p + 16 * h : 2 * p + 8 * h;
}

// Offsets inside one anchor's arena.
struct ArenaLayout {
  int64_t lens;      // int32[B]
  int64_t counter;   // int32 (append completion counter)
  int64_t kept_n;    // int32[B * Hkv]: per sequence, or per (sequence, kv head)
  int64_t kept_idx;  // int32[B * Hkv * kept_cap]
  int64_t rec;       // records
  int64_t gmeta;     // float2 [B*Hkv][cap/g][D] (per-channel keys)
  int64_t resid;     // bf16 K rows [B*Hkv][g][D] (per-channel keys)
  int64_t scales;    // uint32 [B*Hkv][cap] bf16 (K, V) scales (symmetric scheme)
  int64_t total;
  int64_t cap;       // positions per slab (max_ctx rounded up to kTile)
  int rec_bytes;
};

// mla: records are [B][cap][(width + rope) * 2 bytes]; kv heads = 1.
KVK_HD ArenaLayout arena_layout(int mla, int B, int Hkv, int max_ctx, int D, int bits,
                                int g, int key_axis, int kept_cap, int width, int rope,
                                int scheme = kSchemeGrouped) {
  ArenaLayout A;
  A.cap = ((int64_t)max_ctx + kTile - 1) / kTile * kTile;
  int64_t off = 0;
  A.lens = off;
  off = align256(off + 4 * (int64_t)B);
  A.counter = off;
  off = align256(off + 4);
  A.kept_n = off;
  off = align256(off + 4 * (int64_t)B * Hkv);
  A.kept_idx = off;
  off = align256(off + 4 * (int64_t)B * Hkv * kept_cap);
  A.rec = off;
  A.scales = -1;
  if (mla) {
    A.rec_bytes = bits == 16 ? (width + rope) * 2 : mla_q_rec_bytes(width, rope, bits);
    off = align256(off + (int64_t)B * A.cap * A.rec_bytes);
    A.gmeta = A.resid = -1;
    if (bits != 16) {
      A.scales = off;  // per-position metadata plane
      off = align256(off + (int64_t)B * A.cap * mla_q_meta_bytes(scheme));
    }
  } else if (bits != 16 && scheme == kSchemeSym) {
    A.rec_bytes = sym_rec_bytes(bits, D);
    off = align256(off + (int64_t)B * Hkv * A.cap * A.rec_bytes);
    A.scales = off;
    off = align256(off + (int64_t)B * Hkv * A.cap * 4);
    A.gmeta = A.resid = -1;
  } else {
    A.rec_bytes = rec_layout(bits, D, g, key_axis).rec;
    off = align256(off + (int64_t)B * Hkv * A.cap * A.rec_bytes);
    if (bits != 16 && key_axis == 1) {
      A.gmeta = off;
      off = align256(off + (int64_t)B * Hkv * (A.cap / g) * D * 8);
      A.resid = off;
      off = align256(off + (int64_t)B * Hkv * g * D * 2);
    } else {
      A.gmeta = A.resid = -1;
    }
  }
  A.total = off;
  return A;
}

}  // namespace kvk
