// Guard zones around the sub-buffers of a handle's device arena.
//
// Every buffer taken from the arena is followed by a guard zone: the bytes
// from the buffer's end up to the next 1024-byte boundary plus one more
// 1024-byte block. At create time the zones are filled with a fixed byte;
// elasto_check_guards verifies on the device that every zone still holds it,
// so a kernel that writes past the end of its output (a wrong tail bound, a
// TMA box beyond the map's extent) is caught by the tests without a memory
// checker. The zone table lives in a small device allocation of its own.
#pragma once
#include <string>
#include <vector>

#include "common.h"

namespace elasto {

constexpr unsigned char kGuardByte = 0xA5;

struct GuardedArena {
  static constexpr size_t kAlign = 1024;
  static constexpr size_t kGuard = 1024;
  struct Zone {
    size_t off = 0;
    size_t bytes = 0;
    std::string name;
  };
  size_t off = 0;
  std::vector<Zone> zones;
  // device copy of the zone table (offsets, lengths) and the per-zone count
  // of damaged bytes; set up by upload()
  unsigned long long* d_off = nullptr;
  unsigned long long* d_len = nullptr;
  unsigned int* d_bad = nullptr;

  // Offset of a new buffer of `bytes` bytes, 1024-byte aligned, followed by
  // its guard zone.
  size_t take(size_t bytes, const char* name = "arena buffer") {
    const size_t r = (off + kAlign - 1) / kAlign * kAlign;
    const size_t end = r + bytes;
    const size_t zend = (end + kAlign - 1) / kAlign * kAlign + kGuard;
    zones.push_back(Zone{end, zend - end, name});
    off = zend;
    return r;
  }
  // Device zone table + fill of every zone with kGuardByte (synchronous).
  elasto_status upload(char* base);
  // Synchronises `s`, then counts damaged bytes per zone on the device.
  // Returns the number of damaged zones (< 0: CUDA error) and the first
  // damaged zone's name.
  int check(char* base, cudaStream_t s, std::string* first_bad) const;
  void release();
};

// Fill / check kernels (elementwise.cu): zone z covers len[z] bytes at
// base + off[z].
cudaError_t guard_fill_launch(char* base, const unsigned long long* off, const unsigned long long* len, int nz,
                              cudaStream_t s);
cudaError_t guard_check_launch(const char* base, const unsigned long long* off, const unsigned long long* len, int nz,
                               unsigned int* bad, cudaStream_t s);

}  // namespace elasto
