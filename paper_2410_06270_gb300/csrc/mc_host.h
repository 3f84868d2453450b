// mc_host.h -- host-side helpers shared by the library's translation units:
// thread-local error text and argument validation.
#pragma once
#include <stdarg.h>
#include <stddef.h>
#include <stdint.h>
#include <stdio.h>

#include "../../include/mc.h"
#include "mc_layout.h"

namespace mc {

int set_error(int code, const char *fmt, ...);
void clear_error();

// Validates a shape (and optionally a bit table).  Returns MC_OK or an error
// code with the message set.
int check_shape(const mc_shape *s);
int check_bits(const mc_shape *s, const int8_t *bits_host);

// Byte offsets of every (expert, matrix) inside a packed buffer.
void layout_offsets(const mc_shape *s, const int8_t *bits, uint64_t off[kMaxE][3], uint64_t *total);

inline bool aligned(const void *p, size_t a) { return ((uintptr_t)p % a) == 0; }

}  // namespace mc
